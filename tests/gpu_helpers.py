"""Shared helpers of the GPU parity tests (device buffers via torch)."""
import numpy as np


def dlmz():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_11249_gb300 import dlmz as d
    return d


def to_dev(a):
    import torch
    return torch.from_numpy(np.array(a, copy=True, order="C")).cuda()


def ptr(t):
    return 0 if t is None else t.data_ptr()
