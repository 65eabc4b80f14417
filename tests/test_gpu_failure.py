"""Failure detection on the GPU without a fault: a bounded device wait that runs out.

Every mbarrier wait in the library's kernels has a time limit; when it runs
out the kernel records ERR_TIMEOUT and winds down, and the host call returns
DLMZ_ETIMEOUT.  The self-test kernel waits (limit 1 ms) on an mbarrier that
expects an arrival nobody makes.  Afterwards the error word is clear and the
context still runs the tensor-core GEMM correctly.
"""
import numpy as np
import pytest

from tests.gpu_helpers import dlmz, ptr

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_stays_usable(dev):
    import torch
    d = dlmz()
    assert d.selftest_wait_timeout(1000) == d.ETIMEOUT
    assert d.selftest_wait_timeout(200) == d.ETIMEOUT
    d.check()  # the timeout bit was reported once and cleared
    g = torch.Generator(device="cuda").manual_seed(3)
    A = torch.randn(256, 128, device="cuda", generator=g).to(torch.bfloat16)
    B = torch.randn(512, 128, device="cuda", generator=g).to(torch.bfloat16)
    D = torch.empty(256, 512, dtype=torch.float32, device="cuda")
    d.gemm_bf16(ptr(A), ptr(B), ptr(D), 256, 512, 128)
    d.check()
    ref = A.double() @ B.double().T
    assert float((D.double() - ref).abs().max()) < 1e-3


def test_cluster_wait_times_out_only_without_the_peer(dev):
    """The cluster-scope bounded wait of the quantiser's CTA pairs: it completes when the other CTA
    of the cluster arrives through distributed shared memory and gives up (ETIMEOUT, context
    usable) when it does not."""
    d = dlmz()
    assert d.selftest_cluster_wait(1000, 1) == 0
    assert d.selftest_cluster_wait(1000, 0) == d.ETIMEOUT
    assert d.selftest_cluster_wait(200, 0) == d.ETIMEOUT
    assert d.selftest_cluster_wait(1000, 1) == 0
    d.check()
    assert d.selftest_cluster_wait(0, 0) == d.EINVAL
    assert d.selftest_cluster_wait(1000, 2) == d.EINVAL


def test_selftest_rejects_bad_limits(dev):
    d = dlmz()
    assert d.selftest_wait_timeout(0) == d.EINVAL
    assert d.selftest_wait_timeout(2_000_000) == d.EINVAL
