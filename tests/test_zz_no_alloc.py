"""The allocation-free selection entry point agrees with the allocating one.

dlmz_select_smallest_noalloc serves callers that cannot call cudaMalloc
(device memory owned by another allocator, paths that cannot take
cudaMalloc's device synchronisation, fixed memory budgets): its scratch is a
static device array.  This file is collected last so a failure here comes
after every other test has run; it also passes alone in a fresh process,
where its first call performs the per-device set-up.
"""
import numpy as np
import pytest

from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu


def test_noalloc_select_matches_allocating_entry_point_twice(dev):
    import torch
    d = dlmz()
    for call, (groups, g, k, span) in enumerate([(64, 1024, 32, 1 << 20), (300, 200, 17, 9)]):
        rng = np.random.default_rng(call)
        keys = to_dev(rng.integers(0, span, (groups, g)).astype(np.int64))
        ref = torch.empty(groups, k, dtype=torch.int32, device="cuda")
        got = torch.full((groups, k), -1, dtype=torch.int32, device="cuda")
        d.select_smallest(ptr(keys), groups, g, k, ptr(ref))
        d.select_smallest_noalloc(ptr(keys), groups, g, k, ptr(got))
        d.check()
        assert torch.equal(ref, got), call


def test_noalloc_select_rejects_too_many_groups(dev):
    import torch
    d = dlmz()
    keys = torch.zeros(2, dtype=torch.int64, device="cuda")
    out = torch.zeros(2, dtype=torch.int32, device="cuda")
    with pytest.raises(d.DlmzError) as e:
        d.select_smallest_noalloc(ptr(keys), 65537, 1, 1, ptr(out))
    assert e.value.code == d.EINVAL
