"""GPU selector vs the oracle's (key, position) ordering, bit-exact."""
import numpy as np
import pytest

from oracle import selector as S
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("groups,g,k,span", [(1, 1, 1, 3), (5, 10, 3, 4), (7, 100, 32, 50), (3, 1024, 32, 1 << 40),
                                             (2, 1024, 32, 5), (4, 4096, 64, 1000),
                                             (6, 2048, 64, 0)])  # span 0: full 64-bit keys with repeats
def test_select_smallest(dev, groups, g, k, span):
    import torch
    d = dlmz()
    rng = np.random.default_rng(g * 7 + k)
    if span:
        keys = rng.integers(0, span, (groups, g)).astype(np.uint64)
    else:  # every byte of the key matters (the high bit set too), and a tenth of the keys repeat others
        keys = rng.integers(0, 1 << 62, (groups, g)).astype(np.uint64) * np.uint64(3)
        rep = rng.random((groups, g)) < 0.1
        keys[rep] = keys[:, :1].repeat(g, axis=1)[rep]
    out = torch.empty(groups, k, dtype=torch.int32, device="cuda")
    d.select_smallest(ptr(to_dev(keys.view(np.int64))), groups, g, k, ptr(out))
    d.check()
    got = out.cpu().numpy()
    for i in range(groups):
        ref = sorted(S.smallest(keys[i], np.arange(g), k))
        assert got[i].tolist() == ref
