"""GPU quantiser vs the oracle, bit-exact on identical float32 logits."""
import numpy as np
import pytest

from oracle import quantizer as Q
from paper_2608_11249_gb300 import sources
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu


def _rows(V, n, seed):
    l = sources.synthetic_logits(seed, 0, 0, n, V)
    extra = [np.zeros(V), np.full(V, -1e30), np.linspace(-100, 100, V)]
    x = np.zeros(V); x[V // 3] = 1e6; extra.append(x)
    x = np.full(V, -3e38); x[-1] = 3e38; extra.append(x)
    x = np.zeros(V); x[[1, V - 1]] = 7.0; extra.append(x)  # tie for the maximum
    return np.concatenate([l, np.array(extra, dtype=np.float32)]).astype(np.float32)


@pytest.mark.parametrize("V,n", [(2, 9), (4, 33), (37, 70), (256, 300), (300, 50), (512, 40), (1000, 20), (1001, 7),
                                 (5000, 17), (126464, 5), (152064, 3),
                                 # more rows than SMs: each CTA of the large-vocabulary kernel walks several rows
                                 (1000, 1300), (4100, 700),
                                 # the smallest halves of the two-CTA kernel (V = 516: 65 and 64 float4s)
                                 # and a vocabulary whose rows start at every word offset modulo 4
                                 (516, 11), (1028, 9)])
def test_quantize_bit_exact(dev, V, n):
    import torch
    d = dlmz()
    l = _rows(V, n, V)
    rows = l.shape[0]
    P = Q.precision_for_vocab(V)
    ref = Q.quantize(l, P)
    dl = to_dev(l)
    cdf = torch.empty(rows, V + 1, dtype=torch.int32, device="cuda")
    W = torch.empty(rows, dtype=torch.int64, device="cuda")
    A = torch.empty(rows, dtype=torch.int64, device="cuda")
    Hq = torch.empty(rows, dtype=torch.int32, device="cuda")
    top = torch.empty(rows, dtype=torch.int32, device="cuda")
    d.quantize(ptr(dl), rows, V, P, ptr(cdf), ptr(W), ptr(A), ptr(Hq), ptr(top))
    d.check()
    assert np.array_equal(cdf.cpu().numpy().view(np.uint32), ref["cdf"])
    assert np.array_equal(W.cpu().numpy().view(np.uint64), ref["W"])
    assert np.array_equal(A.cpu().numpy().view(np.uint64), ref["A"])
    assert np.array_equal(Hq.cpu().numpy(), ref["Hq"].astype(np.int32))
    assert np.array_equal(top.cpu().numpy(), ref["top"].astype(np.int32))


@pytest.mark.parametrize("V,n", [(5000, 9), (126464, 4)])
def test_quantize_unaligned_buffers(dev, V, n):
    """CDF rows off a 16-byte boundary (one CTA per row in flight) and logits off a 16-byte boundary
    (the generic kernel) give the same tables as the aligned case."""
    import torch
    d = dlmz()
    l = _rows(V, n, V + 1)
    rows = l.shape[0]
    P = Q.precision_for_vocab(V)
    ref = Q.quantize(l, P)
    W = torch.empty(rows, dtype=torch.int64, device="cuda")
    Hq = torch.empty(rows, dtype=torch.int32, device="cuda")
    cbuf = torch.empty(rows * (V + 1) + 4, dtype=torch.int32, device="cuda")
    cdf = cbuf[1:1 + rows * (V + 1)]  # 4 bytes past an aligned start
    d.quantize(ptr(to_dev(l)), rows, V, P, ptr(cdf), ptr(W), 0, ptr(Hq), 0)
    d.check()
    assert np.array_equal(cdf.cpu().numpy().view(np.uint32).reshape(rows, V + 1), ref["cdf"])
    assert np.array_equal(Hq.cpu().numpy(), ref["Hq"].astype(np.int32))
    lbuf = torch.zeros(rows * V + 4, dtype=torch.float32, device="cuda")
    lbuf[1:1 + rows * V] = torch.from_numpy(l.ravel()).cuda()
    cdf2 = torch.empty(rows, V + 1, dtype=torch.int32, device="cuda")
    d.quantize(ptr(lbuf[1:]), rows, V, P, ptr(cdf2), ptr(W), 0, ptr(Hq), 0)
    d.check()
    assert np.array_equal(cdf2.cpu().numpy().view(np.uint32), ref["cdf"])
    assert np.array_equal(W.cpu().numpy().view(np.uint64), ref["W"])


def test_quantize_isolated_workload_rows(dev):
    """Rows of the isolated quantise+select workload (N(0,3) + spike U(5,15), V = 126464)."""
    import torch
    d = dlmz()
    V, rows = 126464, 24
    l = sources.spiked_rows(0, 1000, rows, V)
    ref = Q.quantize(l, 24)
    cdf = torch.empty(rows, V + 1, dtype=torch.int32, device="cuda")
    W = torch.empty(rows, dtype=torch.int64, device="cuda")
    Hq = torch.empty(rows, dtype=torch.int32, device="cuda")
    d.quantize(ptr(to_dev(l)), rows, V, 24, ptr(cdf), ptr(W), 0, ptr(Hq), 0)
    d.check()
    assert np.array_equal(cdf.cpu().numpy().view(np.uint32), ref["cdf"])
    assert np.array_equal(Hq.cpu().numpy(), ref["Hq"].astype(np.int32))


@pytest.mark.parametrize("V", [64, 1000, 1001, 5000, 126464])
def test_quantize_rejects_non_finite(dev, V):
    """NaN / +inf / -inf among positive and negative logits: EBADINPUT, tables in range, context usable."""
    import torch
    d = dlmz()
    l = np.linspace(-5, 5, 6 * V, dtype=np.float32).reshape(6, V)
    l[1, 5] = np.nan
    l[2, V - 1] = np.inf
    l[3, 0] = -np.inf
    l[4, [1, V // 2]] = [np.nan, np.inf]
    P = Q.precision_for_vocab(V)
    cdf = torch.empty(6, V + 1, dtype=torch.int32, device="cuda")
    W = torch.empty(6, dtype=torch.int64, device="cuda")
    Hq = torch.empty(6, dtype=torch.int32, device="cuda")
    d.quantize(ptr(to_dev(l)), 6, V, P, ptr(cdf), ptr(W), 0, ptr(Hq), 0)
    with pytest.raises(d.DlmzError) as e:
        d.check()
    assert e.value.code == d.EBADINPUT
    d.check()  # flag cleared
    c = cdf.cpu().numpy().view(np.uint32).astype(np.int64)
    ref = Q.quantize(l[[0, 5]], P)  # the finite rows are still exact
    assert np.array_equal(c[[0, 5]], ref["cdf"].astype(np.int64))
    for i in (1, 2, 3, 4):  # the others stay non-decreasing tables within [0, 2^P]
        assert c[i, 0] == 0 and c[i, -1] <= (1 << P) and np.all(np.diff(c[i]) >= 0)
