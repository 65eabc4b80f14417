"""Parity at the workloads' own sizes, on outputs the oracle can compute one by one.

* byte workload (8-layer d=512 bf16, 1024 windows x 512) in the benchmark's
  launch configuration: sampled windows' logits vs the oracle, and a full
  512 KiB batch round trip through the device-resident API;
* layers of the 8B-shaped (d=4096, 32 heads, FFN 12288) and 7B GQA-shaped
  (d=3584, 28/4 heads, FFN 18944) models, one layer deep, sampled rows, within
  twice the divergence of the oracle's own float32-contraction evaluation;
* the isolated quantise+select workload (65536 x 126464 logits) at full size,
  sampled rows and groups bit-exact;
* the tiny float32 byte model, full round trip, compressed size vs the oracle
  on a sample of windows.
"""
import numpy as np
import pytest

from oracle import model as OM
from oracle import pipeline as OP
from oracle import quantizer as OQ
from oracle import selector as OS
from paper_2608_11249_gb300 import sources
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def _forward_sampled(d, spec, nc, L, row0, rpc, sample, seed, tol=None):
    """GPU logits of sampled windows vs the oracle.  ``tol``: a fixed max-abs bound (rms a
    quarter of it); None: at most twice the divergence of the oracle's own float32-contraction
    evaluation on the same rows (the wide layers, where bf16 rounding flips spread)."""
    import torch
    nl, dm, nh, nkv, F, V, dt = spec
    m = d.Model(nl, dm, nh, nkv, F, V, d.BF16 if dt == "bf16" else d.FP32, seed=seed)
    rng = np.random.default_rng(seed)
    state = rng.integers(0, V, (nc, L)).astype(np.int32)
    state[rng.random((nc, L)) < 0.5] = V
    logits = torch.empty(nc * rpc, V, dtype=torch.float32, device="cuda")
    m.forward_logits(ptr(to_dev(state)), nc, L, row0, rpc, ptr(logits))
    d.check()
    got = logits.view(nc, rpc, V)
    w = OM.Weights(OM.ModelConfig(*spec, seed=seed))
    for c in sample:
        rows = np.arange(row0, row0 + rpc)
        ref = OM.forward(w, state[c], rows=rows)
        diff = got[c].cpu().numpy() - ref
        err = float(np.max(np.abs(diff)))
        rms = float(np.sqrt(np.mean(diff ** 2)))
        if tol is not None:
            assert err <= tol and rms <= tol / 4, (c, err, rms)
        else:
            alt = OM.forward(w, state[c], rows=rows, matmul_dtype=np.float32) - ref
            nerr, nrms = float(np.max(np.abs(alt))), float(np.sqrt(np.mean(alt ** 2)))
            print("%s window %d: GPU vs oracle max-abs %.4g rms %.4g; oracle float32 vs float64 max-abs %.4g rms %.4g"
                  % (spec[:6], c, err, rms, nerr, nrms))
            assert err <= 2 * nerr and rms <= 2 * nrms, (c, err, rms, nerr, nrms)
    m.close()


def test_byte_workload_full_batch(dev):
    import torch
    d = dlmz()
    spec = (8, 512, 8, 8, 2048, 256, "bf16")
    _forward_sampled(d, spec, 1024, 512, 128, 128, [0, 777, 1023], 0, 2e-2)
    m = d.Model(8, 512, 8, 8, 2048, 256, d.BF16, seed=0)
    data = sources.markov_bytes(1024 * 512, seed=3)
    din = to_dev(np.frombuffer(data, dtype=np.uint8))
    cap = m.compress_bound(len(data), 512)
    dc = torch.empty(cap, dtype=torch.uint8, device="cuda")
    pol = d.policy(d.TOPK_CONF, 8, 128)
    n = m.compress_device(ptr(din), len(data), 512, pol, ptr(dc), cap, batch_chunks=1024)
    back = torch.empty(len(data), dtype=torch.uint8, device="cuda")
    k = m.decompress_device(ptr(dc), n, ptr(back), len(data))
    assert k == len(data) and torch.equal(back, din)
    assert 7.9 < 8.0 * n / len(data) < 8.5  # random-init model: about 8 bits per byte


@pytest.mark.parametrize("spec", [(1, 4096, 32, 32, 12288, 1024, "bf16"),   # 8B-shaped layer, hd 128
                                  (1, 3584, 28, 4, 18944, 1024, "bf16")])   # 7B GQA-shaped layer, 7:1
def test_large_model_layers(dev, spec):
    d = dlmz()
    _forward_sampled(d, spec, 3, 256, 0, 256, [0, 2], 5)


def test_isolated_quantize_select_full_size(dev):
    import torch
    d = dlmz()
    R, V, G, K = 65536, 126464, 1024, 32
    g = torch.Generator(device="cuda").manual_seed(0)
    logits = torch.randn(R, V, device="cuda", generator=g)
    logits.mul_(3.0)
    cols = torch.randint(0, V, (R,), device="cuda", generator=g)
    logits[torch.arange(R, device="cuda"), cols] += torch.rand(R, device="cuda", generator=g) * 10.0 + 5.0
    cdf = torch.empty(R, V + 1, dtype=torch.int32, device="cuda")
    W = torch.empty(R, dtype=torch.int64, device="cuda")
    Hq = torch.empty(R, dtype=torch.int32, device="cuda")
    d.quantize(ptr(logits), R, V, 24, ptr(cdf), ptr(W), 0, ptr(Hq), 0)
    keys = Hq.to(torch.int64)
    sel = torch.empty(R // G, K, dtype=torch.int32, device="cuda")
    d.select_smallest(ptr(keys), R // G, G, K, ptr(sel))
    d.check()
    rng = np.random.default_rng(1)
    rows = torch.as_tensor(np.concatenate([[0, R - 1], rng.integers(0, R, 14)]), device="cuda")
    ref = OQ.quantize(logits[rows].cpu().numpy(), 24)
    assert np.array_equal(cdf[rows].cpu().numpy().view(np.uint32), ref["cdf"])
    assert np.array_equal(W[rows].cpu().numpy().view(np.uint64), ref["W"])
    assert np.array_equal(Hq[rows].cpu().numpy(), ref["Hq"].astype(np.int32))
    for grp in (0, 31, 63):
        hq = Hq[grp * G:(grp + 1) * G].cpu().numpy()
        want = sorted(OS.smallest(hq, np.arange(G), K))
        assert sel[grp].cpu().numpy().tolist() == want


def test_tiny_float32_workload(dev):
    d = dlmz()
    spec = (2, 128, 4, 4, 512, 256, "f32")
    m = d.Model(2, 128, 4, 4, 512, 256, d.FP32, seed=0)
    data = sources.markov_bytes(16 * 1024, seed=0)
    pol = d.policy(d.TOPK_CONF, 4, 64)
    blob = m.compress(data, 1024, pol)
    assert m.decompress(blob) == data
    # compressed size of two windows vs the oracle's end-to-end compression of them
    sub = data[:2048]
    gsub = m.compress(sub, 1024, pol)
    w = OM.Weights(OM.ModelConfig(*spec, seed=0))
    osub = OP.compress(w, sub, 1024, OS.Policy(kind=OS.TOPK_CONF, k=4, block=64))
    assert abs(len(gsub) - len(osub)) <= 0.005 * len(osub)
