"""The 8B-shaped and 7B GQA-shaped models at full size on the GPU.

* 8B-shaped: 32 layers, d = 4096, 32 heads (head dim 128), FFN 12288,
  V = 126464, windows of 1024 tokens, top-16 by confidence over the window.
* 7B GQA-shaped: 28 layers, d = 3584, 28 query / 4 KV heads (head dim 128),
  FFN 18944, V = 152064, windows of 2048, entropy threshold 0.5 bits with
  m = 1 and at most 64 positions per step.

Logits of one denoising step at full depth are compared with the oracle's
float64 forward (weights generated layer by layer by the oracle's own
counter-based draws) on sampled rows, within twice the divergence of the
oracle's own float32-contraction evaluation; whole files round-trip bit-exactly
through dlmz_compress / dlmz_decompress, also with the LM head slabbed.
The oracle's own end-to-end compression of a window of these models (about
1e15 float64 operations per window) is out of reach on the host, so the
compressed-size criterion is checked on the smaller models
(test_gpu_roundtrip.py) and the coder on identical logits at these
vocabularies (test_gpu_coder.py).
"""
import numpy as np
import pytest

from oracle import model as OM
from paper_2608_11249_gb300 import sources
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

C4 = (32, 4096, 32, 32, 12288, 126464, "bf16")
C5 = (28, 3584, 28, 4, 18944, 152064, "bf16")
# At 28-32 layers of d = 3584-4096 no evaluation that sums in another order than the
# oracle's float64 stays within the 2e-2 max-abs that holds for the byte model: one
# bf16 storage rounding that lands on the other side spreads through the next
# 4096-wide contraction into every element, and the flips compound layer by layer
# (measured on the oracle itself: float32 instead of float64 contractions, every
# rounding point kept, moves the 8B-shaped logits by rms 0.0034 after one layer,
# 0.0094 after 8).  The bound is therefore set live on the same rows: the GPU may
# differ from the float64 oracle by at most twice what the oracle's own float32
# evaluation does, in max-abs and in rms.
NOISE_FACTOR = 2.0


def _state(V, nc, L, seed, frac_masked=0.5):
    """Windows of Zipf-bigram tokens with a random half of the positions masked (a mid-step state)."""
    rng = np.random.default_rng(seed)
    tok = sources.zipf_bigram_tokens(nc * L, V, seed=seed).reshape(nc, L).astype(np.int32)
    tok[rng.random((nc, L)) < frac_masked] = V
    return tok


def _full_depth_logits(spec, nc, L, seed, check_window, row0, rpc):
    import torch
    d = dlmz()
    nl, dm, nh, nkv, F, V, _ = spec
    m = d.Model(nl, dm, nh, nkv, F, V, d.BF16, seed=seed)
    state = _state(V, nc, L, seed)
    logits = torch.empty(nc * rpc, V, dtype=torch.float32, device="cuda")
    m.forward_logits(ptr(to_dev(state)), nc, L, row0, rpc, ptr(logits))
    d.check()
    got = logits.view(nc, rpc, V)[check_window].cpu().numpy()
    m.close()
    del logits
    torch.cuda.empty_cache()
    rows = np.arange(row0, row0 + rpc)
    cfg = OM.ModelConfig(*spec, seed=seed)
    ref = OM.forward(OM.Weights(cfg, lazy=True), state[check_window], rows=rows)
    alt = OM.forward(OM.Weights(cfg, lazy=True), state[check_window], rows=rows, matmul_dtype=np.float32)
    stats = lambda x: (float(np.max(np.abs(x))), float(np.sqrt(np.mean(x ** 2))))
    (err, rms), (nerr, nrms) = stats(got - ref), stats(alt - ref)
    print("full-depth logits %s: GPU vs oracle max-abs %.4g rms %.4g; oracle float32 vs float64 max-abs %.4g rms %.4g"
          " (logit std %.3g)" % (spec[:6], err, rms, nerr, nrms, float(ref.std())))
    assert err <= NOISE_FACTOR * nerr and rms <= NOISE_FACTOR * nrms, (err, rms, nerr, nrms)


def test_8b_shaped_full_depth_logits(dev):
    # the benchmark's launch configuration: a batch of 512 windows of 1024 tokens; 8 rows of window 1
    _full_depth_logits(C4, 512, 1024, 7, 1, 508, 8)


def test_7b_gqa_shaped_full_depth_logits(dev):
    # windows of 512 (the float64 oracle over a 2048-token window takes minutes); 16 rows of window 0
    _full_depth_logits(C5, 64, 512, 8, 0, 240, 16)


def test_8b_shaped_roundtrip(dev):
    d = dlmz()
    nl, dm, nh, nkv, F, V, _ = C4
    m = d.Model(nl, dm, nh, nkv, F, V, d.BF16, seed=9)
    data = sources.tokens_to_bytes(sources.zipf_bigram_tokens(2 * 1024 + 100, V, seed=9))
    pol = d.policy(d.TOPK_CONF, 16, 0)
    blob = m.compress(data, 1024, pol)
    assert m.decompress(blob) == data
    bits_per_token = 8.0 * len(blob) / (len(data) // 4)
    # random-init model: log2(V) = 16.95 bits plus the cross-entropy excess of random logits of
    # std 0.02 sqrt(d) = 1.28 (about 1.3 bits)
    assert 16.9 < bits_per_token < 19.5
    # candidate logits in slabs (the budget holds 4096 rows): the same file
    m.set_logits_budget(4096 * V * 4)
    assert m.compress(data, 1024, pol) == blob
    assert m.decompress(blob) == data
    m.close()


def test_7b_gqa_shaped_roundtrip(dev):
    d = dlmz()
    nl, dm, nh, nkv, F, V, _ = C5
    m = d.Model(nl, dm, nh, nkv, F, V, d.BF16, seed=10)
    # a short prefix: one tail window of 384 tokens of the 2048-token windowing
    data = sources.tokens_to_bytes(sources.zipf_bigram_tokens(384, V, seed=10))
    pol = d.policy(d.ENTROPY, 0, 0, 0.5, 1, 64)
    blob = m.compress(data, 2048, pol)
    assert m.decompress(blob) == data
    m.set_logits_budget(100 * V * 4)
    assert m.compress(data, 2048, pol) == blob
    m.close()
