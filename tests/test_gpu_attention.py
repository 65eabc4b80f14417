"""GPU bidirectional attention (Definition 3) through dlmz_attention_bf16 vs the oracle.

Inputs are bf16-rounded on the host and the oracle's float64 attention runs on
the same rounded values.  "drift" inputs make the scores grow (or shrink) along
the key positions by about 20 log2 units per window, so the tensor-core
kernel's running maximum is raised (and O rescaled) across 128-key tiles in the
growing windows and never in the shrinking ones; "flat" inputs keep every score
small.

Tolerance: |out - ref| <= 1e-2 max|v|.  The bf16 output rounds by up to 2^-9
relative; on the tensor cores P is an f16 value of ex2.approx (relative error
about 2^-10) and the row sum adds those f16 values in a pairwise f16 tree (7
roundings of 2^-11 at most); V is converted from bf16 to f16 exactly.
"""
import numpy as np
import pytest

from oracle import model as OM
from tests.gpu_helpers import dlmz, ptr

pytestmark = pytest.mark.gpu

CASES = [
    # (L, windows, heads, kv heads, head_dim, inputs)   -- path exercised
    (128, 200, 4, 2, 64, "drift"),   # tcgen05: one key tile per item, 800 items (2-3 per persistent CTA)
    (1024, 2, 4, 4, 64, "drift"),    # tcgen05: 8 key tiles per item, running max raised across tiles
    (512, 3, 8, 1, 64, "drift"),     # tcgen05: 8:1 GQA
    (256, 2, 4, 2, 64, "flat"),      # tcgen05: small scores
    (1024, 2, 32, 32, 128, "drift"), # tcgen05 head_dim 128: the 8B-shaped MHA (32 heads) at windows of 1024
    (2048, 1, 28, 4, 128, "drift"),  # tcgen05 head_dim 128: the 7B-shaped 7:1 GQA at windows of 2048
    (256, 3, 8, 2, 128, "flat"),     # tcgen05 head_dim 128: small scores, 4:1 GQA
    (128, 160, 2, 1, 128, "drift"),  # tcgen05 head_dim 128: 320 one-tile items, ~2 per persistent CTA
    (256, 400, 2, 1, 64, "drift"),   # tcgen05 one-tile kernel: 1600 items, ~5 per persistent CTA
    (512, 160, 2, 2, 128, "drift"),  # tcgen05 head_dim 128, two query tiles per CTA: 640 items of 4 key tiles
    (96, 2, 4, 2, 64, "drift"),      # CUDA-core mma kernel (L % 128 != 0)
    (64, 2, 2, 1, 128, "drift"),     # CUDA-core mma kernel, head_dim 128
    (40, 3, 4, 2, 32, "drift"),      # CUDA-core scalar kernel, head_dim 32
]


def _inputs(rng, L, nc, nh, nkv, hd, kind):
    q = rng.normal(0.0, 0.5, (nc, L, nh, hd))
    k = rng.normal(0.0, 0.5, (nc, L, nkv, hd))
    v = rng.normal(0.0, 1.0, (nc, L, nkv, hd))
    if kind == "drift":
        u = rng.normal(size=(nkv, hd))
        u /= np.linalg.norm(u, axis=1, keepdims=True)
        grow = 40.0 * np.arange(L) / L  # per-key magnitude along u
        for w in range(nc):
            g = grow if w % 2 == 0 else grow[::-1]
            k[w] += g[:, None, None] * u[None]
            q[w] += 3.0 * np.repeat(u, nh // nkv, axis=0)[None]
    else:
        q *= 0.6
        k *= 0.6
    return q, k, v


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_attention_matches_oracle(dev, ci):
    import torch
    d = dlmz()
    L, nc, nh, nkv, hd, kind = CASES[ci]
    rng = np.random.default_rng(100 + ci)
    q, k, v = _inputs(rng, L, nc, nh, nkv, hd, kind)
    width = (nh + 2 * nkv) * hd
    ld = width + 8  # a row pitch wider than the heads
    rows = np.zeros((nc * L, ld), dtype=np.float32)
    rows[:, :nh * hd] = q.reshape(nc * L, nh * hd)
    rows[:, nh * hd:(nh + nkv) * hd] = k.reshape(nc * L, nkv * hd)
    rows[:, (nh + nkv) * hd:width] = v.reshape(nc * L, nkv * hd)
    rows_bf = torch.from_numpy(rows).to(torch.bfloat16)
    rounded = rows_bf.double().numpy()
    out = torch.empty(nc * L, nh * hd, dtype=torch.bfloat16, device="cuda")
    d.attention_bf16(ptr(rows_bf.cuda()), ld, nc, L, nh, nkv, hd, ptr(out))
    d.check()
    got = out.double().cpu().numpy().reshape(nc, L, nh * hd)
    vmax = np.abs(rounded[:, (nh + nkv) * hd:width]).max()
    for w in range(nc):
        r = rounded[w * L:(w + 1) * L]
        ref = OM.attention(r[:, :nh * hd], r[:, nh * hd:(nh + nkv) * hd], r[:, (nh + nkv) * hd:width], nh, nkv, hd)
        err = np.abs(got[w] - ref).max()
        assert err <= 1e-2 * vmax, (w, err, vmax)


def test_attention_rejects_bad_shapes(dev):
    import torch
    d = dlmz()
    buf = torch.zeros(256, 512, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(256, 256, dtype=torch.bfloat16, device="cuda")
    for args in [(512, 2, 128, 4, 3, 64),    # n_heads not a multiple of n_kv_heads
                 (256, 2, 128, 4, 2, 64),    # ld below (n_heads + 2 n_kv_heads) head_dim
                 (516, 2, 128, 4, 2, 64),    # ld not a multiple of 8
                 (512, 2, 128, 4, 2, 12),    # head_dim not a multiple of 8
                 (512, 2, 128, 2, 2, 256)]:  # head_dim above 128
        with pytest.raises(d.DlmzError) as e:
            d.attention_bf16(ptr(buf), *args, ptr(out))
        assert e.value.code == d.EINVAL, args
