"""GPU masked-DLM forward (Definition 3) vs the oracle forward.

Tolerances: max |logit error| <= 1e-4 for float32 models and <= 2e-2 for
bf16 models, on the same seeded weights and states.
"""
import numpy as np
import pytest

from oracle import model as OM
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu

MODELS = [
    # (n_layers, d, heads, kv, ffn, V, dtype, L, nc, row0, rpc)   -- path exercised
    (2, 64, 4, 2, 96, 37, "f32", 40, 3, 0, 40),          # CUDA-core GEMM + attention, GQA, hd 16
    (2, 128, 4, 4, 512, 256, "f32", 100, 2, 64, 36),     # tiny byte model shape (hd 32), ragged row window
    (1, 48, 3, 1, 40, 11, "bf16", 20, 2, 5, 10),         # bf16 on CUDA cores (odd shapes)
    (2, 256, 4, 4, 256, 256, "bf16", 192, 3, 0, 192),    # tcgen05 GEMMs (RoPE/SwiGLU/residual epilogues), mma attention hd 64
    (2, 512, 4, 2, 512, 512, "bf16", 130, 2, 2, 128),    # tcgen05 + GQA, hd 128, ragged window (130)
    (1, 256, 8, 1, 384, 300, "bf16", 77, 2, 0, 77),      # 8:1 GQA hd 32, LM head on CUDA cores (V = 300)
    (2, 256, 4, 2, 256, 256, "bf16", 256, 2, 0, 256),    # tcgen05 attention (L % 128 == 0, hd 64), GQA 2:1
    (2, 512, 8, 8, 512, 256, "bf16", 512, 2, 128, 128),  # byte-workload head shape: L 512, hd 64, block rows
    (1, 256, 4, 2, 256, 256, "bf16", 256, 80, 0, 256),   # 640 attention work items: persistent CTAs take 2-3 each
]


@pytest.mark.parametrize("mi", range(len(MODELS)))
def test_forward_matches_oracle(dev, mi):
    import torch
    d = dlmz()
    nl, dm, nh, nkv, F, V, dt, L, nc, row0, rpc = MODELS[mi]
    m = d.Model(nl, dm, nh, nkv, F, V, d.BF16 if dt == "bf16" else d.FP32, seed=11 + mi)
    rng = np.random.default_rng(mi)
    state = rng.integers(0, V + 1, (nc, L)).astype(np.int32)
    state[:, rng.random(L) < 0.3] = V  # masked columns
    logits = torch.empty(nc * rpc, V, dtype=torch.float32, device="cuda")
    m.forward_logits(ptr(to_dev(state)), nc, L, row0, rpc, ptr(logits))
    d.check()
    got = logits.cpu().numpy().reshape(nc, rpc, V)
    w = OM.Weights(OM.ModelConfig(nl, dm, nh, nkv, F, V, dt, seed=11 + mi))
    tol = 2e-2 if dt == "bf16" else 1e-4
    for c in range(nc):
        ref = OM.forward(w, state[c], rows=np.arange(row0, row0 + rpc))
        err = np.max(np.abs(got[c] - ref))
        assert err <= tol, (c, err)


def test_gemm_tensor_core_vs_float64(dev):
    import torch
    d = dlmz()
    rng = np.random.default_rng(3)
    # the last two cases give each persistent CTA several tiles, so both accumulators and every
    # ring stage turn over many times
    for (M, N, K) in [(128, 256, 64), (300, 512, 192), (1000, 768, 512), (77, 256, 2048), (8192, 2048, 256),
                      (2560, 1280, 1024)]:
        A = torch.from_numpy(rng.normal(size=(M, K)).astype(np.float32)).to(torch.bfloat16)
        B = torch.from_numpy(rng.normal(size=(N, K)).astype(np.float32)).to(torch.bfloat16)
        ref = A.double() @ B.double().T
        Ad, Bd = A.cuda(), B.cuda()
        D = torch.empty(M, N, dtype=torch.float32, device="cuda")
        d.gemm_bf16(ptr(Ad), ptr(Bd), ptr(D), M, N, K)
        d.check()
        err = (D.cpu().double() - ref).abs().max().item()
        assert err <= 1e-3 * np.sqrt(K), (M, N, K, err)


def test_forward_is_batch_invariant(dev):
    """A window's logits do not depend on the other windows of the batch."""
    import torch
    d = dlmz()
    m = d.Model(2, 256, 4, 4, 256, 256, d.BF16, seed=3)
    rng = np.random.default_rng(9)
    L = 128
    state = rng.integers(0, 257, (5, L)).astype(np.int32)
    big = torch.empty(5 * L, 256, dtype=torch.float32, device="cuda")
    m.forward_logits(ptr(to_dev(state)), 5, L, 0, L, ptr(big))
    one = torch.empty(L, 256, dtype=torch.float32, device="cuda")
    m.forward_logits(ptr(to_dev(state[3:4])), 1, L, 0, L, ptr(one))
    d.check()
    assert torch.equal(big[3 * L:4 * L], one)
