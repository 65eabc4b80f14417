"""GPU attention-based initial context (Sec. 3.4, policy 4) vs the oracle.

The scores come from floating-point attention maps, so they are compared
within a tolerance: float32 models 1e-4 relative, bf16 models 2e-2 relative
(the forward's bf16 storage moves q and k by a few ulps per layer; the same
2e-2 the logits get).  The chosen positions may then differ from the oracle's
only where the oracle's own scores are within that tolerance of its c-th best.
"""
import numpy as np
import pytest

from oracle import container as OC
from oracle import context as OX
from oracle import model as OM
from oracle import pipeline as OP
from oracle import selector as S
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu

MODELS = [
    # spec, L, windows, relative tolerance
    ((2, 64, 4, 2, 96, 37, "f32"), 40, 3, 1e-4),             # CUDA-core path, GQA, hd 16
    ((2, 256, 4, 4, 256, 256, "bf16"), 128, 3, 2e-2),        # tensor-core GEMMs + attention (hd 64)
    ((1, 512, 8, 8, 512, 256, "bf16"), 512, 2, 2e-2),        # byte-workload shape (one layer)
]


def _model(d, spec, seed):
    nl, dm, h, kv, F, V, dt = spec
    return d.Model(nl, dm, h, kv, F, V, d.BF16 if dt == "bf16" else d.FP32, seed=seed)


@pytest.mark.parametrize("mi", range(len(MODELS)))
def test_scores_match_oracle(dev, mi):
    import torch
    d = dlmz()
    spec, L, nc, tol = MODELS[mi]
    m = _model(d, spec, 20 + mi)
    sym = np.random.default_rng(mi).integers(0, spec[5], (nc, L)).astype(np.int32)
    scores = torch.empty(nc, L, dtype=torch.float32, device="cuda")
    m.context_scores(ptr(to_dev(sym)), nc, L, ptr(scores))
    d.check()
    got = scores.cpu().numpy()
    w = OM.Weights(OM.ModelConfig(*spec, seed=20 + mi))
    for c in range(nc):
        ref = OX.attention_scores(w, sym[c])
        err = np.max(np.abs(got[c] - ref)) / np.mean(ref)
        assert err <= tol, (c, err)


CASES = [
    ((2, 64, 4, 2, 96, 37, "f32"), "bytes", 40, 3, S.Policy(kind=S.UNIFORM, k=8), 1e-4),      # V <= 256: bytes
    ((1, 64, 4, 2, 96, 5000, "f32"), "tokens", 40, 4, S.Policy(kind=S.ENTROPY, tau_bits=0.5), 1e-4),
    ((2, 256, 4, 4, 256, 256, "bf16"), "bytes", 128, 6, S.Policy(kind=S.TOPK_CONF, k=8, block=64), 2e-2),
]


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_compress_with_attention_context(dev, ci):
    d = dlmz()
    spec, kind, L, c, opol, tol = CASES[ci]
    m = _model(d, spec, 30 + ci)
    V = spec[5]
    rng = np.random.default_rng(ci)
    if kind == "bytes":
        sym = rng.integers(0, V, 3 * L + 17)
        data = sym.astype(np.uint8).tobytes()
    else:
        sym = rng.integers(0, V, 3 * L + 17)
        data = sym.astype("<u4").tobytes()
    pol = d.policy(opol.kind, opol.k, opol.block, context=d.CONTEXT_ATTENTION, context_c=c)
    blob = m.compress(data, L, pol)
    assert m.decompress(blob) == data
    h, _ = OC.read(blob)
    assert h.ctx_kind == 3 and h.ctx_c == c
    pos = np.frombuffer(h.ctx_pos, dtype="<u4").astype(np.int64)
    w = OM.Weights(OM.ModelConfig(*spec, seed=30 + ci))
    used = 0
    for win in range(h.n_chunks):
        ws = sym[win * L:(win + 1) * L]
        ce = min(c, ws.size)
        p = pos[used:used + ce]
        used += ce
        assert np.all(np.diff(p) > 0) and p.max() < ws.size
        ref = OX.attention_scores(w, ws)
        cth = np.sort(ref)[::-1][ce - 1]
        assert ref[p].min() >= cth - tol * np.mean(ref), win  # near-ties may swap, nothing else
    oblob = OP.compress(w, data, L, opol, context=(OX.ATTENTION, c, 0))
    assert abs(len(blob) - len(oblob)) <= 0.005 * len(oblob) + 8, (len(blob), len(oblob))
    bad = bytearray(blob)
    bad[80:84] = (L + 5).to_bytes(4, "little")  # a stored position outside its window
    with pytest.raises(d.DlmzError) as e:
        m.decompress(bytes(bad))
    assert e.value.code == d.ECORRUPT
