"""Pins for the oracle forward pass (Definition 3): closed forms and library routines."""
import numpy as np
import pytest
import scipy.special

from oracle import model as M
from oracle import weights as W

TINY = M.ModelConfig(n_layers=2, d=32, n_heads=4, n_kv_heads=2, ffn=48, vocab=11, dtype="f32", seed=7)


def _weights(cfg=TINY):
    return M.Weights(cfg)


def test_attention_matches_torch_sdpa():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(1)
    L, H, Hkv, hd = 9, 4, 2, 8
    q = rng.normal(size=(L, H * hd))
    k = rng.normal(size=(L, Hkv * hd))
    v = rng.normal(size=(L, Hkv * hd))
    out = M.attention(q, k, v, H, Hkv, hd)
    tq = torch.from_numpy(q).view(L, H, hd).transpose(0, 1)
    tk = torch.from_numpy(k).view(L, Hkv, hd).transpose(0, 1).repeat_interleave(H // Hkv, 0)
    tv = torch.from_numpy(v).view(L, Hkv, hd).transpose(0, 1).repeat_interleave(H // Hkv, 0)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=False)
    ref = ref.transpose(0, 1).reshape(L, H * hd).numpy()
    assert np.allclose(out, ref, atol=1e-12, rtol=1e-10)


def test_attention_uniform_when_scores_vanish():
    rng = np.random.default_rng(2)
    L, hd = 7, 4
    v = rng.normal(size=(L, hd))
    out = M.attention(np.zeros((L, hd)), rng.normal(size=(L, hd)), v, 1, 1, hd)
    assert np.allclose(out, np.broadcast_to(v.mean(0), (L, hd)))


def test_attention_single_position_returns_value():
    rng = np.random.default_rng(3)
    v = rng.normal(size=(1, 6))
    assert np.allclose(M.attention(rng.normal(size=(1, 6)), rng.normal(size=(1, 6)), v, 1, 1, 6), v)


def test_attention_sees_later_positions():
    # bidirectional: the first query attends to a key placed after it
    L, hd = 5, 2
    q = np.zeros((L, hd)); q[0] = [50.0, 0.0]
    k = np.zeros((L, hd)); k[4] = [50.0, 0.0]
    v = np.arange(L * hd, dtype=np.float64).reshape(L, hd)
    out = M.attention(q, k, v, 1, 1, hd)
    assert np.allclose(out[0], v[4], atol=1e-6)


def test_rope_equals_complex_rotation():
    rng = np.random.default_rng(4)
    L, H, hd, theta = 6, 2, 8, 500.0
    u = rng.normal(size=(L, H * hd))
    out = M.rope(u, H, hd, theta).reshape(L, H, hd)
    half = hd // 2
    z = u.reshape(L, H, hd)[..., :half] + 1j * u.reshape(L, H, hd)[..., half:]
    freq = theta ** (-np.arange(half) * 2.0 / hd)
    rot = np.exp(1j * np.arange(L)[:, None, None] * freq[None, None, :])
    ref = z * rot
    assert np.allclose(out[..., :half], ref.real)
    assert np.allclose(out[..., half:], ref.imag)


def test_rope_relative_position():
    rng = np.random.default_rng(5)
    hd = 16
    a, b = rng.normal(size=hd), rng.normal(size=hd)
    u = np.zeros((12, hd)); w = np.zeros((12, hd))
    u[3] = a; w[1] = b; u[9] = a; w[7] = b
    ru, rw = M.rope(u, 1, hd, 10000.0), M.rope(w, 1, hd, 10000.0)
    assert np.isclose(ru[3] @ rw[1], ru[9] @ rw[7])
    assert np.allclose(np.linalg.norm(ru, axis=1), np.linalg.norm(u, axis=1))


def test_rmsnorm_and_silu():
    rng = np.random.default_rng(6)
    x = rng.normal(size=(5, 32)) * 3
    y = M.rmsnorm(x, np.ones(32), 0.0)
    assert np.allclose(np.sqrt((y * y).mean(1)), 1.0)
    assert np.allclose(M.rmsnorm(7 * x, np.ones(32), 0.0), y)
    t = np.linspace(-8, 8, 101)
    assert np.allclose(M.silu(t), t * scipy.special.expit(t))


def test_layers_vanish_when_output_projections_are_zero():
    # Wo = Wdown = 0 => x stays E[s] => logits = head(RMSNorm(E[s]))
    w = _weights()
    for l in range(TINY.n_layers):
        w.t[M.layer_tid(l, M.WO)] = np.zeros_like(w.layer(l, M.WO))
        w.t[M.layer_tid(l, M.WDOWN)] = np.zeros_like(w.layer(l, M.WDOWN))
    s = np.array([0, 3, 11, 11, 5, 10])
    got = M.forward(w, s)
    e = w.embed[s]
    h = e / np.sqrt((e * e).mean(1, keepdims=True) + TINY.norm_eps)
    ref = (h.astype(np.float32).astype(np.float64) @ w.head.T).astype(np.float32)
    assert np.allclose(got, ref, atol=1e-6)


def test_permutation_equivariance_without_rope():
    # with all rotary frequencies zero, a bidirectional model is permutation
    # equivariant; a causal mask would break this
    cfg = M.ModelConfig(**{**TINY.__dict__, "rope_theta": float("inf")})
    w = M.Weights(cfg)
    s = np.array([1, 4, 11, 2, 11, 9, 0])
    perm = np.array([3, 0, 6, 1, 5, 2, 4])
    a = M.forward(w, s)
    b = M.forward(w, s[perm])
    assert np.allclose(a[perm], b, atol=1e-5)


def test_rope_breaks_permutation_equivariance():
    w = _weights()
    s = np.array([1, 4, 11, 2, 11, 9, 0])
    perm = np.array([3, 0, 6, 1, 5, 2, 4])
    assert not np.allclose(M.forward(w, s)[perm], M.forward(w, s[perm]), atol=1e-5)


def test_gqa_equals_mha_with_repeated_kv():
    gqa = _weights()
    mha_cfg = M.ModelConfig(**{**TINY.__dict__, "n_kv_heads": TINY.n_heads})
    t = dict(gqa.t)
    hd, g = TINY.head_dim, TINY.n_heads // TINY.n_kv_heads
    for l in range(TINY.n_layers):
        for which in (M.WK, M.WV):
            wk = gqa.layer(l, which).reshape(TINY.n_kv_heads, hd, TINY.d)
            t[M.layer_tid(l, which)] = np.repeat(wk, g, axis=0).reshape(TINY.n_heads * hd, TINY.d)
    mha = M.Weights(mha_cfg, tensors=t)
    s = np.array([3, 11, 11, 0, 7, 2])
    assert np.allclose(M.forward(gqa, s), M.forward(mha, s), atol=1e-6)


def test_value_path_orientation():
    # Wq = Wk = 0 (uniform attention), one layer, Wgate = 0 (FFN adds 0):
    # x_out = x + mean_rows(v) Wo^T with v = h Wv^T; checks that Wv and Wo are
    # applied as [out x in] matrices.
    cfg = M.ModelConfig(n_layers=1, d=8, n_heads=2, n_kv_heads=2, ffn=8, vocab=5, dtype="f32",
                        rope_theta=10000.0)
    w = M.Weights(cfg)
    rng = np.random.default_rng(8)
    w.t[M.layer_tid(0, M.WQ)] = np.zeros((8, 8))
    w.t[M.layer_tid(0, M.WK)] = np.zeros((8, 8))
    w.t[M.layer_tid(0, M.WGATE)] = np.zeros((8, 8))
    wv = W.round_f32(rng.normal(size=(8, 8)))
    wo = W.round_f32(rng.normal(size=(8, 8)))
    w.t[M.layer_tid(0, M.WV)] = wv
    w.t[M.layer_tid(0, M.WO)] = wo
    s = np.array([0, 1, 2, 5, 4])
    x = w.embed[s]
    h = x / np.sqrt((x * x).mean(1, keepdims=True) + cfg.norm_eps)
    v = np.einsum("oi,li->lo", wv, h)
    xo = x + np.einsum("oi,i->o", wo, v.mean(0))[None, :]
    hf = xo / np.sqrt((xo * xo).mean(1, keepdims=True) + cfg.norm_eps)
    assert np.allclose(M.hidden(w, s), hf, atol=1e-5)


def test_bf16_model_rounds_storage():
    cfg = M.ModelConfig(**{**TINY.__dict__, "dtype": "bf16"})
    w = M.Weights(cfg)
    assert np.array_equal(W.round_bf16(w.embed), w.embed)
    h = M.hidden(w, np.array([1, 2, 11, 3]))
    assert np.array_equal(W.round_bf16(h), h)
    a = M.forward(w, np.array([1, 2, 11, 3]))
    b = M.forward(_weights(), np.array([1, 2, 11, 3]))
    assert np.max(np.abs(a - b)) < 2e-2  # bf16 storage vs float32 storage of the same draws


def _torch_block_forward(cfg, t, state, bf16=False):
    """Definition 3's LLaDA-style block restated with PyTorch float64 CPU library calls.

    Written from the block definition (pre-norm RMSNorm, rotary embedding as a
    complex rotation of the pairs (i, i + hd/2), grouped-query attention via
    scaled_dot_product_attention without a mask, SwiGLU = silu(gate) * up,
    residual adds, final RMSNorm, untied head), not from oracle/model.py.  A
    tensor the model stores is rounded to float32 (torch's own conversion).
    ``bf16``: the bf16 storage points instead -- the residual stays float32,
    the projections read bfloat16(x) and their results are scaled by the
    RMSNorm factor of x (the norm as a row scale), q/k after RoPE, v, the
    attention output, the SwiGLU product and the final normed rows are
    bfloat16 (torch's conversion through float32).
    """
    import torch
    import torch.nn.functional as F

    f64 = torch.float64
    st = lambda a: a.to(torch.float32).to(f64)
    sb = (lambda a: a.to(torch.float32).to(torch.bfloat16).to(f64)) if bf16 else st
    T = {k: torch.from_numpy(np.asarray(v, dtype=np.float64)) for k, v in t.items()}
    hd, L = cfg.d // cfg.n_heads, len(state)
    idx = torch.as_tensor(np.asarray(state), dtype=torch.long)

    def norm(x):
        return x * torch.rsqrt((x * x).mean(-1, keepdim=True) + cfg.norm_eps)

    half = hd // 2
    inv = float(cfg.rope_theta) ** (-torch.arange(half, dtype=f64) * 2.0 / hd)
    rot = torch.polar(torch.ones(L, half, dtype=f64), torch.arange(L, dtype=f64)[:, None] * inv[None, :])

    def rope(u, nh):
        u = u.view(L, nh, hd)
        z = torch.complex(u[..., :half], u[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], -1).reshape(L, nh * hd)

    x = st(T[M.TID_EMBED][idx])
    g = cfg.n_heads // cfg.n_kv_heads
    def proj(x, which):  # the normed projection: norm(x) W^T, or with bf16 storage bf16(x) W^T * scale
        if not bf16:
            return F.linear(st(norm(x)), which)
        return F.linear(sb(x), which) * torch.rsqrt((x * x).mean(-1, keepdim=True) + cfg.norm_eps)

    for l in range(cfg.n_layers):
        P = lambda which: T[M.layer_tid(l, which)]
        q = sb(rope(proj(x, P(M.WQ)), cfg.n_heads)).view(L, cfg.n_heads, hd).transpose(0, 1)
        k = sb(rope(proj(x, P(M.WK)), cfg.n_kv_heads)).view(L, cfg.n_kv_heads, hd).transpose(0, 1)
        v = sb(proj(x, P(M.WV))).view(L, cfg.n_kv_heads, hd).transpose(0, 1)
        o = F.scaled_dot_product_attention(q, k.repeat_interleave(g, 0), v.repeat_interleave(g, 0), is_causal=False)
        x = st(x + F.linear(sb(o.transpose(0, 1).reshape(L, cfg.d)), P(M.WO)))
        a = sb(F.silu(proj(x, P(M.WGATE))) * proj(x, P(M.WUP)))
        x = st(x + F.linear(a, P(M.WDOWN)))
    return st(F.linear(sb(norm(x)), T[M.TID_HEAD])).numpy()


def test_forward_matches_independent_torch_block():
    # nonzero gate and up weights large enough that SiLU is far from x/2 (with
    # N(0, 0.02) weights silu(g) u ~ g u / 2 is nearly symmetric in g and u, so a
    # gate/up swap would hide); GQA, RoPE and two layers exercise the whole block
    pytest.importorskip("torch")
    cfg = M.ModelConfig(n_layers=2, d=32, n_heads=4, n_kv_heads=2, ffn=48, vocab=11, dtype="f32", seed=3)
    rng = np.random.default_rng(21)
    t = {tid: W.round_f32(rng.normal(scale=0.4 if tid >= 2 else 1.0, size=shp))
         for tid, shp in M.tensor_shapes(cfg).items()}
    w = M.Weights(cfg, tensors=t)
    s = np.array([3, 11, 0, 7, 11, 2, 10, 5, 11])
    ours = M.forward(w, s)
    ref = _torch_block_forward(cfg, t, s)
    assert np.max(np.abs(ours - ref)) <= 1e-4 * max(1.0, np.max(np.abs(ref)))
    # the SwiGLU is asymmetric at this scale: exchanging the gate and up weights moves the logits
    t2 = dict(t)
    for l in range(cfg.n_layers):
        t2[M.layer_tid(l, M.WGATE)], t2[M.layer_tid(l, M.WUP)] = t[M.layer_tid(l, M.WUP)], t[M.layer_tid(l, M.WGATE)]
    assert np.max(np.abs(_torch_block_forward(cfg, t2, s) - ref)) > 1e-1


def test_bf16_forward_matches_independent_torch_block():
    # the bf16 storage points (the projections read bf16(x), the norm scales their results)
    pytest.importorskip("torch")
    cfg = M.ModelConfig(n_layers=2, d=32, n_heads=4, n_kv_heads=2, ffn=48, vocab=11, dtype="bf16", seed=3)
    rng = np.random.default_rng(23)
    t = {tid: W.round_bf16(rng.normal(scale=0.4 if tid >= 2 else 1.0, size=shp))
         for tid, shp in M.tensor_shapes(cfg).items()}
    w = M.Weights(cfg, tensors=t)
    s = np.array([3, 11, 0, 7, 11, 2, 10, 5, 11])
    ours = M.forward(w, s)
    ref = _torch_block_forward(cfg, t, s, bf16=True)
    print("bf16 oracle vs torch restatement: max-abs %.3g" % np.max(np.abs(ours - ref)))
    assert np.max(np.abs(ours - ref)) <= 1e-4 * max(1.0, np.max(np.abs(ref)))


def test_ffn_closed_form_single_layer():
    # one layer with Wv = 0 (attention adds nothing): the block output is
    # x + (silu(h Wg^T) * (h Wu^T)) Wd^T with h = RMSNorm(x), x = E[s], written out per element
    cfg = M.ModelConfig(n_layers=1, d=8, n_heads=2, n_kv_heads=2, ffn=6, vocab=5, dtype="f32")
    rng = np.random.default_rng(22)
    w = M.Weights(cfg)
    wg = W.round_f32(rng.normal(scale=0.8, size=(6, 8)))
    wu = W.round_f32(rng.normal(scale=0.8, size=(6, 8)))
    wd = W.round_f32(rng.normal(scale=0.8, size=(8, 6)))
    w.t[M.layer_tid(0, M.WV)] = np.zeros((8, 8))
    w.t[M.layer_tid(0, M.WGATE)] = wg
    w.t[M.layer_tid(0, M.WUP)] = wu
    w.t[M.layer_tid(0, M.WDOWN)] = wd
    s = np.array([4, 0, 5, 2])
    want = np.empty((len(s), 8))
    for r, sym in enumerate(s):
        x = [float(e) for e in w.embed[sym]]
        ms = sum(e * e for e in x) / 8
        h = [e / (ms + cfg.norm_eps) ** 0.5 for e in x]
        a = []
        for f in range(6):
            gf = sum(h[i] * wg[f, i] for i in range(8))
            uf = sum(h[i] * wu[f, i] for i in range(8))
            a.append(gf / (1.0 + np.exp(-gf)) * uf)
        xo = [x[o] + sum(a[f] * wd[o, f] for f in range(6)) for o in range(8)]
        ms = sum(e * e for e in xo) / 8
        want[r] = [e / (ms + cfg.norm_eps) ** 0.5 for e in xo]
    assert np.allclose(M.hidden(w, s), want, atol=1e-5)
