"""Masked, bidirectional diffusion-LM forward pass (oracle side).

Definition 3 (Sec. 3.1): a masked DLM maps a partially observed window
S~ over Sigma u {[MASK]} to one distribution over Sigma for every masked
position, in a single forward pass, and each masked position attends to all
positions regardless of order (no causal mask).

The paper fixes only "masked, bidirectional, LLaDA backbone" (Sec. 1,
Sec. 4).  The block used here is a LLaDA-style pre-norm transformer:

    x = E[s]                                     (E has V+1 rows, row V = [MASK])
    per layer:
        h = RMSNorm(x) * g_attn
        q, k, v = h Wq^T, h Wk^T, h Wv^T          (GQA: n_kv_heads <= n_heads)
        q, k = RoPE(q), RoPE(k)                   (rotate-half pairs (i, i+hd/2))
        o_h = softmax(q_h k_g^T / sqrt(hd)) v_g   (every position, no mask)
        x = x + concat(o_h) Wo^T
        h = RMSNorm(x) * g_ffn
        x = x + (SiLU(h Wg^T) * (h Wu^T)) Wd^T
    logits = (RMSNorm(x) * g_final) Whead^T       (V outputs: Sigma only)

Weights are stored [out x in] (row = one output feature).  Arithmetic is
float64; a tensor that the model stores between operations is rounded to
its storage dtype at that point:

* bf16 models: weights, E, the projection inputs, q/k/v after RoPE, the
  attention output, the SwiGLU product and the LM-head input are bfloat16;
  the residual stream x and the logits are float32.
* f32 models: every stored tensor is float32.

The RMSNorm in front of the QKV and gate/up projections is applied as a row
scale of the projection's result (mathematically the same block): the
projection reads x g rounded to the storage dtype and its float result is
multiplied by 1 / sqrt(mean(x^2) + eps) of the float32 residual x, before
RoPE and SiLU.  The final RMSNorm in front of the LM head is applied to x
directly and its result stored.  (The paper fixes no precision; these
storage points are the reading both implementations follow.)

Parity: pinned by closed forms (uniform attention when Wq = Wk = 0,
logits = head(norm(E[s])) when Wo = Wd = 0, permutation equivariance with
RoPE frequencies set to zero, GQA == MHA with repeated KV heads, RoPE
relative-position identity, single-position attention == V).  Against the
paper's trained LLaDA numbers parity is unpinned (no weights exist here).
"""
from dataclasses import dataclass

import numpy as np

from . import weights as W


@dataclass(frozen=True)
class ModelConfig:
    n_layers: int
    d: int
    n_heads: int
    n_kv_heads: int
    ffn: int
    vocab: int
    dtype: str = "bf16"  # 'f32' | 'bf16'
    rope_theta: float = 10000.0
    norm_eps: float = 1e-5
    seed: int = 0

    @property
    def head_dim(self):
        return self.d // self.n_heads

    @property
    def mask_id(self):
        return self.vocab


# Tensor ids of the counter-based generator (part of the model definition).
TID_EMBED = 0
TID_HEAD = 1
WQ, WK, WV, WO, WGATE, WUP, WDOWN = range(7)


def layer_tid(layer, which):
    return 2 + 8 * layer + which


def tensor_shapes(cfg):
    """Logical shapes, keyed by tensor id."""
    hd = cfg.head_dim
    dkv = cfg.n_kv_heads * hd
    shapes = {TID_EMBED: (cfg.vocab + 1, cfg.d), TID_HEAD: (cfg.vocab, cfg.d)}
    for l in range(cfg.n_layers):
        shapes[layer_tid(l, WQ)] = (cfg.d, cfg.d)
        shapes[layer_tid(l, WK)] = (dkv, cfg.d)
        shapes[layer_tid(l, WV)] = (dkv, cfg.d)
        shapes[layer_tid(l, WO)] = (cfg.d, cfg.d)
        shapes[layer_tid(l, WGATE)] = (cfg.ffn, cfg.d)
        shapes[layer_tid(l, WUP)] = (cfg.ffn, cfg.d)
        shapes[layer_tid(l, WDOWN)] = (cfg.d, cfg.ffn)
    return shapes


class _LazyTensors:
    """Tensors generated on first use (by the C restatement of the draws) for
    full-size models: the embedding and the head are kept, layer tensors only
    while their layer is the most recent one asked for, so a forward over 32
    layers of an 8B-shaped model holds one layer at a time."""

    def __init__(self, cfg):
        self.cfg = cfg
        self.shapes = tensor_shapes(cfg)
        self.keep = {}
        self.layer = {}
        self.layer_id = None

    def __getitem__(self, tid):
        if tid in self.keep:
            return self.keep[tid]
        if tid in (TID_EMBED, TID_HEAD):
            self.keep[tid] = W.init_tensor_c(self.cfg.seed, tid, self.shapes[tid], self.cfg.dtype)
            return self.keep[tid]
        l = (tid - 2) // 8
        if l != self.layer_id:
            self.layer, self.layer_id = {}, l
        if tid not in self.layer:
            self.layer[tid] = W.init_tensor_c(self.cfg.seed, tid, self.shapes[tid], self.cfg.dtype)
        return self.layer[tid]


class Weights:
    """All parameters of a model as float64 arrays holding storage-dtype values.

    ``lazy``: tensors are generated when first used, one layer at a time (for the
    full-size models; needs oracle/build.py's liboracle.so)."""

    def __init__(self, cfg, tensors=None, lazy=False):
        self.cfg = cfg
        shapes = tensor_shapes(cfg)
        if tensors is None:
            tensors = (_LazyTensors(cfg) if lazy else
                       {tid: W.init_tensor(cfg.seed, tid, shp, cfg.dtype) for tid, shp in shapes.items()})
        self.t = tensors
        self.g_attn = [np.ones(cfg.d) for _ in range(cfg.n_layers)]
        self.g_ffn = [np.ones(cfg.d) for _ in range(cfg.n_layers)]
        self.g_final = np.ones(cfg.d)

    def layer(self, l, which):
        return self.t[layer_tid(l, which)]

    @property
    def embed(self):
        return self.t[TID_EMBED]

    @property
    def head(self):
        return self.t[TID_HEAD]


def rms_scale(x, eps):
    """1 / sqrt(mean(x^2) + eps), per row (a column vector)."""
    return 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def rmsnorm(x, g, eps):
    """x / sqrt(mean(x^2) + eps) * g, per row."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def rope(u, n_heads, head_dim, theta):
    """Rotary embedding, rotate-half pairing, position = row index in the window.

    For each head, pair (i, i + hd/2), i < hd/2, rotates by angle
    pos * theta^(-2i/hd).  ``theta = inf`` gives the identity (frequency 0).
    """
    L = u.shape[0]
    half = head_dim // 2
    i = np.arange(half, dtype=np.float64)
    freq = np.power(float(theta), -2.0 * i / head_dim) if np.isfinite(theta) else np.zeros(half)
    ang = np.arange(L, dtype=np.float64)[:, None] * freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    u = u.reshape(L, n_heads, head_dim)
    a, b = u[..., :half], u[..., half:]
    out = np.concatenate([a * c[:, None, :] - b * s[:, None, :], b * c[:, None, :] + a * s[:, None, :]], axis=-1)
    return out.reshape(L, n_heads * head_dim)


def silu(x):
    return x / (1.0 + np.exp(-x))


def _matmul(a, b, dtype):
    """a @ b with products and sums in ``dtype`` (float64, or float32 for the
    accumulation-order experiment), returned as float64."""
    if dtype == np.float64:
        return a @ b
    return (a.astype(dtype) @ b.astype(dtype)).astype(np.float64)


def attention(q, k, v, n_heads, n_kv_heads, head_dim, probs=None, matmul_dtype=np.float64):
    """Bidirectional multi-head / grouped-query attention over one window.

    ``probs`` (a list): receives the head-averaged attention probabilities [L, L].
    """
    L = q.shape[0]
    pavg = np.zeros((L, L)) if probs is not None else None
    group = n_heads // n_kv_heads
    out = np.empty((L, n_heads * head_dim))
    scale = 1.0 / np.sqrt(head_dim)
    for h in range(n_heads):
        g = h // group
        qh = q[:, h * head_dim:(h + 1) * head_dim]
        kg = k[:, g * head_dim:(g + 1) * head_dim]
        vg = v[:, g * head_dim:(g + 1) * head_dim]
        s = _matmul(qh, kg.T, matmul_dtype) * scale
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h * head_dim:(h + 1) * head_dim] = _matmul(p, vg, matmul_dtype)
        if pavg is not None:
            pavg += p / n_heads
    if probs is not None:
        probs.append(pavg)
    return out


def hidden(wts, state, probs=None, matmul_dtype=np.float64):
    """Final normed hidden states [L, d] (the LM head input) for one window.

    ``probs`` (a list): receives each layer's head-averaged attention [L, L].
    ``matmul_dtype``: float64 (the oracle), or float32 to run every
    contraction with float32 products and sums while keeping every storage
    rounding point -- the accumulation-order experiment that measures how far
    two faithful evaluations of the same model drift apart at depth.
    """
    cfg = wts.cfg
    rnd = lambda a: W.storage_round(a, cfg.dtype)
    r32 = W.round_f32
    hd = cfg.head_dim
    mm = lambda a, b: _matmul(a, b, matmul_dtype)
    x = r32(wts.embed[np.asarray(state)])
    for l in range(cfg.n_layers):
        # pre-norm as a row scale of the projections: (x g / rms(x)) W^T = (x g) W^T / rms(x),
        # with x g stored in the model's dtype and the scale applied to the float result
        rs = rms_scale(x, cfg.norm_eps)
        h = rnd(x * wts.g_attn[l])
        q = rs * mm(h, wts.layer(l, WQ).T)
        k = rs * mm(h, wts.layer(l, WK).T)
        v = rs * mm(h, wts.layer(l, WV).T)
        q = rnd(rope(q, cfg.n_heads, hd, cfg.rope_theta))
        k = rnd(rope(k, cfg.n_kv_heads, hd, cfg.rope_theta))
        v = rnd(v)
        o = rnd(attention(q, k, v, cfg.n_heads, cfg.n_kv_heads, hd, probs, matmul_dtype))
        x = r32(x + mm(o, wts.layer(l, WO).T))
        rs = rms_scale(x, cfg.norm_eps)
        h = rnd(x * wts.g_ffn[l])
        a = rnd(silu(rs * mm(h, wts.layer(l, WGATE).T)) * (rs * mm(h, wts.layer(l, WUP).T)))
        x = r32(x + mm(a, wts.layer(l, WDOWN).T))
    return rnd(rmsnorm(x, wts.g_final, cfg.norm_eps))


def forward(wts, state, rows=None, matmul_dtype=np.float64):
    """Logits [len(rows), V] (float32 values in float64) for one window.

    ``state`` holds symbol ids in [0, V] (V = [MASK]); ``rows`` selects the
    positions whose distributions are needed (default: all).
    """
    h = hidden(wts, state, matmul_dtype=matmul_dtype)
    if rows is not None:
        h = h[np.asarray(rows, dtype=np.int64)]
    return W.round_f32(_matmul(h, wts.head.T, matmul_dtype))
