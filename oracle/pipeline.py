"""Iterative DLM compression pipeline (oracle side), Sec. 3.2.

Starting from the masked window S^(0) (fully masked, or with c context
symbols left visible, Sec. 3.4), each step runs the masked DLM over the
current state, turns the distributions of the schedule's candidate positions
into integer tables, lets the commitment schedule (Sec. 3.3) pick positions,
codes their true symbols in ascending position and reveals them, until the
window is complete.  The input is cut into non-overlapping windows of ``chunk_len``
symbols (Sec. 4), each compressed independently into its own stream.

Symbols: bytes when V <= 256, otherwise little-endian uint32 token ids.

``encode_window`` / ``decode_window`` take a ``logits_fn(step, state,
rows)`` so the same schedule/coder logic runs on the DLM forward
(``model.forward``) or on externally supplied logits.

Parity: pinned by decode(encode(x)) == x on exhaustive tiny windows and on
every workload shape, and the coverage constraint sum u_k = n.
"""
import numpy as np

from . import container as C
from . import context as X
from . import model as M
from . import quantizer as Q
from . import rans
from . import ranking
from . import selector as S
from .coder import Decoder, Encoder

# coders: range coder, rANS (statistical coding, Sec. 2.1), symbol ranks (varints)
RANGE, RANS, RANKS = 0, 1, 2
_ENC = {RANGE: Encoder, RANS: rans.Encoder, RANKS: ranking.Encoder}
_DEC = {RANGE: Decoder, RANS: rans.Decoder, RANKS: ranking.Decoder}


class BadInput(ValueError):
    pass


def validate_policy(policy):
    if policy.kind == S.TOPK_CONF:
        if policy.k < 1:
            raise BadInput("top-k policy needs k >= 1")
    elif policy.kind == S.ENTROPY:
        if policy.k_min < 1:
            raise BadInput("entropy policy needs k_min >= 1")
        if policy.k_max and policy.k_max < policy.k_min:
            raise BadInput("k_max < k_min")
    elif policy.kind in (S.UNIFORM, S.PROGRESSIVE):
        if policy.k < 1:
            raise BadInput("left-to-right schedules need k >= 1")
        if policy.kind == S.PROGRESSIVE and not 1 <= policy.growth_q16 <= 64 << 16:
            raise BadInput("growth ratio out of range")
    else:
        raise BadInput("unknown policy kind")


def symbols_from_bytes(data, V):
    if V <= 256:
        return np.frombuffer(bytes(data), dtype=np.uint8).astype(np.int64)
    if len(data) % 4:
        raise BadInput("token input must be a multiple of 4 bytes")
    s = np.frombuffer(bytes(data), dtype="<u4").astype(np.int64)
    if s.size and s.max() >= V:
        raise BadInput("token id >= V")
    return s


def bytes_from_symbols(sym, V):
    if V <= 256:
        return np.asarray(sym, dtype=np.uint8).tobytes()
    return np.asarray(sym, dtype="<u4").tobytes()


def _key(qz, policy):
    return qz["W"] if policy.kind == S.TOPK_CONF else qz["Hq"]


def encode_window(symbols, V, logits_fn, policy, P, trace=None, ctx=(), coder=RANGE):
    """Compress one window; return ((bits, bytes), steps).  ``ctx``: context positions."""
    symbols = np.asarray(symbols, dtype=np.int64)
    n = symbols.size
    state = np.full(n, V, dtype=np.int64)
    ctx = np.asarray(ctx, dtype=np.int64)
    state[ctx] = symbols[ctx]
    enc = _ENC[coder](P)
    tq = Q.tau_q(policy.tau_bits)
    sizes = S.schedule_sizes(int(np.sum(state == V)), policy) if policy.kind in (S.UNIFORM, S.PROGRESSIVE) else None
    step = 0
    while np.any(state == V):
        masked = state == V
        if sizes is not None:  # left to right: the rows are the committed positions
            cand = S.leftmost(masked, sizes[step])
            qz = Q.quantize(logits_fn(step, state.copy(), cand), P)
            sel = [int(p) for p in cand]
            row = {p: i for i, p in enumerate(sel)}
        else:
            cand = S.candidates(masked, policy)
            qz = Q.quantize(logits_fn(step, state.copy(), cand), P)
            key = _key(qz, policy)
            row = {int(p): i for i, p in enumerate(cand)}
            sel = S.select(masked, {p: key[i] for p, i in row.items()}, policy, tq)
        assert sel, "a step must commit at least one position"
        for p in sel:
            i, s = row[p], int(symbols[p])
            if coder == RANKS:
                enc.encode_rank(qz["freq"][i], s)
            else:
                enc.encode(int(qz["cdf"][i, s]), int(qz["freq"][i, s]))
        state[sel] = symbols[sel]
        if trace is not None:
            trace.append(list(sel))
        step += 1
    return enc.finish(), step


def decode_window(stream, n, V, logits_fn, policy, P, ctx=(), ctx_symbols=(), coder=RANGE):
    """Decompress one window of ``n`` symbols from (bits, bytes)."""
    bits, data = stream
    dec = _DEC[coder](data, bits, P)
    state = np.full(n, V, dtype=np.int64)
    state[np.asarray(ctx, dtype=np.int64)] = np.asarray(ctx_symbols, dtype=np.int64)
    tq = Q.tau_q(policy.tau_bits)
    sizes = S.schedule_sizes(int(np.sum(state == V)), policy) if policy.kind in (S.UNIFORM, S.PROGRESSIVE) else None
    step = 0
    while np.any(state == V):
        masked = state == V
        if sizes is not None:
            cand = S.leftmost(masked, sizes[step])
            qz = Q.quantize(logits_fn(step, state.copy(), cand), P)
            sel = [int(p) for p in cand]
            row = {p: i for i, p in enumerate(sel)}
        else:
            cand = S.candidates(masked, policy)
            qz = Q.quantize(logits_fn(step, state.copy(), cand), P)
            key = _key(qz, policy)
            row = {int(p): i for i, p in enumerate(cand)}
            sel = S.select(masked, {p: key[i] for p, i in row.items()}, policy, tq)
        for p in sel:
            state[p] = dec.decode(qz["cdf"][row[p]])
        step += 1
    return state


def model_logits_fn(wts):
    return lambda step, state, rows: M.forward(wts, state, rows)


def compress(wts, data, chunk_len, policy, batch_chunks=1, context=(X.NONE, 0, 0), coder=RANGE):
    """Compress ``data`` with the DLM ``wts``; return the container bytes.

    ``context`` = (kind, c, seed): c symbols per window left visible (Sec. 3.4).
    ``coder``: RANGE or RANS.
    """
    cfg = wts.cfg
    V = cfg.vocab
    validate_policy(policy)
    if chunk_len < 1:
        raise BadInput("chunk_len must be >= 1")
    sym = symbols_from_bytes(data, V)
    P = Q.precision_for_vocab(V)
    n = sym.size
    nchunks = (n + chunk_len - 1) // chunk_len
    fn = model_logits_fn(wts)
    ckind, cc, cseed = context
    if ckind not in (X.NONE, X.CONTIGUOUS, X.RANDOM, X.ATTENTION) or cc < 0 or (ckind == X.NONE) != (cc == 0):
        raise BadInput("bad context")
    streams, ctx_sym, ctx_pos = [], [], []
    for c in range(nchunks):
        win = sym[c * chunk_len:(c + 1) * chunk_len]
        if ckind == X.ATTENTION:
            ctx = X.attention_positions(wts, win, cc)
            ctx_pos.append(ctx)
        else:
            ctx = X.positions(ckind, cc, cseed, win.size, c)
        ctx_sym.append(win[ctx])
        if coder not in _ENC:
            raise BadInput("unknown coder")
        (bits, byts), _ = encode_window(win, V, fn, policy, P, ctx=ctx, coder=coder)
        streams.append((bits, byts))
    block = policy.growth_q16 if policy.kind == S.PROGRESSIVE else policy.block
    h = C.Header(P=P, kind=policy.kind, fingerprint=C.fingerprint(cfg), vocab=V, chunk_len=chunk_len,
                 batch_chunks=batch_chunks, k=policy.k, block=block,
                 tau_q=Q.tau_q(policy.tau_bits), k_min=policy.k_min, k_max=policy.k_max,
                 n_symbols=n, n_chunks=nchunks,
                 crc32=C.window_checksum(bytes(data), chunk_len * (1 if V <= 256 else 4)),
                 coder=coder, ctx_kind=ckind, ctx_c=cc, ctx_seed=cseed,
                 ctx_data=bytes_from_symbols(np.concatenate(ctx_sym) if ctx_sym else [], V),
                 ctx_pos=np.concatenate(ctx_pos).astype("<u4").tobytes() if ctx_pos else b"")
    return C.write(h, streams)


def policy_from_header(h):
    if h.kind == S.PROGRESSIVE:
        return S.Policy(kind=h.kind, k=h.k, growth_q16=h.block)
    return S.Policy(kind=h.kind, k=h.k, block=h.block, tau_bits=h.tau_q / 65536.0, k_min=h.k_min,
                    k_max=h.k_max)


def decompress(wts, blob):
    cfg = wts.cfg
    h, streams = C.read(blob)
    if h.fingerprint != C.fingerprint(cfg):
        raise C.FingerprintError("container was written with another model")
    if h.vocab != cfg.vocab:
        raise C.ContainerError("vocabulary mismatch")
    policy = policy_from_header(h)
    validate_policy(policy)
    fn = model_logits_fn(wts)
    ctx_all = symbols_from_bytes(h.ctx_data, cfg.vocab)
    pos_all = np.frombuffer(h.ctx_pos, dtype="<u4").astype(np.int64)
    out, used = [], 0
    for c, st in enumerate(streams):
        n = min(h.chunk_len, h.n_symbols - c * h.chunk_len)
        if h.ctx_kind == X.ATTENTION:
            ctx = pos_all[used:used + min(h.ctx_c, n)]
            if ctx.size and (ctx.max() >= n or np.any(np.diff(ctx) <= 0)):
                raise C.ContainerError("bad context positions")
        else:
            ctx = X.positions(h.ctx_kind, h.ctx_c, h.ctx_seed, n, c)
        out.append(decode_window(st, n, cfg.vocab, fn, policy, h.P, ctx, ctx_all[used:used + ctx.size], h.coder))
        used += ctx.size
    sym = np.concatenate(out) if out else np.zeros(0, dtype=np.int64)
    data = bytes_from_symbols(sym, cfg.vocab)
    if C.window_checksum(data, h.chunk_len * (1 if cfg.vocab <= 256 else 4)) != h.crc32:
        raise C.ContainerError("checksum mismatch")
    return data
