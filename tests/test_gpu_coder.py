"""GPU quantise + select + range-code steps vs the oracle on identical logits.

Logits come from the seeded ``sources.synthetic_logits`` for (window, step),
so both sides code with the same tables: the streams must agree bit for bit,
and the GPU decoder must recover the symbols from the GPU streams.
"""
import numpy as np
import pytest

from oracle import context as X
from oracle import pipeline as OP
from oracle import quantizer as Q
from oracle import selector as S
from paper_2608_11249_gb300 import sources
from tests.gpu_helpers import dlmz, ptr, to_dev

pytestmark = pytest.mark.gpu


def _gpu_run(d, symbols, V, pol, opol, seed, L, ctx=None, coder_kind=0):
    """Encode all windows on the GPU, then decode; return (bits, streams, decoded).

    ``ctx``: per-window context positions (the caller-side initial context, Sec. 3.4)."""
    import torch
    nc = symbols.shape[0]
    P = Q.precision_for_vocab(V)
    coder = d.Coder(nc, L, V, P, coder_kind)
    coder.reset_encoder()
    sym = to_dev(symbols.astype(np.int32))
    init = np.full((nc, L), V, dtype=np.int32)
    for c in range(nc):
        if ctx is not None:
            init[c, ctx[c]] = symbols[c, ctx[c]]
    state = to_dev(init.copy())
    committed = torch.zeros(nc, dtype=torch.int32, device="cuda")

    def steps(fn):
        step = 0
        if opol.kind in (S.UNIFORM, S.PROGRESSIVE):
            # the caller runs the schedule: rows = the union of the windows' next u_k masked positions
            masked = [np.flatnonzero(init[c] == V) for c in range(nc)]
            t = 0
            for u in S.schedule_sizes(masked[0].size, opol):
                lo = min(int(mk[t]) for mk in masked)
                hi = max(int(mk[t + u - 1]) for mk in masked) + 1
                lg = np.concatenate([sources.synthetic_logits(seed, c, step, L, V)[lo:hi] for c in range(nc)])
                fn(to_dev(lg), lo, hi - lo, d.policy(opol.kind, u, coder=coder_kind))
                t += u
                step += 1
        elif opol.kind == S.TOPK_CONF:
            # a window's own step count keys its logits (a window with fewer masked positions in a
            # block sits out the block's last steps, so its count lags the others')
            wstep = [0] * nc
            B = opol.block or L
            for b0 in range(0, L, B):
                Bl = min(B, L - b0)
                need = [-(-int(np.sum(init[c, b0:b0 + Bl] == V)) // opol.k) for c in range(nc)]
                for t in range(max(need)):
                    lg = np.concatenate([sources.synthetic_logits(seed, c, wstep[c], L, V)[b0:b0 + Bl]
                                         for c in range(nc)])
                    fn(to_dev(lg), b0, Bl, pol)
                    for c in range(nc):
                        wstep[c] += t < need[c]
        else:
            while True:
                lg = np.concatenate([sources.synthetic_logits(seed, c, step, L, V) for c in range(nc)])
                fn(to_dev(lg), 0, L, pol)
                step += 1
                if int((state == V).sum().item()) == 0:
                    break
                assert step <= L

    steps(lambda lg, r0, rpc, p: coder.encode_step(p, ptr(lg), r0, rpc, ptr(sym), ptr(state), ptr(committed)))
    d.check()
    assert np.array_equal(state.cpu().numpy(), symbols)
    bits = torch.empty(nc, dtype=torch.int32, device="cuda")
    cap = coder.capacity_units * 2
    raw = torch.zeros(nc * cap, dtype=torch.uint8, device="cuda")
    coder.finish(ptr(bits), ptr(raw))
    d.check()
    bits_h = bits.cpu().numpy().astype(np.int64)
    raw_h = raw.cpu().numpy()
    streams = [bytes(raw_h[c * cap:c * cap + (bits_h[c] + 7) // 8]) for c in range(nc)]
    # decode from a packed copy of the streams
    offs = np.concatenate([[0], np.cumsum([(b + 7) // 8 for b in bits_h])[:-1]]).astype(np.uint64)
    packed = np.frombuffer(b"".join(streams) + b"\0" * 8, dtype=np.uint8)
    dcoder = d.Coder(nc, L, V, P, coder_kind)
    d_packed, d_offs, d_bits = to_dev(packed), to_dev(offs.view(np.int64)), to_dev(bits_h.astype(np.int32))
    dcoder.load_decoder(ptr(d_packed), ptr(d_offs), ptr(d_bits))
    state.copy_(to_dev(init))
    steps(lambda lg, r0, rpc, p: dcoder.decode_step(p, ptr(lg), r0, rpc, ptr(state), ptr(committed)))
    d.check()
    return bits_h, streams, state.cpu().numpy()


CASES = [
    # V, L, nc, policy
    (4, 6, 5, S.Policy(kind=S.TOPK_CONF, k=2, block=4)),
    (256, 100, 3, S.Policy(kind=S.TOPK_CONF, k=4, block=64)),
    (256, 512, 2, S.Policy(kind=S.TOPK_CONF, k=8, block=128)),
    (37, 50, 4, S.Policy(kind=S.TOPK_CONF, k=3, block=0)),
    (256, 64, 3, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=0)),
    (256, 80, 2, S.Policy(kind=S.ENTROPY, tau_bits=2.0, k_min=2, k_max=5)),
    (5000, 40, 2, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=64)),
    (5000, 33, 2, S.Policy(kind=S.TOPK_CONF, k=16, block=0)),
    # the large vocabularies (P = 24): 8B-shaped top-16 over the whole window, 7B-shaped entropy
    # threshold 0.5 bits with m = 1 and cap 64
    (126464, 40, 2, S.Policy(kind=S.TOPK_CONF, k=16, block=0)),
    (152064, 24, 2, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=64)),
]


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_steps_bit_exact_and_decode(dev, ci):
    d = dlmz()
    V, L, nc, opol = CASES[ci]
    seed = 100 + ci
    rng = np.random.default_rng(seed)
    symbols = rng.integers(0, V, (nc, L))
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max)
    bits, streams, decoded = _gpu_run(d, symbols, V, pol, opol, seed, L)
    P = Q.precision_for_vocab(V)
    for c in range(nc):
        fn = lambda step, state, rows, c=c: sources.synthetic_logits(seed, c, step, L, V)[rows]
        (obits, obytes), _ = OP.encode_window(symbols[c], V, fn, opol, P)
        assert int(bits[c]) == obits, (c, int(bits[c]), obits)
        assert streams[c] == obytes, c
    assert np.array_equal(decoded, symbols)


LR_CASES = [
    # V, L, nc, policy, context (kind, c, seed)
    (256, 100, 3, S.Policy(kind=S.UNIFORM, k=9), (X.NONE, 0, 0)),
    (256, 64, 2, S.Policy(kind=S.PROGRESSIVE, k=1, growth_q16=3 << 15), (X.NONE, 0, 0)),
    (37, 50, 4, S.Policy(kind=S.UNIFORM, k=5), (X.RANDOM, 6, 3)),
    (5000, 33, 2, S.Policy(kind=S.PROGRESSIVE, k=3, growth_q16=2 << 16), (X.CONTIGUOUS, 4, 0)),
    (256, 80, 3, S.Policy(kind=S.TOPK_CONF, k=4, block=16), (X.RANDOM, 11, 8)),
    (256, 40, 2, S.Policy(kind=S.ENTROPY, tau_bits=2.0, k_min=2, k_max=5), (X.RANDOM, 7, 1)),
]


@pytest.mark.parametrize("ci", range(len(LR_CASES)))
def test_schedule_and_context_steps_bit_exact(dev, ci):
    """Uniform/progressive schedules (Sec. 3.3) and context (Sec. 3.4) on identical logits: streams bit for bit."""
    d = dlmz()
    V, L, nc, opol, (ck, cc, cs) = LR_CASES[ci]
    seed = 200 + ci
    symbols = np.random.default_rng(seed).integers(0, V, (nc, L))
    ctx = [X.positions(ck, cc, cs, L, c) for c in range(nc)]
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max, opol.growth_q16)
    bits, streams, decoded = _gpu_run(d, symbols, V, pol, opol, seed, L, ctx)
    P = Q.precision_for_vocab(V)
    for c in range(nc):
        fn = lambda step, state, rows, c=c: sources.synthetic_logits(seed, c, step, L, V)[rows]
        (obits, obytes), _ = OP.encode_window(symbols[c], V, fn, opol, P, ctx=ctx[c])
        assert int(bits[c]) == obits and streams[c] == obytes, c
    assert np.array_equal(decoded, symbols)


RANS_CASES = [
    # V, L, nc, policy, context
    (4, 6, 5, S.Policy(kind=S.TOPK_CONF, k=2, block=4), (X.NONE, 0, 0)),
    (256, 512, 2, S.Policy(kind=S.TOPK_CONF, k=8, block=128), (X.NONE, 0, 0)),
    (256, 64, 3, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=0), (X.NONE, 0, 0)),
    (5000, 40, 2, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=64), (X.RANDOM, 5, 2)),
    (126464, 24, 2, S.Policy(kind=S.UNIFORM, k=4), (X.NONE, 0, 0)),
    (37, 50, 4, S.Policy(kind=S.PROGRESSIVE, k=1, growth_q16=3 << 15), (X.CONTIGUOUS, 3, 0)),
]


@pytest.mark.parametrize("ci", range(len(RANS_CASES)))
def test_rans_steps_bit_exact_and_decode(dev, ci):
    """The paper's rANS coder (Sec. 2.1) on identical logits: streams bit for bit, then decoded."""
    d = dlmz()
    V, L, nc, opol, (ck, cc, cs) = RANS_CASES[ci]
    seed = 300 + ci
    symbols = np.random.default_rng(seed).integers(0, V, (nc, L))
    ctx = [X.positions(ck, cc, cs, L, c) for c in range(nc)]
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max, opol.growth_q16,
                   coder=d.CODER_RANS)
    bits, streams, decoded = _gpu_run(d, symbols, V, pol, opol, seed, L, ctx, d.CODER_RANS)
    P = Q.precision_for_vocab(V)
    for c in range(nc):
        fn = lambda step, state, rows, c=c: sources.synthetic_logits(seed, c, step, L, V)[rows]
        (obits, obytes), _ = OP.encode_window(symbols[c], V, fn, opol, P, ctx=ctx[c], coder=OP.RANS)
        assert int(bits[c]) == obits and streams[c] == obytes, c
    assert np.array_equal(decoded, symbols)


def test_coder_kind_must_match(dev):
    d = dlmz()
    coder = d.Coder(2, 8, 256, 16, d.CODER_RANS)
    lg = to_dev(np.zeros((16, 256), dtype=np.float32))
    st = to_dev(np.full((2, 8), 256, dtype=np.int32))
    sym = to_dev(np.zeros((2, 8), dtype=np.int32))
    with pytest.raises(d.DlmzError) as e:
        coder.encode_step(d.policy(d.TOPK_CONF, 1), ptr(lg), 0, 8, ptr(sym), ptr(st), 0)
    assert e.value.code == d.EINVAL


RANK_CASES = [
    # V, L, nc, policy, context
    (4, 6, 5, S.Policy(kind=S.TOPK_CONF, k=2, block=4), (X.NONE, 0, 0)),
    (256, 100, 3, S.Policy(kind=S.TOPK_CONF, k=4, block=64), (X.NONE, 0, 0)),
    (256, 64, 3, S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=0), (X.RANDOM, 4, 1)),
    (5000, 33, 2, S.Policy(kind=S.UNIFORM, k=5), (X.NONE, 0, 0)),
    (37, 50, 2, S.Policy(kind=S.PROGRESSIVE, k=2, growth_q16=3 << 15), (X.CONTIGUOUS, 2, 0)),
]


@pytest.mark.parametrize("ci", range(len(RANK_CASES)))
def test_rank_steps_bit_exact_and_decode(dev, ci):
    """Symbol ranking (varint ranks) on identical logits: rank streams byte for byte, then decoded."""
    d = dlmz()
    V, L, nc, opol, (ck, cc, cs) = RANK_CASES[ci]
    seed = 400 + ci
    symbols = np.random.default_rng(seed).integers(0, V, (nc, L))
    ctx = [X.positions(ck, cc, cs, L, c) for c in range(nc)]
    pol = d.policy(opol.kind, opol.k, opol.block, opol.tau_bits, opol.k_min, opol.k_max, opol.growth_q16,
                   coder=d.CODER_RANKS)
    bits, streams, decoded = _gpu_run(d, symbols, V, pol, opol, seed, L, ctx, d.CODER_RANKS)
    P = Q.precision_for_vocab(V)
    for c in range(nc):
        fn = lambda step, state, rows, c=c: sources.synthetic_logits(seed, c, step, L, V)[rows]
        (obits, obytes), _ = OP.encode_window(symbols[c], V, fn, opol, P, ctx=ctx[c], coder=OP.RANKS)
        assert int(bits[c]) == obits and streams[c] == obytes, c
    assert np.array_equal(decoded, symbols)
