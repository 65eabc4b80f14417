"""Pins for the left-to-right schedules (Sec. 3.3) and the initial context (Sec. 3.4), oracle side."""
import itertools
from fractions import Fraction

import numpy as np
import pytest
import scipy.stats

from oracle import container as C
from oracle import context as X
from oracle import model as M
from oracle import pipeline as PL
from oracle import selector as S

TINY4 = M.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)


@pytest.fixture(scope="module")
def w4():
    return M.Weights(TINY4)


def uni(K):
    return S.Policy(kind=S.UNIFORM, k=K)


def prog(u1, r_q16):
    return S.Policy(kind=S.PROGRESSIVE, k=u1, growth_q16=r_q16)


# ---- schedule sizes -------------------------------------------------------------------

@pytest.mark.parametrize("n", [1, 2, 7, 64, 100, 513])
@pytest.mark.parametrize("K", [1, 2, 3, 8, 64, 1000])
def test_uniform_covers_in_K_steps(n, K):
    u = S.schedule_sizes(n, uni(K))
    assert sum(u) == n                                   # coverage, sum u_k = n
    assert len(u) == min(K, n)                           # K forwards (fewer only when K > n)
    assert all(x == n // min(K, n) for x in u[:-1])      # u = floor(n / K) per step
    assert u[-1] >= u[0]


def test_uniform_extremes():
    assert S.schedule_sizes(9, uni(1)) == [9]            # one-shot
    assert S.schedule_sizes(9, uni(9)) == [1] * 9        # autoregressive
    assert S.schedule_sizes(0, uni(3)) == []


def test_progressive_r1_is_uniform_steps():
    # r = 1 reduces to committing u_1 per step (Sec. 3.3, paragraph 2)
    assert S.schedule_sizes(23, prog(5, 65536)) == [5, 5, 5, 5, 3]


def test_progressive_doubling_closed_form():
    assert S.schedule_sizes(100, prog(1, 2 << 16)) == [1, 2, 4, 8, 16, 32, 37]


@pytest.mark.parametrize("u1,num,den", [(2, 3, 2), (3, 5, 4), (1, 9, 8)])
def test_progressive_matches_exact_rounding_for_dyadic_r(u1, num, den):
    # for r = num / den with den a power of two the fixed-point sequence is exact:
    # u_k = floor(u_1 r^(k-1) + 1/2) (round half up) while the remainder lasts
    n = 400
    r = Fraction(num, den)
    got = S.schedule_sizes(n, prog(u1, num * 65536 // den))
    want, rem, k = [], n, 0
    while rem:
        x = Fraction(u1) * r ** k
        u = min(max(1, int(x + Fraction(1, 2))), rem)
        want.append(u)
        rem -= u
        k += 1
    assert got == want and sum(got) == n


def test_progressive_grows_and_covers():
    for n in (1, 5, 77, 512):
        for u1 in (1, 3, 16):
            for r in (65536, 70000, 3 << 15, 4 << 16):
                u = S.schedule_sizes(n, prog(u1, r))
                assert sum(u) == n and all(x >= 1 for x in u)
                assert all(a <= b for a, b in zip(u[:-2], u[1:-1]))  # non-decreasing before the remainder


# ---- initial context -------------------------------------------------------------------

def test_contiguous_context_is_the_prefix():
    assert X.positions(X.CONTIGUOUS, 3, 0, 10, 5).tolist() == [0, 1, 2]
    assert X.positions(X.CONTIGUOUS, 30, 0, 10, 5).tolist() == list(range(10))
    assert X.positions(X.NONE, 0, 0, 10, 0).size == 0


def test_random_context_distinct_sorted_in_range():
    for n in (1, 2, 5, 64, 513):
        for c in (1, 2, 7, 600):
            for w in range(4):
                p = X.positions(X.RANDOM, c, 11, n, w)
                assert p.size == min(c, n)
                assert np.all(np.diff(p) > 0) and p.min() >= 0 and p.max() < n
    assert np.array_equal(X.positions(X.RANDOM, 4, 3, 50, 7), X.positions(X.RANDOM, 4, 3, 50, 7))
    assert not np.array_equal(X.positions(X.RANDOM, 4, 3, 50, 7), X.positions(X.RANDOM, 4, 3, 50, 8))


def test_random_context_is_uniform():
    # each of n positions is chosen with probability c / n: chi-square over 4000 windows
    n, c, W = 20, 3, 4000
    counts = np.zeros(n)
    for w in range(W):
        counts[X.positions(X.RANDOM, c, 5, n, w)] += 1
    chi2 = scipy.stats.chisquare(counts).pvalue
    assert chi2 > 1e-3
    # pairs too: the draw is a uniform c-subset (Fisher-Yates), not c independent picks
    pairs = np.zeros((n, n))
    for w in range(W):
        p = X.positions(X.RANDOM, 2, 9, n, w)
        pairs[p[0], p[1]] += 1
    iu = np.triu_indices(n, 1)
    assert scipy.stats.chisquare(pairs[iu]).pvalue > 1e-3


# ---- pipeline ------------------------------------------------------------------------------

def test_left_to_right_commit_order(w4):
    fn = PL.model_logits_fn(w4)
    sym = np.random.default_rng(0).integers(0, 4, 11)
    for pol in (uni(4), prog(1, 2 << 16)):
        trace = []
        stream, steps = PL.encode_window(sym, 4, fn, pol, 16, trace)
        sizes = S.schedule_sizes(11, pol)
        assert [len(t) for t in trace] == sizes and steps == len(sizes)
        assert sum(trace, []) == list(range(11))          # contiguous left-to-right blocks
        assert PL.decode_window(stream, 11, 4, fn, pol, 16).tolist() == sym.tolist()


def test_context_positions_are_not_coded(w4):
    fn = PL.model_logits_fn(w4)
    sym = np.random.default_rng(1).integers(0, 4, 13)
    ctx = X.positions(X.RANDOM, 4, 2, 13, 0)
    for pol in (uni(3), prog(2, 3 << 15), S.Policy(kind=S.TOPK_CONF, k=2, block=4),
                S.Policy(kind=S.ENTROPY, tau_bits=1.5, k_min=1)):
        trace = []
        stream, _ = PL.encode_window(sym, 4, fn, pol, 16, trace, ctx=ctx)
        coded = sorted(sum(trace, []))
        assert coded == sorted(set(range(13)) - set(ctx.tolist()))
        out = PL.decode_window(stream, 13, 4, fn, pol, 16, ctx, sym[ctx])
        assert out.tolist() == sym.tolist()


LR_POLICIES = [uni(1), uni(2), uni(5), prog(1, 2 << 16), prog(2, 65536)]
CONTEXTS = [(X.NONE, 0, 0), (X.CONTIGUOUS, 2, 0), (X.RANDOM, 1, 4), (X.RANDOM, 3, 8)]


@pytest.mark.parametrize("pi", range(len(LR_POLICIES)))
def test_exhaustive_tiny_windows_left_to_right(w4, pi):
    pol = LR_POLICIES[pi]
    for ctx in CONTEXTS:
        for L in range(0, 5):
            for seq in itertools.product(range(4), repeat=L):
                data = bytes(seq)
                blob = PL.compress(w4, data, 3, pol, context=ctx)
                assert PL.decompress(w4, blob) == data


def test_context_container_round_trip_and_size(w4):
    data = bytes(np.random.default_rng(2).integers(0, 4, 21).astype(np.uint8))
    pol = S.Policy(kind=S.TOPK_CONF, k=2, block=4)
    blob = PL.compress(w4, data, 8, pol, context=(X.RANDOM, 3, 77))
    h, streams = C.read(blob)
    assert (h.ctx_kind, h.ctx_c, h.ctx_seed) == (X.RANDOM, 3, 77)
    assert len(h.ctx_data) == 3 + 3 + 3                 # windows of 8, 8, 5: three context bytes each
    assert blob[4] == 2 and PL.decompress(w4, blob) == data
    ctx0 = X.positions(X.RANDOM, 3, 77, 8, 0)
    assert list(h.ctx_data[:3]) == [data[p] for p in ctx0]
    plain = PL.compress(w4, data, 8, pol)
    assert plain[4] == 1                                 # no context: the version-1 layout
    for bad in (blob[:70], blob[:64] + b"\x07" + blob[65:], blob[:80] + blob[83:]):
        with pytest.raises(C.ContainerError):
            PL.decompress(w4, bad)


def test_bad_policies_rejected(w4):
    for pol in (uni(0), prog(0, 65536), prog(1, 0), prog(1, (64 << 16) + 1)):
        with pytest.raises(PL.BadInput):
            PL.compress(w4, b"\x00\x01", 4, pol)
    with pytest.raises(PL.BadInput):
        PL.compress(w4, b"\x00\x01", 4, uni(1), context=(X.RANDOM, 0, 1))
