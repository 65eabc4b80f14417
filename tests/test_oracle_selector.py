"""Pins for the oracle commitment schedules (Sec. 3.3): brute force and coverage."""
import itertools

import numpy as np
import pytest

from oracle import selector as S


def _brute_best(cand, keys, k):
    """The unique k-subset whose members all precede every non-member in (key, pos)."""
    order_key = {p: (keys[p], p) for p in cand}
    hits = []
    for sub in itertools.combinations(cand, k):
        inside = set(sub)
        outside = [p for p in cand if p not in inside]
        if all(order_key[a] < order_key[b] for a in inside for b in outside):
            hits.append(sorted(sub))
    assert len(hits) == 1
    return hits[0]


def test_topk_matches_brute_force_with_ties():
    rng = np.random.default_rng(0)
    for trial in range(300):
        n = int(rng.integers(1, 11))
        masked = rng.random(n) < 0.7
        if not masked.any():
            masked[rng.integers(0, n)] = True
        keys = {p: int(rng.integers(0, 4)) for p in range(n)}  # many forced ties
        k = int(rng.integers(1, 6))
        pol = S.Policy(kind=S.TOPK_CONF, k=k, block=0)
        cand = [int(p) for p in np.flatnonzero(masked)]
        got = S.select(masked, keys, pol)
        assert got == _brute_best(cand, keys, min(k, len(cand)))


def test_topk_stays_in_leftmost_incomplete_block():
    masked = np.array([0, 0, 0, 0, 0, 1, 0, 1, 1, 1, 1, 1], dtype=bool)
    keys = {p: 100 - p for p in range(12)}  # later positions more confident
    pol = S.Policy(kind=S.TOPK_CONF, k=3, block=4)
    # block 0 complete; block 1 = [4, 8) has masked {5, 7}: only those
    assert S.select(masked, keys, pol) == [5, 7]
    pol0 = S.Policy(kind=S.TOPK_CONF, k=3, block=0)
    assert S.select(masked, keys, pol0) == [9, 10, 11]


def _brute_entropy(cand, keys, tq, m, kmax):
    below = [p for p in cand if keys[p] <= tq]
    if len(below) < m:
        chosen = _brute_best(cand, keys, min(m, len(cand)))
    else:
        chosen = below
    if kmax and len(chosen) > kmax:
        chosen = _brute_best(chosen, keys, kmax)
    return sorted(chosen)


def test_entropy_schedule_matches_brute_force():
    rng = np.random.default_rng(1)
    for trial in range(300):
        n = int(rng.integers(1, 11))
        masked = rng.random(n) < 0.8
        if not masked.any():
            masked[0] = True
        keys = {p: int(rng.integers(0, 6)) for p in range(n)}
        tq = int(rng.integers(0, 6))
        m = int(rng.integers(1, 4))
        kmax = int(rng.integers(0, 5))
        if kmax and kmax < m:
            kmax = m
        pol = S.Policy(kind=S.ENTROPY, tau_bits=tq / 65536.0, k_min=m, k_max=kmax)
        cand = [int(p) for p in np.flatnonzero(masked)]
        assert S.select(masked, keys, pol, tq) == _brute_entropy(cand, keys, tq, m, kmax)


def test_entropy_threshold_is_inclusive():
    masked = np.ones(4, dtype=bool)
    keys = {0: 5, 1: 3, 2: 4, 3: 9}
    pol = S.Policy(kind=S.ENTROPY, k_min=1)
    assert S.select(masked, keys, pol, 4) == [1, 2]


@pytest.mark.parametrize("L,block,k", [(64, 16, 4), (50, 16, 3), (37, 0, 5), (10, 3, 2), (8, 0, 8), (9, 0, 1)])
def test_coverage_and_step_count_topk(L, block, k):
    rng = np.random.default_rng(L * 31 + k)
    masked = np.ones(L, dtype=bool)
    pol = S.Policy(kind=S.TOPK_CONF, k=k, block=block)
    steps, total = 0, 0
    while masked.any():
        keys = {p: int(rng.integers(0, 1000)) for p in range(L)}
        sel = S.select(masked, keys, pol)
        assert sel and all(masked[p] for p in sel) and len(sel) <= k
        masked[sel] = False
        steps += 1
        total += len(sel)
    assert total == L  # sum_k u_k = n
    B = L if block == 0 else block
    expect = sum(-(-min(B, L - s) // k) for s in range(0, L, B))
    assert steps == expect
    if block == 0 and k == 1:
        assert steps == L  # K = n: the autoregressive extreme
    if block == 0 and k >= L:
        assert steps == 1  # K = 1: one shot


def test_coverage_entropy():
    rng = np.random.default_rng(5)
    L = 40
    masked = np.ones(L, dtype=bool)
    pol = S.Policy(kind=S.ENTROPY, k_min=2, k_max=6)
    total = 0
    while masked.any():
        keys = {p: int(rng.integers(0, 100)) for p in range(L)}
        sel = S.select(masked, keys, pol, 10)
        assert 1 <= len(sel) <= 6
        masked[sel] = False
        total += len(sel)
    assert total == L
