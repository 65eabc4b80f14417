"""Pins for the oracle quantiser: CDF invariants, closed forms, entropy fidelity."""
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats

from oracle import quantizer as Q
from paper_2608_11249_gb300 import sources


def test_exp_table_against_float_powers():
    T = Q.exp_table()
    assert T[0] == 2 ** 31
    for j in range(256):
        exact = 2.0 ** (31 - j / 256.0)
        assert abs(int(T[j]) - exact) <= 0.5 + 1e-6
    assert np.all(np.diff(T.astype(np.int64)) < 0)


def test_scale_constant():
    c = float(Q._C)
    exact = 256.0 * math.log2(math.e)
    assert abs(c - exact) <= np.spacing(np.float32(exact)) / 2


def test_log2q16_against_math_log2():
    rng = np.random.default_rng(0)
    Wv = np.concatenate([rng.integers(2 ** 31, 2 ** 49, 5000, dtype=np.uint64),
                         np.array([2 ** 31, 2 ** 32 - 1, 2 ** 32, 2 ** 48, 3 * 2 ** 40], dtype=np.uint64)])
    got = Q.log2q16(Wv).astype(np.float64) / 65536.0
    ref = np.log2(Wv.astype(np.float64))
    err = ref - got
    assert np.all(err >= -1e-9) and np.all(err < 2.0 ** -15)
    assert Q.log2q16(np.array([2 ** 31], dtype=np.uint64))[0] == 31 << 16


def _check_invariants(out, P):
    cdf, f = out["cdf"].astype(np.int64), out["freq"].astype(np.int64)
    assert np.all(cdf[:, 0] == 0) and np.all(cdf[:, -1] == 1 << P)
    assert np.all(np.diff(cdf, axis=1) == f)
    assert np.all(f >= 1)


@pytest.mark.parametrize("V,P", [(4, 16), (256, 16), (300, 16), (5000, 24)])
def test_cdf_invariants_random_and_adversarial(V, P):
    rng = np.random.default_rng(V)
    rows = [rng.normal(0, s, V) for s in (0.01, 1, 3, 30)]
    rows.append(np.zeros(V))
    rows.append(np.full(V, -1e30))
    x = rng.normal(0, 1, V); x[V // 2] += 1e6; rows.append(x)
    x = np.full(V, -3e38); x[-1] = 3e38; rows.append(x)
    rows.append(np.linspace(-100, 100, V))
    l = np.array(rows, dtype=np.float32)
    out = Q.quantize(l, P)
    _check_invariants(out, P)


def test_uniform_row_closed_form():
    out = Q.quantize(np.zeros((1, 256), dtype=np.float32), 16)
    assert np.all(out["freq"] == 256)
    assert out["W"][0] == 256 * 2 ** 31
    assert out["Hq"][0] == 8 << 16  # log2(256) bits exactly


def test_single_spike_closed_form():
    for V, P in ((256, 16), (5000, 24)):
        l = np.zeros((1, V), dtype=np.float32)
        l[0, 17] = 1000.0
        out = Q.quantize(l, P)
        f = out["freq"][0]
        assert f[17] == (1 << P) - V + 1
        assert np.all(np.delete(f, 17) == 1)
        assert out["W"][0] == 2 ** 31 and out["Hq"][0] == 0


def test_top_is_lowest_index_of_maximum():
    l = np.zeros((1, 10), dtype=np.float32)
    l[0, [3, 7]] = 5.0
    assert Q.quantize(l, 16)["top"][0] == 3


def test_entropy_fidelity():
    rng = np.random.default_rng(1)
    for V, P in ((256, 16), (3000, 24)):
        for s in (0.1, 1.0, 3.0, 8.0):
            l = rng.normal(0, s, (20, V)).astype(np.float32)
            l[np.arange(20), rng.integers(0, V, 20)] += rng.uniform(0, 15, 20).astype(np.float32)
            out = Q.quantize(l, P)
            p = scipy.special.softmax(l.astype(np.float64), axis=1)
            H = scipy.stats.entropy(p, base=2, axis=1)
            assert np.max(np.abs(out["Hq"] / 65536.0 - H)) <= 0.01


def test_kl_of_quantized_table_is_small():
    rng = np.random.default_rng(2)
    l = rng.normal(0, 2, (50, 256)).astype(np.float32)
    out = Q.quantize(l, 16)
    p = scipy.special.softmax(l.astype(np.float64), axis=1)
    qf = out["freq"] / 65536.0
    kl = (p * np.log2(p / qf)).sum(1)
    # min-1 floor + 1/512-bit log grid: well below 0.01 bits per symbol here
    assert np.all(kl >= -1e-12) and np.max(kl) < 0.01


def test_confidence_key_orders_by_max_probability():
    rng = np.random.default_rng(3)
    l = rng.normal(0, 2, (200, 256)).astype(np.float32)
    out = Q.quantize(l, 16)
    pmax = scipy.special.softmax(l.astype(np.float64), axis=1).max(1)
    a, b = np.argsort(out["W"]), np.argsort(-pmax)
    # W is a 1/512-bit quantisation of 1/p_max: rank agreement is near perfect
    assert scipy.stats.spearmanr(out["W"].astype(np.float64), -pmax).statistic > 0.999
    assert a.shape == b.shape


def test_rejects_non_finite():
    l = np.zeros((1, 8), dtype=np.float32)
    l[0, 2] = np.nan
    with pytest.raises(ValueError):
        Q.quantize(l, 16)


def test_isolated_workload_rows():
    rows = sources.spiked_rows(0, 0, 4, 126464)
    out = Q.quantize(rows, 24)
    _check_invariants(out, 24)
    assert np.all(out["Hq"] >= 0)


def test_tau_q():
    assert Q.tau_q(0.5) == 32768
    assert Q.tau_q(0.0) == 0
