"""Pins for the oracle's counter-based weight generator and rounding helpers."""
import math

import numpy as np
import pytest
import scipy.stats

from oracle import weights as W


def test_splitmix64_published_vector():
    # SplitMix64 seeded with 1234567: the reference outputs published with
    # the algorithm (Vigna's splitmix64.c test sequence).
    got = [int(x) for x in W.stream_outputs(np.uint64(1234567), 0, 5)]
    assert got == [6457827717110365317, 3203168211198807973, 9817491932198370423,
                   4593380528125082431, 16408922859458223821]


def test_stream_is_counter_based():
    a = W.stream_outputs(np.uint64(99), 0, 50)
    b = W.stream_outputs(np.uint64(99), 17, 10)
    assert np.array_equal(a[17:27], b)


def test_normal_draws_distribution():
    z = W.normal_draws(0, 5, 200_001)
    assert abs(z.mean()) < 0.01
    assert abs(z.std() - 1.0) < 0.01
    assert scipy.stats.kstest(z, "norm").pvalue > 1e-3
    assert abs(scipy.stats.kurtosis(z, fisher=False) - 3.0) < 0.05


def test_box_muller_pairs_lie_on_radius():
    # each pair (z0, z1) has z0^2 + z1^2 = -2 ln a with a in (0, 1]: the
    # radii follow the chi distribution with 2 degrees of freedom
    z = W.normal_draws(1, 2, 100_000)
    r2 = z[0::2] ** 2 + z[1::2] ** 2
    assert scipy.stats.kstest(r2, "chi2", args=(2,)).pvalue > 1e-3


def test_init_tensor_std_and_storage():
    t = W.init_tensor(0, 3, (64, 128), "bf16")
    assert t.shape == (64, 128)
    assert abs(t.std() - 0.02) < 0.001
    assert np.array_equal(W.round_bf16(t), t)  # already bf16 values
    t32 = W.init_tensor(0, 3, (64, 128), "f32")
    assert np.array_equal(t32.astype(np.float32).astype(np.float64), t32)
    assert np.max(np.abs(t32 - t)) <= np.max(np.abs(t32)) * 2 ** -8


def test_round_bf16_matches_torch_on_float32_inputs():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(0, 1, 10000), rng.normal(0, 1e-20, 1000), rng.normal(0, 1e20, 1000)])
    x = x.astype(np.float32).astype(np.float64)
    ref = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(W.round_bf16(x), ref)


def test_round_bf16_ties_to_even():
    one = 1.0
    ulp = 2.0 ** -7
    assert W.round_bf16(np.array([one + ulp / 2]))[0] == one          # tie -> even (1.0)
    assert W.round_bf16(np.array([one + 3 * ulp / 2]))[0] == one + 2 * ulp  # tie -> even
    assert W.round_bf16(np.array([one + ulp / 2 + 2 ** -30]))[0] == one + ulp
    assert W.round_bf16(np.array([-(one + 3 * ulp / 2)]))[0] == -(one + 2 * ulp)
    assert W.round_bf16(np.array([0.0]))[0] == 0.0


def test_two_pi_constant():
    assert math.tau == 2 * math.pi
