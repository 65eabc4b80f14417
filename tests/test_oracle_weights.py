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


def test_c_draws_equal_the_numpy_definition():
    # the C restatement (used for the full-size models) against the numpy definition:
    # float64 draws within a few ulp (libm vs numpy log/cos/sin), identical after bf16 /
    # float32 rounding, from even and odd starting elements
    from oracle import build
    build.build()
    for tid, n0, count in ((3, 0, 100_001), (7, 12_345, 54_321), (1, 1, 4)):
        ref = W.normal_draws(11, tid, n0 + count)[n0:]
        got = W.normal_draws_c(11, tid, count, n0=n0, threads=3)
        assert np.allclose(got, ref, rtol=1e-14, atol=1e-15)
        assert np.array_equal(W.round_bf16(got * W.STD), W.round_bf16(ref * W.STD))
    for dt in ("f32", "bf16"):
        assert np.array_equal(W.init_tensor_c(5, 9, (64, 48), dt), W.init_tensor(5, 9, (64, 48), dt))
    # the C storage rounding is the oracle's: ties to even at bf16's 8-bit significand, just above
    # a tie, signs, zero, tiny and large magnitudes; float32 likewise
    import ctypes
    lib = W._native()
    x = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 0.0, 1.0 + 2.0 ** -8 + 2.0 ** -30,
                  3.0e-30, -7.25e12, 1.0 + 2.0 ** -24, 1.0 + 3 * 2.0 ** -24, 0.1])
    for mode, ref in ((2, W.round_bf16(x)), (1, W.round_f32(x))):
        out = np.empty_like(x)
        lib.oracle_round.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p]
        lib.oracle_round(x.ctypes.data, x.size, mode, out.ctypes.data)
        assert np.array_equal(out, ref), mode


def test_lazy_weights_forward_equals_eager():
    from oracle import build
    from oracle import model as M
    build.build()
    cfg = M.ModelConfig(n_layers=3, d=32, n_heads=4, n_kv_heads=2, ffn=64, vocab=50, dtype="bf16", seed=4)
    s = np.array([1, 50, 7, 50, 49, 0, 3])
    assert np.array_equal(M.forward(M.Weights(cfg, lazy=True), s), M.forward(M.Weights(cfg), s))
