"""Pins for the oracle rANS coder (statistical coding, Sec. 2.1 / Sec. 4)."""
import itertools

import numpy as np
import pytest

from oracle import coder as RC
from oracle import container as C
from oracle import model as M
from oracle import pipeline as PL
from oracle import rans as R
from oracle import selector as S


def _table(rng, V, P):
    f = rng.integers(1, 50, V).astype(np.float64)
    f = np.floor(f / f.sum() * ((1 << P) - V)).astype(np.int64) + 1
    f[0] += (1 << P) - f.sum()
    return np.concatenate([[0], np.cumsum(f)]), f


def _roundtrip(pairs_sym, cdf, f, P):
    e = R.Encoder(P)
    for s in pairs_sym:
        e.encode(int(cdf[s]), int(f[s]))
    bits, data = e.finish()
    d = R.Decoder(data, bits, P)
    return bits, data, [d.decode(cdf) for _ in pairs_sym]


def test_hand_computed_streams():
    # certain symbol (f = 2^P): the state stays L = 2^31
    e = R.Encoder(2)
    e.encode(0, 4)
    assert e.finish() == (64, (1 << 31).to_bytes(8, "big"))
    # x = floor(2^31 / 1) 2^2 + 0 + 1
    e = R.Encoder(2)
    e.encode(1, 1)
    assert e.finish() == (64, (2 ** 33 + 1).to_bytes(8, "big"))
    # two symbols, coded in reverse: (8, 8) then (3, 5) with P = 4:
    # x1 = (2^31 // 8) 16 + 0 + 8 = 2^32 + 8;  x2 = (x1 // 5) 16 + (x1 mod 5) + 3
    e = R.Encoder(4)
    e.encode(3, 5)
    e.encode(8, 8)
    x1 = 2 ** 32 + 8
    assert e.finish() == (64, ((x1 // 5) * 16 + x1 % 5 + 3).to_bytes(8, "big"))


def test_word_emission():
    # f = 1 at P = 24 adds 24 bits per symbol: after a few symbols a word must be emitted
    e = R.Encoder(24)
    for _ in range(5):
        e.encode(7, 1)
    bits, data = e.finish()
    assert bits == 64 + 32 * ((bits - 64) // 32) and bits > 64
    d = R.Decoder(data, bits, 24)
    cdf = np.array([0, 7, 8, 1 << 24])
    assert [d.decode(cdf) for _ in range(5)] == [1] * 5


@pytest.mark.parametrize("P,V", [(2, 3), (8, 7), (16, 256), (24, 5000)])
def test_random_round_trip_and_length_bound(P, V):
    rng = np.random.default_rng(P * 1000 + V)
    cdf, f = _table(rng, V, P)
    for n in (0, 1, 2, 17, 600):
        sym = rng.integers(0, V, n)
        bits, data, out = _roundtrip(sym, cdf, f, P)
        assert out == sym.tolist()
        ideal = float(-np.log2(f[sym] / 2.0 ** P).sum())
        assert ideal - 1e-9 <= bits <= ideal + 64 + 32   # flushed state + one partial word
        assert len(data) == bits // 8


def test_exhaustive_tiny_alphabet():
    P = 4
    f = np.array([1, 2, 12, 1])
    cdf = np.concatenate([[0], np.cumsum(f)])
    for n in range(0, 7):
        for seq in itertools.product(range(4), repeat=n):
            _, _, out = _roundtrip(list(seq), cdf, f, P)
            assert out == list(seq)


def test_extreme_frequencies():
    for P, V in ((16, 256), (24, 126464)):
        f = np.ones(V, dtype=np.int64)
        f[-1] += (1 << P) - V              # last symbol takes all the remainder
        cdf = np.concatenate([[0], np.cumsum(f)])
        sym = [V - 1] * 50 + [0, V - 2, V - 1] * 20
        _, _, out = _roundtrip(sym, cdf, f, P)
        assert out == sym


def test_same_symbols_as_range_coder_close_length():
    rng = np.random.default_rng(7)
    cdf, f = _table(rng, 256, 16)
    sym = rng.integers(0, 256, 2000)
    rbits, _, out = _roundtrip(sym, cdf, f, 16)
    e = RC.Encoder(16)
    for s in sym:
        e.encode(int(cdf[s]), int(f[s]))
    gbits, gdata = e.finish()
    d = RC.Decoder(gdata, gbits, 16)
    assert [d.decode(cdf) for _ in sym] == out == sym.tolist()
    assert abs(rbits - gbits) <= 96


TINY4 = M.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)


@pytest.fixture(scope="module")
def w4():
    return M.Weights(TINY4)


@pytest.mark.parametrize("pol", [S.Policy(kind=S.TOPK_CONF, k=2, block=2), S.Policy(kind=S.ENTROPY, tau_bits=1.5),
                                 S.Policy(kind=S.UNIFORM, k=2)])
def test_pipeline_round_trips_with_rans(w4, pol):
    for L in range(0, 5):
        for seq in itertools.product(range(4), repeat=L):
            data = bytes(seq)
            blob = PL.compress(w4, data, 3, pol, coder=PL.RANS)
            assert PL.decompress(w4, blob) == data
    blob = PL.compress(w4, b"\x01\x02\x03\x00\x01", 4, pol, coder=PL.RANS)
    h, _ = C.read(blob)
    assert h.coder == PL.RANS and blob[5] == 1
    with pytest.raises(C.ContainerError):
        C.read(blob[:5] + b"\x03" + blob[6:])
