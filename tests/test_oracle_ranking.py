"""Pins for the oracle symbol ranking (Definition "Symbol Ranking"; Sec. 4 varints)."""
import itertools

import numpy as np
import pytest

from oracle import container as C
from oracle import model as M
from oracle import pipeline as PL
from oracle import quantizer as Q
from oracle import ranking as K
from oracle import selector as S


def test_rank_is_position_in_sorted_order():
    rng = np.random.default_rng(0)
    for V in (1, 2, 5, 37, 256):
        for _ in range(20):
            freq = rng.integers(1, 6, V)              # many ties
            order = sorted(range(V), key=lambda v: (-freq[v], v))
            for s in range(V):
                assert K.rank_of(freq, s) == order.index(s)
                assert K.symbol_of(freq, K.rank_of(freq, s)) == s


def test_most_probable_symbol_has_rank_zero():
    l = np.random.default_rng(1).normal(0, 3, (20, 300)).astype(np.float32)
    qz = Q.quantize(l, 16)
    for i in range(20):
        assert K.rank_of(qz["freq"][i], int(qz["top"][i])) == 0


def test_varint_round_trip_and_lengths():
    for n in (0, 1, 127, 128, 255, 16383, 16384, 126463, 2 ** 28 - 1):
        v = K.varint(n)
        assert len(v) == max(1, (n.bit_length() + 6) // 7)
        e = K.Encoder(16)
        e.out += v
        bits, data = e.finish()
        f = np.ones(2 ** 28, dtype=np.int64) if n >= 1 << 20 else np.ones(max(n + 1, 2), dtype=np.int64)
        if n < 1 << 20:
            cdf = np.concatenate([[0], np.cumsum(f)])
            assert K.Decoder(data, bits, 16).decode(cdf) == n  # all-equal table: rank = symbol
    assert K.varint(300) == bytes([0xAC, 0x02])                  # LEB128: low group first


def test_corrupt_rank_streams():
    cdf = np.array([0, 3, 4])
    with pytest.raises(K.CorruptStream):
        K.Decoder(b"\x02", 8, 16).decode(cdf)                    # rank 2 of 2 symbols
    with pytest.raises(K.CorruptStream):
        K.Decoder(b"\x80", 8, 16).decode(cdf)                    # truncated varint


TINY4 = M.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)


@pytest.mark.parametrize("pol", [S.Policy(kind=S.TOPK_CONF, k=2, block=2), S.Policy(kind=S.ENTROPY, tau_bits=1.5),
                                 S.Policy(kind=S.PROGRESSIVE, k=1, growth_q16=2 << 16)])
def test_pipeline_round_trips_with_ranks(pol):
    w = M.Weights(TINY4)
    for L in range(0, 5):
        for seq in itertools.product(range(4), repeat=L):
            data = bytes(seq)
            blob = PL.compress(w, data, 3, pol, coder=PL.RANKS)
            assert PL.decompress(w, blob) == data
    blob = PL.compress(w, b"\x03\x02\x01\x00", 4, pol, coder=PL.RANKS)
    h, streams = C.read(blob)
    assert h.coder == PL.RANKS and sum(b for b, _ in streams) == 8 * 4  # four ranks < 128: one byte each
