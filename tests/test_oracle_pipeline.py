"""Pins for the oracle pipeline (Sec. 3.2): exhaustive round trips, edge cases, corruption."""
import itertools

import numpy as np
import pytest

from oracle import container as C
from oracle import model as M
from oracle import pipeline as PL
from oracle import selector as S
from paper_2608_11249_gb300 import sources

TINY4 = M.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)


@pytest.fixture(scope="module")
def w4():
    return M.Weights(TINY4)


POLICIES = [
    S.Policy(kind=S.TOPK_CONF, k=1, block=0),
    S.Policy(kind=S.TOPK_CONF, k=2, block=2),
    S.Policy(kind=S.TOPK_CONF, k=5, block=0),
    S.Policy(kind=S.ENTROPY, tau_bits=1.5, k_min=1, k_max=0),
    S.Policy(kind=S.ENTROPY, tau_bits=1.9, k_min=2, k_max=3),
]


@pytest.mark.parametrize("pi", range(len(POLICIES)))
def test_exhaustive_tiny_windows(w4, pi):
    pol = POLICIES[pi]
    for L in range(0, 5):
        for seq in itertools.product(range(4), repeat=L):
            data = bytes(seq)
            blob = PL.compress(w4, data, 8, pol)
            assert PL.decompress(w4, blob) == data


def test_decoder_replays_every_selection_order(w4):
    # record the encoder's selection trace and check the decoder's forward
    # calls see exactly the same states
    pol = S.Policy(kind=S.ENTROPY, tau_bits=1.2, k_min=1, k_max=2)
    fn = PL.model_logits_fn(w4)
    for seq in itertools.product(range(4), repeat=5):
        seen_enc, seen_dec = [], []
        fe = lambda step, st, rows: (seen_enc.append(st.tolist()), fn(step, st, rows))[1]
        fd = lambda step, st, rows: (seen_dec.append(st.tolist()), fn(step, st, rows))[1]
        trace = []
        stream, steps = PL.encode_window(np.array(seq), 4, fe, pol, 16, trace)
        out = PL.decode_window(stream, 5, 4, fd, pol, 16)
        assert out.tolist() == list(seq)
        assert seen_enc == seen_dec
        assert sum(len(t) for t in trace) == 5


def test_ragged_tail_empty_and_single(w4):
    pol = S.Policy(kind=S.TOPK_CONF, k=2, block=4)
    for n in (0, 1, 7, 9, 16, 17):
        data = bytes(np.random.default_rng(n).integers(0, 4, n).astype(np.uint8))
        blob = PL.compress(w4, data, 8, pol)
        h, streams = C.read(blob)
        assert h.n_chunks == -(-n // 8) and h.n_symbols == n
        assert PL.decompress(w4, blob) == data


def test_token_vocab_roundtrip():
    cfg = M.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=2, ffn=16, vocab=5000, dtype="bf16", seed=2)
    w = M.Weights(cfg)
    tok = sources.zipf_bigram_tokens(40, 5000, seed=3)
    data = sources.tokens_to_bytes(tok)
    pol = S.Policy(kind=S.ENTROPY, tau_bits=0.5, k_min=1, k_max=64)
    blob = PL.compress(w, data, 16, pol)
    assert C.read(blob)[0].P == 24
    assert PL.decompress(w, blob) == data
    with pytest.raises(PL.BadInput):
        PL.compress(w, data[:-1], 16, pol)
    bad = np.array([5000], dtype="<u4").tobytes()
    with pytest.raises(PL.BadInput):
        PL.compress(w, bad, 16, pol)


def test_workload_shaped_bytes_roundtrip_and_size():
    cfg = M.ModelConfig(n_layers=1, d=32, n_heads=2, n_kv_heads=2, ffn=64, vocab=256, dtype="f32", seed=0)
    w = M.Weights(cfg)
    data = sources.markov_bytes(300, seed=0)
    pol = S.Policy(kind=S.TOPK_CONF, k=4, block=64)
    blob = PL.compress(w, data, 128, pol)
    assert PL.decompress(w, blob) == data
    # random-init model is near uniform: about 8 bits per byte plus header
    h, streams = C.read(blob)
    bits = sum(b for b, _ in streams)
    assert 7.5 * len(data) < bits < 8.3 * len(data)


def test_corruption_is_reported(w4):
    pol = S.Policy(kind=S.TOPK_CONF, k=2, block=4)
    data = bytes(np.random.default_rng(0).integers(0, 4, 30).astype(np.uint8))
    blob = PL.compress(w4, data, 8, pol)
    with pytest.raises(C.ContainerError):
        PL.decompress(w4, b"XXXX" + blob[4:])
    with pytest.raises(C.ContainerError):
        PL.decompress(w4, blob[:5] + b"\x07" + blob[6:])
    with pytest.raises(C.ContainerError):
        PL.decompress(w4, blob[:-1])
    with pytest.raises(C.ContainerError):
        PL.decompress(w4, blob[:40])
    other = M.Weights(M.ModelConfig(**{**TINY4.__dict__, "seed": 2}))
    with pytest.raises(C.FingerprintError):
        PL.decompress(other, blob)
    # a flipped stream bit decodes to other symbols: the checksum reports it
    flipped = bytearray(blob)
    flipped[-3] ^= 0x10
    with pytest.raises((C.ContainerError, Exception)):
        PL.decompress(w4, bytes(flipped))


def test_header_roundtrip():
    h = C.Header(P=16, kind=1, fingerprint=123, vocab=256, chunk_len=512, batch_chunks=1024, k=8,
                 block=128, tau_q=32768, k_min=1, k_max=64, n_symbols=10 ** 6, n_chunks=1954,
                 crc32=0xDEADBEEF)
    streams = [(i * 3 + 1, bytes((i * 3 + 1 + 7) // 8)) for i in range(1954)]
    h2, s2 = C.read(C.write(h, streams))
    assert h2 == h and s2 == streams


def test_policy_validation(w4):
    with pytest.raises(PL.BadInput):
        PL.compress(w4, b"\x00", 8, S.Policy(kind=S.TOPK_CONF, k=0))
    with pytest.raises(PL.BadInput):
        PL.compress(w4, b"\x00", 8, S.Policy(kind=S.ENTROPY, k_min=0))
    with pytest.raises(PL.BadInput):
        PL.compress(w4, b"\x00", 0, S.Policy(kind=S.TOPK_CONF, k=1))
