"""Pins for the attention-based initial context (Sec. 3.4, policy 4; Attention Rollout), oracle side."""
import itertools

import numpy as np
import pytest

from oracle import container as C
from oracle import context as X
from oracle import model as M
from oracle import pipeline as PL
from oracle import selector as S

CFG = M.ModelConfig(n_layers=3, d=32, n_heads=4, n_kv_heads=2, ffn=48, vocab=11, dtype="f32", seed=5)


def _zero_qk(cfg):
    w = M.Weights(cfg)
    t = dict(w.t)
    for l in range(cfg.n_layers):
        for which in (M.WQ, M.WK):
            tid = M.layer_tid(l, which)
            t[tid] = np.zeros_like(t[tid])
    return M.Weights(cfg, tensors=t)


def test_rollout_identity_and_conservation():
    rng = np.random.default_rng(0)
    n = 9
    masked = rng.random(n) < 0.5
    eye = [np.eye(n)] * 3
    assert np.array_equal(X.rollout_scores(eye, masked), masked.astype(float))  # no mixing: visible get 0
    maps = []
    for _ in range(4):  # random row-stochastic maps
        a = rng.random((n, n))
        maps.append(a / a.sum(1, keepdims=True))
    s = X.rollout_scores(maps, masked)
    assert abs(s.sum() - masked.sum()) < 1e-12 and np.all(s >= 0)  # rows sum to 1: mass conserved


@pytest.mark.parametrize("N", [1, 2, 5])
def test_rollout_uniform_closed_form(N):
    n, k = 10, 4
    masked = np.zeros(n, dtype=bool)
    masked[[1, 4, 6, 9]] = True
    s = X.rollout_scores([np.full((n, n), 1.0 / n)] * N, masked)
    vis = ~masked
    assert np.allclose(s[vis], (1 - 0.5 ** N) * k / n, rtol=1e-12, atol=0)


def test_attention_maps_are_row_stochastic():
    w = M.Weights(CFG)
    state = np.random.default_rng(1).integers(0, 12, 15)
    maps = []
    M.hidden(w, state, maps)
    assert len(maps) == CFG.n_layers
    for a in maps:
        assert a.shape == (15, 15) and np.allclose(a.sum(1), 1.0) and np.all(a > 0)


def test_zero_qk_gives_uniform_attention_and_the_prefix():
    w = _zero_qk(CFG)
    sym = np.random.default_rng(2).integers(0, 11, 12)
    maps = []
    M.hidden(w, np.where(np.arange(12) % 2 == 0, 11, sym), maps)
    assert all(np.allclose(a, 1.0 / 12) for a in maps)
    score = X.attention_scores(w, sym)  # n even: each pass masks 6 of 12
    assert np.allclose(score, (1 - 0.5 ** CFG.n_layers) * 6 / 12)
    assert X.attention_positions(w, sym, 4).tolist() == [0, 1, 2, 3]  # all tied: lower positions first


def test_positions_are_the_top_scores():
    w = M.Weights(CFG)
    sym = np.random.default_rng(3).integers(0, 11, 17)
    score = X.attention_scores(w, sym)
    pos = X.attention_positions(w, sym, 5)
    assert pos.size == 5 and np.all(np.diff(pos) > 0)
    rest = np.setdiff1d(np.arange(17), pos)
    assert score[pos].min() >= score[rest].max()
    assert X.attention_positions(w, sym, 40).tolist() == list(range(17))


TINY4 = M.ModelConfig(n_layers=1, d=16, n_heads=2, n_kv_heads=1, ffn=16, vocab=4, dtype="f32", seed=1)


def test_pipeline_round_trips_with_attention_context():
    w = M.Weights(TINY4)
    for pol in (S.Policy(kind=S.UNIFORM, k=2), S.Policy(kind=S.ENTROPY, tau_bits=1.5)):
        for L in range(0, 5):
            for seq in itertools.product(range(4), repeat=L):
                data = bytes(seq)
                blob = PL.compress(w, data, 3, pol, context=(X.ATTENTION, 1, 0))
                assert PL.decompress(w, blob) == data
    data = bytes(np.random.default_rng(4).integers(0, 4, 19).astype(np.uint8))
    blob = PL.compress(w, data, 8, S.Policy(kind=S.TOPK_CONF, k=2, block=4), context=(X.ATTENTION, 2, 0))
    h, _ = C.read(blob)
    assert h.ctx_kind == X.ATTENTION and len(h.ctx_pos) == 4 * 6 and len(h.ctx_data) == 6
    pos = np.frombuffer(h.ctx_pos, dtype="<u4")
    assert pos[:2].tolist() == X.attention_positions(w, np.frombuffer(data[:8], dtype=np.uint8), 2).tolist()
    bad = bytearray(blob)
    bad[80:84] = (100).to_bytes(4, "little")  # a position outside its window
    with pytest.raises(C.ContainerError):
        PL.decompress(w, bytes(bad))
