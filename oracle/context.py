"""Initial context (oracle side), Sec. 3.4.

``c`` symbols of each window are left unmasked before the first step and
stored in the compressed file; the schedules then cover only the masked
positions.  Two of the paper's policies are built:

* ``CONTIGUOUS`` -- the first c positions (the classical prefix).
* ``ATTENTION`` -- attention-based context (Sec. 3.4, policy 4): two forwards,
  one with the even positions masked and one with the odd ones masked (the
  others showing their true symbols), score every position by the attention
  it receives from the masked ones, aggregated over the layers by Attention
  Rollout (Abnar & Zuidema 2020): with A_l the head-averaged attention of
  layer l and Ã_l = A_l / 2 + I / 2, R = Ã_N ... Ã_1 and
  score_j = sum over masked i of R[i, j], read from the pass in which j is
  visible.  The c highest scores (ties: lower position) are the context.  The
  positions depend on the data, so the file stores them.
* ``RANDOM`` -- c positions drawn uniformly at random.  Reading: the draw is
  a partial Fisher-Yates shuffle (Durstenfeld 1964) of [0, n): for i = 0 ..
  c-1, swap slot i with slot i + (o_i mod (n - i)), where o_i is output i of
  the SplitMix64 stream of the window (state = output w of the stream with
  state ``seed``, as for the weights); the first c slots, sorted, are the
  context.  The header stores ``seed``, so the positions cost no space; the
  symbols are stored raw.

A window shorter than c keeps all its symbols as context (c_eff = min(c, n)).

Parity: pinned by distinct/sorted/in-range positions, the contiguous prefix,
the uniformity of the random draw (chi-square over many windows), and round
trips with every schedule.
"""
import numpy as np

from .weights import stream_outputs, tensor_state

NONE = 0
CONTIGUOUS = 1
RANDOM = 2
ATTENTION = 3


def positions(kind, c, seed, n, window):
    """Sorted context positions of window ``window`` (length ``n``)."""
    ce = min(c, n)
    if kind == NONE or ce == 0:
        return np.zeros(0, dtype=np.int64)
    if kind == CONTIGUOUS:
        return np.arange(ce, dtype=np.int64)
    if kind != RANDOM:
        raise ValueError("positions of this context kind depend on the data (see attention_positions)")
    out = stream_outputs(np.uint64(tensor_state(seed, window)), 0, ce)
    slot = list(range(n))
    for i in range(ce):
        j = i + int(out[i]) % (n - i)
        slot[i], slot[j] = slot[j], slot[i]
    return np.array(sorted(slot[:ce]), dtype=np.int64)


def rollout_scores(maps, masked):
    """score_j = sum_i masked_i R[i, j], R = Ã_N ... Ã_1, Ã_l = A_l / 2 + I / 2."""
    v = np.asarray(masked, dtype=np.float64)
    for A in reversed(maps):
        v = 0.5 * (v @ A) + 0.5 * v
    return v


def attention_scores(wts, symbols):
    """Per-position importance from the two complementary masked forwards."""
    from .model import hidden
    n = len(symbols)
    V = wts.cfg.vocab
    score = np.zeros(n)
    for parity in (0, 1):  # parity 0: even positions masked, odd visible
        masked = (np.arange(n) % 2) == parity
        state = np.where(masked, V, np.asarray(symbols, dtype=np.int64))
        maps = []
        hidden(wts, state, maps)
        s = rollout_scores(maps, masked)
        score[~masked] = s[~masked]
    return score


def attention_positions(wts, symbols, c):
    """The min(c, n) positions with the highest attention scores, ascending."""
    n = len(symbols)
    ce = min(c, n)
    if ce == 0:
        return np.zeros(0, dtype=np.int64)
    score = attention_scores(wts, symbols)
    order = sorted(range(n), key=lambda j: (-score[j], j))
    return np.array(sorted(order[:ce]), dtype=np.int64)
