"""Initial context (oracle side), Sec. 3.4.

``c`` symbols of each window are left unmasked before the first step and
stored in the compressed file; the schedules then cover only the masked
positions.  Two of the paper's policies are built:

* ``CONTIGUOUS`` -- the first c positions (the classical prefix).
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


def positions(kind, c, seed, n, window):
    """Sorted context positions of window ``window`` (length ``n``)."""
    ce = min(c, n)
    if kind == NONE or ce == 0:
        return np.zeros(0, dtype=np.int64)
    if kind == CONTIGUOUS:
        return np.arange(ce, dtype=np.int64)
    if kind != RANDOM:
        raise ValueError("unknown context kind")
    out = stream_outputs(np.uint64(tensor_state(seed, window)), 0, ce)
    slot = list(range(n))
    for i in range(ce):
        j = i + int(out[i]) % (n - i)
        slot[i], slot[j] = slot[j], slot[i]
    return np.array(sorted(slot[:ce]), dtype=np.int64)
