"""Symbol commitment schedules (oracle side), Sec. 3.3.

Two schedules are on the path:

* ``TOPK_CONF`` -- max-confidence top-k inside left-to-right blocks.  The
  paper builds on LLaDA (Sec. 1, Sec. 4) and the workloads here commit k
  positions per step by maximum confidence within a block.  Reading: the
  window is cut into ceil(L / B) blocks of B positions (B = 0 means one
  block of L); the candidates are the still-masked positions of the
  leftmost block that has any; the min(k, #candidates) candidates with the
  smallest (W, position) are committed (smaller W <=> larger max
  probability).  Selection never spills into the next block within a step.
* ``ENTROPY`` -- entropy-based schedule (Sec. 3.3, paragraph 3): commit every
  masked position with H <= tau; if fewer than m qualify, commit the m
  lowest-entropy positions instead.  Ties in entropy are broken by position.
  An optional cap ``k_max`` (0 = none) keeps only the k_max lowest-entropy
  positions of the selection.

Both are deterministic given their hyper-parameters, so the decoder replays
them from the header alone (Sec. 3.3, last paragraph).  Within a step the
committed symbols are coded in ascending position.

Parity: pinned by brute force over all k-subsets of small candidate sets
(with forced ties), the coverage constraint sum u_k = n (Sec. 3.3), and
K = n / k for fixed k.
"""
from dataclasses import dataclass

import numpy as np

TOPK_CONF = 0
ENTROPY = 1


@dataclass(frozen=True)
class Policy:
    kind: int = TOPK_CONF
    k: int = 1
    block: int = 0
    tau_bits: float = 0.0
    k_min: int = 1
    k_max: int = 0


def active_block(masked, block):
    """(start, end) of the leftmost block that still has a masked position."""
    L = len(masked)
    B = L if block == 0 else block
    idx = np.flatnonzero(masked)
    if idx.size == 0:
        return None
    start = (idx[0] // B) * B
    return start, min(start + B, L)


def candidates(masked, policy):
    """Positions whose distributions the schedule looks at in this step."""
    masked = np.asarray(masked, dtype=bool)
    if policy.kind == TOPK_CONF:
        blk = active_block(masked, policy.block)
        if blk is None:
            return np.zeros(0, dtype=np.int64)
        s, e = blk
        return s + np.flatnonzero(masked[s:e])
    return np.flatnonzero(masked)


def smallest(keys, pos, count):
    """The ``count`` positions with the smallest (key, position), any order."""
    order = sorted(range(len(pos)), key=lambda i: (int(keys[i]), int(pos[i])))
    return [int(pos[i]) for i in order[:count]]


def select(masked, key_of_pos, policy, tau_q=None):
    """Positions committed at this step, ascending.

    ``key_of_pos`` maps position -> score: ``W`` for TOPK_CONF, ``Hq`` for
    ENTROPY.  ``tau_q`` is the threshold in Hq units.
    """
    cand = candidates(masked, policy)
    if cand.size == 0:
        return []
    keys = [int(key_of_pos[int(p)]) for p in cand]
    if policy.kind == TOPK_CONF:
        chosen = smallest(keys, cand, min(policy.k, len(cand)))
    else:
        below = [int(p) for p, k in zip(cand, keys) if k <= tau_q]
        if len(below) < policy.k_min:
            chosen = smallest(keys, cand, min(policy.k_min, len(cand)))
        else:
            chosen = below
        if policy.k_max and len(chosen) > policy.k_max:
            kk = [int(key_of_pos[p]) for p in chosen]
            chosen = smallest(kk, chosen, policy.k_max)
    return sorted(chosen)
