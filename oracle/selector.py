"""Symbol commitment schedules (oracle side), Sec. 3.3.

Four schedules:

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

* ``UNIFORM`` -- uniform block schedule (Sec. 3.3, paragraph 1): with K = ``k``
  steps, u = floor(n / K) symbols are committed per step in contiguous
  left-to-right order (n = masked positions of the window).  Reading: K is
  capped at n, and the last step commits the remainder n - (K - 1) u, so
  exactly K forwards cover the window.
* ``PROGRESSIVE`` -- geometric schedule (Sec. 3.3, paragraph 2): u_k =
  round(u_1 r^(k-1)) symbols left to right, u_1 = ``k``.  Reading: r is
  carried as a 16.16 fixed-point integer ``growth_q16`` and the sequence as
  x_1 = u_1 2^16, x_(k+1) = floor(x_k r_q / 2^16) (exact integers, so every
  implementation agrees); u_k = max(1, floor((x_k + 2^15) / 2^16)), and the
  last step takes what remains.  r = 1 gives u_k = u_1 (uniform steps).

All are deterministic given their hyper-parameters, so the decoder replays
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
UNIFORM = 2
PROGRESSIVE = 3


@dataclass(frozen=True)
class Policy:
    kind: int = TOPK_CONF
    k: int = 1
    block: int = 0
    tau_bits: float = 0.0
    k_min: int = 1
    k_max: int = 0
    growth_q16: int = 65536


def schedule_sizes(n, policy):
    """u_1, ..., u_K of the left-to-right schedules for n masked positions (sum = n)."""
    if n <= 0:
        return []
    if policy.kind == UNIFORM:
        K = min(policy.k, n)
        u = n // K
        return [u] * (K - 1) + [n - (K - 1) * u]
    if policy.kind == PROGRESSIVE:
        sizes, rem, x = [], n, policy.k << 16
        while rem > 0:
            u = max(1, (x + (1 << 15)) >> 16)
            u = min(u, rem)
            sizes.append(u)
            rem -= u
            x = min((x * policy.growth_q16) >> 16, n << 16)
        return sizes
    raise ValueError("not a left-to-right schedule")


def leftmost(masked, count):
    """The ``count`` leftmost masked positions."""
    return np.flatnonzero(np.asarray(masked, dtype=bool))[:count]


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
