"""Logits -> integer frequency table, CDF and scores (oracle side).

The paper feeds each committed symbol's predicted distribution to a
statistical coder (rANS; Sec. 2.1, Sec. 3.2, Sec. 4 "Implementation
Details") and scores masked positions by their entropy (Sec. 3.3, entropy
schedule).  It does not say how a distribution becomes the integer table a
coder needs; encoder and decoder must build bit-identical tables from the
same logits, so this module fixes a rule with a single IEEE-exact float32
operation per element followed by integer arithmetic only (no reduction
whose result depends on summation order):

1. ``m = max_v l_v``; ``top`` = lowest v with ``l_v == m``.
2. ``t_v = fl32(fl32(m - l_v) * C)`` with ``C = fl32(256 log2 e)``;
   ``q_v = rint_even(min(t_v, 8191))``  (q_v ~ 256 * log2(p_top / p_v)).
3. ``w_v = T[q_v mod 256] >> (q_v div 256)``,
   ``T[j] = round(2^31 * 2^(-j/256))``  (so w_v ~ 2^31 p_v / p_top).
4. ``W = sum w_v``, ``A = sum w_v q_v``  (exact integers).
5. Precision ``P`` (total 2^P); ``R = 2^P - V``;
   ``f_v = 1 + floor(w_v R / W)``; the remainder
   ``D = R - sum floor(w_v R / W)`` (0 <= D < V) goes to ``top``.
   ``CDF[0] = 0``, ``CDF[v+1] = CDF[v] + f_v``, ``CDF[V] = 2^P``.
6. Scores: confidence key ``W`` (smaller W <=> larger p_max = 2^31/W);
   entropy ``H_q = log2q16(W) - 31*2^16 + floor(2^8 A / W)`` in units of
   2^-16 bit, i.e. the entropy (Sec. 3.3, base 2) of the distribution
   w/W, with ``log2q16`` the digit-by-digit binary logarithm below.

``P = 16`` when V <= 4096 and ``P = 24`` above (a 2^16 total with every
frequency >= 1 cannot hold more than 65536 symbols).

Parity: pinned by CDF invariants (monotone, exact total, all f >= 1),
closed forms (uniform row, single spike), entropy fidelity against
``scipy.stats.entropy`` of the float64 softmax, the table T against an
independent float computation, and ``log2q16`` against ``math.log2``.
"""
import math
from decimal import Decimal, getcontext

import numpy as np

QMAX = 8191


def precision_for_vocab(V):
    return 16 if V <= 4096 else 24


def exp_table():
    """T[j] = round(2^31 * 2^(-j/256)) for j = 0..255, by exact integer roots.

    2^(31 - j/256) = N^(1/256) with N = 2^(7936 - j); the nearest integer x
    satisfies x = floor(root) + [ (2 floor(root) + 1)^256 <= 2^256 N ].
    """
    out = []
    for j in range(256):
        n = 1 << (7936 - j)
        lo, hi = 1, 1 << 32
        while hi - lo > 1:  # floor of the 256th root
            mid = (lo + hi) // 2
            if mid ** 256 <= n:
                lo = mid
            else:
                hi = mid
        x = lo
        if (2 * x + 1) ** 256 <= (n << 256):
            x += 1
        out.append(x)
    return np.array(out, dtype=np.uint64)


def scale_constant():
    """C = the float32 nearest to 256 * log2(e), from 50-digit arithmetic."""
    getcontext().prec = 50
    exact = Decimal(256) / Decimal(2).ln()
    c = np.float32(float(exact))
    # float(exact) is within half a double ulp; confirm the float32 rounding
    # is not ambiguous at that distance.
    lo = np.nextafter(c, np.float32(0))
    hi = np.nextafter(c, np.float32(np.inf))
    assert abs(Decimal(float(c)) - exact) < abs(Decimal(float(lo)) - exact)
    assert abs(Decimal(float(c)) - exact) < abs(Decimal(float(hi)) - exact)
    return c


_T = exp_table()
_C = scale_constant()


def log2q16(W):
    """Digit-by-digit binary logarithm: ~floor(2^16 log2 W) for integers W >= 2^31.

    Normalise W to y in [1, 2) as Q1.31 (y = W >> (n - 31), n = bit length
    - 1), then 16 times: square (Q2.62 -> Q2.31 by truncation); a result
    >= 2 yields bit 1 and is halved.  Works on uint64 arrays.
    """
    W = np.asarray(W, dtype=np.uint64)
    n = np.array([int(w).bit_length() - 1 for w in W.ravel()], dtype=np.uint64).reshape(W.shape)
    assert np.all(n >= 31)
    y = W >> (n - np.uint64(31))
    frac = np.zeros_like(W)
    two = np.uint64(1 << 32)
    for _ in range(16):
        y = (y * y) >> np.uint64(31)
        frac = frac << np.uint64(1)
        big = y >= two
        frac = frac | big.astype(np.uint64)
        y = np.where(big, y >> np.uint64(1), y)
    return (n << np.uint64(16)) + frac


def quantize(logits, P=None):
    """Quantise rows of float32 logits.

    Returns dict with ``cdf`` [rows, V+1] uint32, ``freq`` [rows, V] uint32,
    ``W`` uint64, ``A`` uint64, ``Hq`` int64, ``top`` int64, ``q`` int64.
    """
    l = np.ascontiguousarray(logits, dtype=np.float32)
    if l.ndim == 1:
        l = l[None, :]
    if not np.all(np.isfinite(l)):
        raise ValueError("non-finite logits")
    rows, V = l.shape
    if P is None:
        P = precision_for_vocab(V)
    assert (1 << P) > V and P <= 24
    m = l.max(axis=1)
    top = np.argmax(l == m[:, None], axis=1)
    with np.errstate(over="ignore"):
        t = (m[:, None] - l) * _C  # float32 sub, float32 mul
    q = np.rint(np.minimum(t, np.float32(QMAX))).astype(np.int64)
    w = _T[q & 255] >> (q >> 8).astype(np.uint64)
    Wsum = w.sum(axis=1, dtype=np.uint64)
    A = (w * q.astype(np.uint64)).sum(axis=1, dtype=np.uint64)
    R = np.uint64((1 << P) - V)
    fl = (w * R) // Wsum[:, None]
    D = R - fl.sum(axis=1, dtype=np.uint64)
    f = fl + np.uint64(1)
    f[np.arange(rows), top] += D
    cdf = np.zeros((rows, V + 1), dtype=np.uint64)
    cdf[:, 1:] = np.cumsum(f, axis=1, dtype=np.uint64)
    assert np.all(cdf[:, V] == (1 << P))
    lg = log2q16(Wsum).astype(np.int64)
    ent = ((A // Wsum) << np.uint64(8)) + (((A % Wsum) << np.uint64(8)) // Wsum)
    Hq = lg - (31 << 16) + ent.astype(np.int64)
    return {
        "cdf": cdf.astype(np.uint32),
        "freq": f.astype(np.uint32),
        "W": Wsum,
        "A": A,
        "Hq": Hq,
        "top": top.astype(np.int64),
        "q": q,
        "P": P,
    }


def tau_q(tau_bits):
    """Entropy threshold in the 2^-16-bit units of ``Hq``."""
    return int(math.floor(tau_bits * 65536.0))
