"""Seeded synthetic inputs shaped like the paper's workloads.

The paper measures on the first 1 MB / 10 MB of enwik8 (Sec. 4) with the
LLaDA tokenizer; neither is available here, so these sources stand in for
them with the shapes and statistics of the workloads:

* ``markov_bytes``  -- order-2 Markov bytes: for every context (a, b) the
  next-byte distribution is a seeded permutation of 0..255 with
  probabilities proportional to rank^-s (Zipf, s = 1.1).
* ``zipf_bigram_tokens`` -- token ids in [0, V): next = pi_a(rank) with
  rank ~ Zipf(s = 1.05) over V and pi_a(r) = (alpha_a r + beta_a) mod V an
  affine bijection keyed by the previous token a (alpha_a coprime to V).
* ``synthetic_logits`` -- float32 logits for driving the quantizer,
  selector and coder directly: N(0, sigma) per entry plus, per row, a spike
  of +U(0, spike_max) at a uniformly drawn column.
* ``spiked_rows`` -- the isolated quantiser workload's rows: N(0, 3) plus a
  spike of +U(5, 15) at a uniformly drawn column.

This module holds input generation only (none of the method's arithmetic)
and is shared by the tests, the benchmark and the oracle-side checks.
"""
import numpy as np


def _zipf_cdf(n, s):
    w = np.arange(1, n + 1, dtype=np.float64) ** (-s)
    c = np.cumsum(w)
    return c / c[-1]


def _zipf_ranks(rng, count, n, s):
    cdf = _zipf_cdf(n, s)
    r = np.searchsorted(cdf, rng.random(count), side="right")
    return np.minimum(r, n - 1)


def markov_bytes(n, seed=0, s=1.1):
    """``n`` bytes from the seeded order-2 Markov / Zipf(s) source."""
    rng = np.random.default_rng([seed, 0x6D61726B])
    perm = np.argsort(rng.random((65536, 256)), axis=1).astype(np.uint8)
    ranks = _zipf_ranks(rng, n, 256, s)
    out = np.empty(n, dtype=np.uint8)
    a, b = rng.integers(0, 256, 2)
    flat = perm.reshape(-1)
    # sequential by nature: each byte's row depends on the two before it
    ctx = int(a) * 256 + int(b)
    for i in range(n):
        nxt = flat[ctx * 256 + ranks[i]]
        out[i] = nxt
        ctx = ((ctx & 0xFF) << 8) | int(nxt)
    return out.tobytes()


def _affine_keys(V, seed):
    rng = np.random.default_rng([seed, 0x7A697066])
    alpha = rng.integers(1, V, V, dtype=np.int64)
    bad = np.gcd(alpha, V) != 1
    while bad.any():
        alpha[bad] = rng.integers(1, V, int(bad.sum()), dtype=np.int64)
        bad = np.gcd(alpha, V) != 1
    beta = rng.integers(0, V, V, dtype=np.int64)
    return alpha, beta


def zipf_bigram_tokens(n, V, seed=0, s=1.05):
    """``n`` token ids (uint32) from the seeded Zipf bigram source."""
    alpha, beta = _affine_keys(V, seed)
    rng = np.random.default_rng([seed, 0x746F6B73])
    ranks = _zipf_ranks(rng, n, V, s)
    out = np.empty(n, dtype=np.uint32)
    prev = int(rng.integers(0, V))
    for i in range(n):
        prev = int((alpha[prev] * int(ranks[i]) + beta[prev]) % V)
        out[i] = prev
    return out


def tokens_to_bytes(tokens):
    return np.asarray(tokens, dtype="<u4").tobytes()


def synthetic_logits(seed, chunk, step, L, V, sigma=1.0, spike_max=20.0):
    """float32 logits [L, V] for window ``chunk`` at step ``step``."""
    rng = np.random.default_rng([seed, chunk, step, 0x6C6F6769])
    x = rng.normal(0.0, sigma, (L, V))
    col = rng.integers(0, V, L)
    x[np.arange(L), col] += rng.uniform(0.0, spike_max, L)
    return x.astype(np.float32)


def spiked_rows(seed, row0, nrows, V):
    """Rows row0 .. row0+nrows-1 of the isolated quantiser workload (float32).

    Each row is generated from its own seeded stream, so any subset of rows
    can be regenerated without the others.
    """
    out = np.empty((nrows, V), dtype=np.float32)
    for i in range(nrows):
        rng = np.random.default_rng([seed, row0 + i, 0x73706B])
        x = rng.normal(0.0, 3.0, V)
        x[rng.integers(0, V)] += rng.uniform(5.0, 15.0)
        out[i] = x.astype(np.float32)
    return out


def entropy_rate_markov(seed=0, s=1.1):
    """Entropy rate (bits/byte) of the order-2 source: H of the Zipf row."""
    w = np.arange(1, 257, dtype=np.float64) ** (-s)
    p = w / w.sum()
    return float(-(p * np.log2(p)).sum())


def entropy_rate_zipf_tokens(V, s=1.05):
    """Entropy rate (bits/token) of the bigram source: H of Zipf(s) over V."""
    w = np.arange(1, V + 1, dtype=np.float64) ** (-s)
    p = w / w.sum()
    return float(-(p * np.log2(p)).sum())


__all__ = [
    "markov_bytes", "zipf_bigram_tokens", "tokens_to_bytes", "synthetic_logits", "spiked_rows",
    "entropy_rate_markov", "entropy_rate_zipf_tokens",
]
