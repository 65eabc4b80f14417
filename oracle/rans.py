"""rANS coder (oracle side), the paper's statistical coder (Sec. 2.1, Sec. 4).

Range asymmetric numeral systems (Duda 2013) with a 64-bit state and 32-bit
output words, over the same integer tables (total 2^P, P <= 24) as the range
coder.  Reading (the paper names rANS but not its parameters): state
x in [L, 2^32 L), L = 2^31;

* encode(c, f) (symbols in reverse decode order): if x >= 2^(63-P) f, emit
  the low 32 bits of x and shift x right by 32; then
  x = floor(x / f) 2^P + (x mod f) + c.
* flush: the final state, 8 bytes big-endian, leads the stream; the emitted
  words follow in reverse order of emission (4 bytes big-endian each), so the
  decoder reads forward.  Bit length = 64 + 32 * words.
* decode: slot = x mod 2^P selects s with CDF[s] <= slot < CDF[s+1];
  x = f (x >> P) + slot - c; if x < L, x = 2^32 x + next word (zero beyond the
  stream).

rANS is last-in first-out while the pipeline decodes step by step, so the
encoder buffers the (c, f) pairs of a window and codes them in reverse when
the window is finished.  A stream costs the ideal sum -log2(f / 2^P) plus at
most about 64 bits (the flushed state; its first 31 bits carry no
information).

Parity: pinned by hand-computed streams of one symbol, round trips (random,
exhaustive tiny alphabets, extreme frequencies), the length bound, and
agreement of decoded symbols with the range coder's.
"""
L_STATE = 1 << 31
MASK32 = (1 << 32) - 1


class CorruptStream(Exception):
    pass


class Encoder:
    def __init__(self, P):
        assert 1 <= P <= 31
        self.P = P
        self.pairs = []

    def encode(self, c, f):
        assert f >= 1 and c + f <= (1 << self.P)
        self.pairs.append((c, f))

    def finish(self):
        """Return (bit_length, bytes)."""
        P = self.P
        x = L_STATE
        words = []
        for c, f in reversed(self.pairs):
            if x >= ((L_STATE >> P) << 32) * f:
                words.append(x & MASK32)
                x >>= 32
            x = ((x // f) << P) + (x % f) + c
        out = x.to_bytes(8, "big") + b"".join(w.to_bytes(4, "big") for w in reversed(words))
        return 64 + 32 * len(words), out


class Decoder:
    def __init__(self, data, bits, P):
        self.P = P
        self.data = data
        self.nbytes = (bits + 7) // 8
        assert len(data) >= self.nbytes
        self.x = int.from_bytes(self._take(8), "big")
        self.pos = 8

    def _take(self, n, at=0):
        return bytes(self.data[i] if i < self.nbytes else 0 for i in range(at, at + n))

    def decode(self, cdf):
        """Decode one symbol with ``cdf`` (length V+1, CDF[V] = 2^P)."""
        P = self.P
        slot = self.x & ((1 << P) - 1)
        lo, hi = 0, len(cdf) - 1  # find s with cdf[s] <= slot < cdf[s+1]
        while hi - lo > 1:
            mid = (lo + hi) // 2
            if cdf[mid] <= slot:
                lo = mid
            else:
                hi = mid
        s = lo
        c, f = int(cdf[s]), int(cdf[s + 1]) - int(cdf[s])
        self.x = f * (self.x >> P) + slot - c
        if self.x < L_STATE:
            self.x = (self.x << 32) | int.from_bytes(self._take(4, self.pos), "big")
            self.pos += 4
        return s
