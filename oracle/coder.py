"""Range coder with minimal termination (oracle side).

The paper codes each committed symbol under its predicted distribution with
a statistical coder (rANS, Sec. 2.1 and Sec. 4 "Implementation Details").
The coder here is a range coder over the same integer tables (total 2^P):
it has the same interface (encode (c, f) pairs, decode slot -> symbol) and
adds no per-stream flush beyond the bits that identify the final interval,
so a stream of n symbols costs at most sum -log2(f/2^P) + 1 bit plus
n * 2^(P-48) * log2(e) bits of range truncation.

State (encoder): ``low`` and ``rng`` are the current interval in a 64-bit
window below the emitted 16-bit units; the initial interval is
[0, 2^64 - 1).

* encode(c, f): ``r = rng >> P; low += r * c; rng = r * f``; a carry out of
  the window adds 1 to the emitted units (propagating through 0xFFFF);
  while ``rng < 2^48`` emit ``low >> 48`` and shift both left by 16.
* finish: the shortest t (0..64) for which a multiple ``v`` of 2^(64-t)
  lies in [low, low + rng); emit the top t bits of v (after a possible carry).
  Bit length = 16 * units + t; bytes are the units big-endian followed by
  the t bits MSB-first, zero-padded.
* decoder: keeps ``val = code - low`` (code = the stream read as a number,
  zero beyond its end) and ``rng``; ``slot = val // (rng >> P)`` selects the
  symbol s with CDF[s] <= slot < CDF[s+1]; a slot >= 2^P cannot come from
  the encoder and marks the stream corrupt.

Parity: pinned by round trips (random, exhaustive tiny alphabets, carry
chains), and the per-stream length bound against the ideal code length.
"""
MASK64 = (1 << 64) - 1
RENORM = 1 << 48


class CorruptStream(Exception):
    pass


class Encoder:
    def __init__(self, P):
        self.P = P
        self.low = 0
        self.rng = MASK64
        self.units = []

    def _carry(self):
        i = len(self.units) - 1
        while True:
            assert i >= 0, "carry out of the stream (interval left [0, 1))"
            self.units[i] = (self.units[i] + 1) & 0xFFFF
            if self.units[i] != 0:
                return
            i -= 1

    def encode(self, c, f):
        assert f >= 1 and c + f <= (1 << self.P)
        r = self.rng >> self.P
        self.low += r * c
        self.rng = r * f
        if self.low > MASK64:
            self.low &= MASK64
            self._carry()
        while self.rng < RENORM:
            self.units.append(self.low >> 48)
            self.low = (self.low << 16) & MASK64
            self.rng <<= 16

    def finish(self):
        """Return (bit_length, bytes)."""
        hi = self.low + self.rng - 1  # largest value inside the interval
        for t in range(65):
            g = 1 << (64 - t)
            v = -(-self.low // g) * g  # smallest multiple of g >= low
            if v <= hi:
                break
        if v > MASK64:
            v &= MASK64
            self._carry()
        tail_bits = t
        tail = v >> (64 - t) if t else 0
        bits = 16 * len(self.units) + tail_bits
        out = bytearray()
        for u in self.units:
            out += bytes((u >> 8, u & 0xFF))
        nb = (tail_bits + 7) // 8
        if nb:
            tail_aligned = tail << (8 * nb - tail_bits)
            out += tail_aligned.to_bytes(nb, "big")
        assert len(out) == (bits + 7) // 8
        return bits, bytes(out)


class Decoder:
    def __init__(self, data, bits, P):
        self.P = P
        self.data = data
        self.nbytes = (bits + 7) // 8
        assert len(data) >= self.nbytes
        self.pos = 0  # next unit index
        self.rng = MASK64
        self.val = 0
        for _ in range(4):
            self.val = (self.val << 16) | self._unit()

    def _unit(self):
        i = 2 * self.pos
        self.pos += 1
        hi = self.data[i] if i < self.nbytes else 0
        lo = self.data[i + 1] if i + 1 < self.nbytes else 0
        return (hi << 8) | lo

    def decode(self, cdf):
        """Decode one symbol with ``cdf`` (length V+1, CDF[V] = 2^P)."""
        r = self.rng >> self.P
        slot = self.val // r
        if slot >= (1 << self.P):
            raise CorruptStream("slot outside the table")
        lo, hi = 0, len(cdf) - 1  # find s with cdf[s] <= slot < cdf[s+1]
        while hi - lo > 1:
            mid = (lo + hi) // 2
            if cdf[mid] <= slot:
                lo = mid
            else:
                hi = mid
        s = lo
        self.val -= r * int(cdf[s])
        self.rng = r * (int(cdf[s + 1]) - int(cdf[s]))
        while self.rng < RENORM:
            self.val = ((self.val << 16) | self._unit()) & MASK64
            self.rng <<= 16
        return s
