"""Symbol ranking (oracle side), the paper's ranking pipeline (Definition
"Symbol Ranking"; Sec. 4: ranks written as byte-aligned varints).

Each coded symbol is replaced by its rank under the step's distribution.
Reading (the definition orders symbols by probability and leaves ties open):
the order is by the quantised integer frequency f (the coders' table, so
every implementation agrees), larger first, ties by symbol index:
rank(s) = #{v : f_v > f_s} + #{v < s : f_v = f_s}.  Ranks are written as
LEB128 varints (7 bits per byte, low group first), one stream per window.
The general-purpose back-end compressor the paper applies to the rank bytes
is a third-party program and not part of this path.

Parity: pinned by brute-force sorting, the identity symbol -> rank -> symbol
over whole tables, varint round trips and pipeline round trips.
"""
import numpy as np


class CorruptStream(Exception):
    pass


def rank_of(freq, s):
    f = freq[s]
    return int(np.sum(freq > f) + np.sum(freq[:s] == f))


def symbol_of(freq, r):
    order = sorted(range(len(freq)), key=lambda v: (-int(freq[v]), v))
    return order[r]


def varint(n):
    out = bytearray()
    while True:
        b = n & 0x7F
        n >>= 7
        if n:
            out.append(b | 0x80)
        else:
            out.append(b)
            return bytes(out)


class Encoder:
    def __init__(self, P):
        self.out = bytearray()

    def encode_rank(self, freq, s):
        self.out += varint(rank_of(np.asarray(freq), s))

    def finish(self):
        return 8 * len(self.out), bytes(self.out)


class Decoder:
    def __init__(self, data, bits, P):
        self.data = bytes(data[:(bits + 7) // 8])
        self.pos = 0

    def decode(self, cdf):
        n, shift = 0, 0
        while True:
            if self.pos >= len(self.data) or shift > 28:
                raise CorruptStream("truncated rank")
            b = self.data[self.pos]
            self.pos += 1
            n |= (b & 0x7F) << shift
            shift += 7
            if not b & 0x80:
                break
        freq = np.diff(np.asarray(cdf, dtype=np.int64))
        if n >= freq.size:
            raise CorruptStream("rank outside the alphabet")
        return symbol_of(freq, n)
