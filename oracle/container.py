"""Compressed-file container (oracle side).

Only the header is side information: the schedule's hyper-parameters
(Sec. 3.3, last paragraph) and the window size w (Sec. 4, "Implementation
Details") are stored so the decompressor replays every decision.  Layout
(little-endian, 64-byte fixed header):

    off size field
      0   4  magic "DLMZ"
      4   1  version (1; 2 when the windows carry an initial context)
      5   1  coder (0 = range coder, 1 = rANS, 2 = symbol ranks as varints)
      6   1  P, CDF precision bits
      7   1  policy kind (0 = top-k confidence, 1 = entropy, 2 = uniform block,
             3 = progressive; for 3 the block field holds r in 16.16 fixed point)
      8   8  model fingerprint (FNV-1a 64 of the model configuration)
     16   4  V (vocabulary size)
     20   4  chunk_len (the window w)
     24   4  batch_chunks (chunks per forward batch)
     28   4  k          32 4 block      36 4 tau_q (2^-16 bit)
     40   4  k_min      44 4 k_max
     48   8  n_symbols
     56   4  n_chunks
     60   4  checksum: CRC-32 (IEEE) of the little-endian CRC-32s of the
             windows' input bytes, window by window
   version 2 only (initial context, Sec. 3.4: the visible symbols are stored):
     64   4  context kind (1 = contiguous, 2 = random, 3 = attention-based)
     68   4  c, context symbols per window
     72   8  seed of the random positions
     80   -  kind 3 only: the context positions, window by window (min(c, window
             length) each, ascending, u32)
      -   -  the context symbols, window by window (min(c, window length) each,
             ascending position; 1 byte each when V <= 256, else u32)
      -   -  n_chunks LEB128 varints: bit length of each chunk's stream
      -   -  streams, chunk by chunk, ceil(bits / 8) bytes each

Parity: pinned by parse(write(h)) == h and by the corruption tests
(bad magic / version / fingerprint / truncated lengths or streams).
"""
import struct
import zlib
from dataclasses import dataclass

MAGIC = b"DLMZ"
VERSION = 1
VERSION_CONTEXT = 2
HEADER = struct.Struct("<4sBBBBQIIIIIIIIQII")
EXT = struct.Struct("<IIQ")
assert HEADER.size == 64 and EXT.size == 16


class ContainerError(Exception):
    pass


class FingerprintError(ContainerError):
    pass


def fnv1a64(data):
    h = 0xCBF29CE484222325
    for b in data:
        h ^= b
        h = (h * 0x100000001B3) & ((1 << 64) - 1)
    return h


def fingerprint(cfg):
    """FNV-1a 64 over the packed model configuration."""
    dt = 1 if cfg.dtype == "bf16" else 0
    blob = struct.pack(
        "<IIIIIIIffQ", cfg.n_layers, cfg.d, cfg.n_heads, cfg.n_kv_heads, cfg.ffn, cfg.vocab, dt,
        cfg.rope_theta, cfg.norm_eps, cfg.seed)
    return fnv1a64(blob)


@dataclass
class Header:
    P: int
    kind: int
    fingerprint: int
    vocab: int
    chunk_len: int
    batch_chunks: int
    k: int
    block: int
    tau_q: int
    k_min: int
    k_max: int
    n_symbols: int
    n_chunks: int
    crc32: int
    coder: int = 0
    ctx_kind: int = 0
    ctx_c: int = 0
    ctx_seed: int = 0
    ctx_data: bytes = b""
    ctx_pos: bytes = b""


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


def read_varint(buf, pos):
    n = 0
    shift = 0
    while True:
        if pos >= len(buf) or shift > 63:
            raise ContainerError("truncated length table")
        b = buf[pos]
        pos += 1
        n |= (b & 0x7F) << shift
        shift += 7
        if not b & 0x80:
            return n, pos


def write(h, streams):
    """``streams``: list of (bits, bytes) per chunk."""
    ver = VERSION_CONTEXT if h.ctx_c else VERSION
    out = bytearray(HEADER.pack(
        MAGIC, ver, h.coder, h.P, h.kind, h.fingerprint, h.vocab, h.chunk_len, h.batch_chunks, h.k,
        h.block, h.tau_q, h.k_min, h.k_max, h.n_symbols, h.n_chunks, h.crc32))
    if ver == VERSION_CONTEXT:
        out += EXT.pack(h.ctx_kind, h.ctx_c, h.ctx_seed) + h.ctx_pos + h.ctx_data
    for bits, _ in streams:
        out += varint(bits)
    for bits, data in streams:
        assert len(data) == (bits + 7) // 8
        out += data
    return bytes(out)


def read(buf):
    """Return (Header, [(bits, bytes)]); raise ContainerError on bad input."""
    if len(buf) < HEADER.size:
        raise ContainerError("truncated header")
    f = HEADER.unpack_from(buf, 0)
    if f[0] != MAGIC:
        raise ContainerError("bad magic")
    if f[1] not in (VERSION, VERSION_CONTEXT):
        raise ContainerError("unsupported version")
    if f[2] not in (0, 1, 2):
        raise ContainerError("unknown coder")
    h = Header(*f[3:], coder=f[2])
    if h.chunk_len == 0 and h.n_symbols:
        raise ContainerError("zero chunk length")
    exp_chunks = (h.n_symbols + h.chunk_len - 1) // h.chunk_len if h.chunk_len else 0
    if h.n_chunks != exp_chunks:
        raise ContainerError("chunk count does not match the symbol count")
    pos = HEADER.size
    if f[1] == VERSION_CONTEXT:
        if len(buf) < pos + EXT.size:
            raise ContainerError("truncated header")
        h.ctx_kind, h.ctx_c, h.ctx_seed = EXT.unpack_from(buf, pos)
        pos += EXT.size
        if h.ctx_kind not in (1, 2, 3) or h.ctx_c == 0:
            raise ContainerError("bad context")
        sb = 1 if h.vocab <= 256 else 4
        full, tail = divmod(h.n_symbols, h.chunk_len)
        count = full * min(h.ctx_c, h.chunk_len) + min(h.ctx_c, tail)
        if h.ctx_kind == 3:
            if pos + 4 * count > len(buf):
                raise ContainerError("truncated context")
            h.ctx_pos = bytes(buf[pos:pos + 4 * count])
            pos += 4 * count
        nb = sb * count
        if pos + nb > len(buf):
            raise ContainerError("truncated context")
        h.ctx_data = bytes(buf[pos:pos + nb])
        pos += nb
    lens = []
    for _ in range(h.n_chunks):
        n, pos = read_varint(buf, pos)
        lens.append(n)
    streams = []
    for bits in lens:
        nb = (bits + 7) // 8
        if pos + nb > len(buf):
            raise ContainerError("truncated stream")
        streams.append((bits, bytes(buf[pos:pos + nb])))
        pos += nb
    if pos != len(buf):
        raise ContainerError("trailing bytes")
    return h, streams


def crc32(data):
    return zlib.crc32(data) & 0xFFFFFFFF


def window_checksum(data, window_bytes):
    """CRC-32 of the per-window CRC-32s (each little-endian u32)."""
    if window_bytes == 0:
        return crc32(b"")
    crcs = b"".join(struct.pack("<I", crc32(data[i:i + window_bytes]))
                    for i in range(0, len(data), window_bytes))
    return crc32(crcs)
