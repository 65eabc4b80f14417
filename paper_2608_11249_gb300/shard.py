"""Data-parallel sharding of the compression path across ranks (one GPU each).

Windows are compressed independently (Sec. 4: non-overlapping windows also
allow processing across several GPUs), so an input is split into contiguous,
window-aligned shards, one per rank, with no communication while coding.  The
only exchange is at the end: the ranks' containers are gathered, in rank
order, into one multi-part file:

    "DLMP" | u32 n_parts | n_parts x u64 part size | parts (each a DLMZ container)

Each part decompresses on its own, so decompression shards the same way.
"""
import struct

MAGIC = b"DLMP"


def shard_range(n_bytes, chunk_bytes, rank, world):
    """Byte range [lo, hi) of rank's shard: whole windows, balanced across ranks."""
    if chunk_bytes <= 0 or world <= 0 or not 0 <= rank < world:
        raise ValueError("bad shard arguments")
    n_windows = -(-n_bytes // chunk_bytes)
    per, extra = divmod(n_windows, world)
    w0 = rank * per + min(rank, extra)
    w1 = w0 + per + (1 if rank < extra else 0)
    return min(w0 * chunk_bytes, n_bytes), min(w1 * chunk_bytes, n_bytes)


def rank_batch(step, rank, world, n_batches):
    """Batch index a rank codes at a benchmark step (ranks never share a batch in a step)."""
    return (step * world + rank) % n_batches


def pack_parts(parts):
    head = MAGIC + struct.pack("<I", len(parts)) + b"".join(struct.pack("<Q", len(p)) for p in parts)
    return head + b"".join(parts)


def unpack_parts(blob):
    if len(blob) < 8 or blob[:4] != MAGIC:
        raise ValueError("not a multi-part container")
    (n,) = struct.unpack_from("<I", blob, 4)
    pos = 8 + 8 * n
    if len(blob) < pos:
        raise ValueError("truncated multi-part index")
    sizes = struct.unpack_from("<%dQ" % n, blob, 8)
    parts = []
    for s in sizes:
        if pos + s > len(blob):
            raise ValueError("truncated part")
        parts.append(bytes(blob[pos:pos + s]))
        pos += s
    if pos != len(blob):
        raise ValueError("trailing bytes")
    return parts


def gather_parts(part, group=None):
    """Gather every rank's container to rank 0 (None on the other ranks)."""
    import torch.distributed as dist
    world = dist.get_world_size(group)
    out = [None] * world if dist.get_rank(group) == 0 else None
    dist.gather_object(part, out, dst=0, group=group)
    return pack_parts(out) if out is not None else None


def max_over_ranks(value, group=None, device=None):
    """Max of a per-rank float (the slowest rank sets a step's time).

    ``device`` is where the reduction tensor lives (a CUDA device for NCCL).
    """
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return float(t.item())
