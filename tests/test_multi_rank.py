"""World-size-2 gloo tests of the sharded (multi-GPU) path, on the CPU.

Each rank compresses its shard of windows independently (the oracle stands
in for the per-rank GPU codec), rank 0 gathers the parts into one
multi-part container, and every part decompresses back to its shard.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2608_11249_gb300 import shard


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, data, chunk, results):
    import torch.distributed as dist

    from oracle import model as OM
    from oracle import pipeline as OP
    from oracle import selector as OS

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = OM.Weights(OM.ModelConfig(1, 16, 2, 2, 16, 256, "f32", seed=4))
        lo, hi = shard.shard_range(len(data), chunk, rank, world)
        part = OP.compress(w, data[lo:hi], chunk, OS.Policy(kind=OS.TOPK_CONF, k=3, block=8))
        blob = shard.gather_parts(part)
        t = shard.max_over_ranks(10.0 + rank)
        if rank == 0:
            parts = shard.unpack_parts(blob)
            out = b"".join(OP.decompress(w, p) for p in parts)
            results[rank] = (out == data, len(parts), t)
        else:
            results[rank] = (blob is None, 0, t)
    finally:
        dist.destroy_process_group()


def test_two_rank_shard_compress_gather_decompress():
    data = bytes((i * 37 + (i >> 3)) & 0xFF for i in range(75))
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    results = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, data, 16, results)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    ok0, nparts, t0 = results[0]
    ok1, _, t1 = results[1]
    assert ok0 and nparts == 2 and ok1
    assert t0 == t1 == 11.0  # max over ranks


@pytest.mark.parametrize("n,chunk,world", [(0, 8, 2), (7, 8, 2), (75, 16, 2), (1000, 64, 3), (100, 10, 8)])
def test_shard_ranges_cover_input_in_whole_windows(n, chunk, world):
    spans = [shard.shard_range(n, chunk, r, world) for r in range(world)]
    assert spans[0][0] == 0 and spans[-1][1] == n
    for (a, b), (c, _) in zip(spans, spans[1:]):
        assert b == c and a <= b
    for a, b in spans:
        assert a == b or (a % chunk == 0 and (b % chunk == 0 or b == n))
    windows = [-(-(b - a) // chunk) for a, b in spans]
    assert max(windows) - min(windows) <= 1  # balanced to within one window


def test_rank_batches_are_distinct_per_step():
    for world in (1, 2, 4, 8):
        for step in range(5):
            got = [shard.rank_batch(step, r, world, 8) for r in range(world)]
            assert len(set(got)) == world


def test_parts_roundtrip_and_errors():
    parts = [b"abc", b"", b"x" * 100]
    blob = shard.pack_parts(parts)
    assert shard.unpack_parts(blob) == parts
    for bad in (blob[:-1], b"XXXX" + blob[4:], blob + b"\0", blob[:6]):
        with pytest.raises(ValueError):
            shard.unpack_parts(bad)
