"""N > 1 host logic on CPU with gloo, world size 2: disjoint shards of
independent slabs, no data-path exchange, and the max-over-ranks timing."""
import os
import socket

import pytest

from paper_2506_15745_gb300.shard import max_over_ranks, shard_range, sum_over_ranks


def test_shard_range_partitions():
    for n in (0, 1, 7, 112, 5120):
        for world in (1, 2, 3, 8):
            ranges = [shard_range(n, r, world) for r in range(world)]
            assert ranges[0][0] == 0 and ranges[-1][1] == n
            for (a, b), (c, d) in zip(ranges, ranges[1:]):
                assert b == c
            sizes = [b - a for a, b in ranges]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        shard_range(4, 2, 2)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        begin, end = shard_range(8, rank, world)        # e.g. 8 streams over the ranks
        t = max_over_ranks(1.5 + rank)                   # per-rank pass time
        units = sum_over_ranks(end - begin)
        out.put((rank, begin, end, t, units))
    finally:
        dist.destroy_process_group()


def test_gloo_two_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [(r[1], r[2]) for r in res] == [(0, 4), (4, 8)]
    assert all(r[3] == 2.5 for r in res)
    assert all(r[4] == 8 for r in res)
