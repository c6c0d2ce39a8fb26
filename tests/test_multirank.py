"""N > 1 host logic of bench.py with world_size-2 gloo ranks on CPU.

The path needs no exchange between GPUs: the headline workload runs as
replicas, and the per-request workload splits its requests (each rank builds,
compiles and decodes its own share). The only cross-rank work is the timing
reduction (max over ranks) and the whole-job throughput.
"""
from __future__ import annotations

import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank(rank: int, world: int, port: int, out):
    import torch.distributed as dist
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    local_ms = [12.5, 20.0][rank]
    m = bench.reduce_max(local_ms, dist, "cpu")
    v = bench.job_throughput(1000.0, world, m * 1e-3)
    dist.barrier()
    out.put((rank, m, v))
    dist.destroy_process_group()


def test_two_rank_timing_reduction():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, m, v in res:
        assert m == pytest.approx(20.0)
        assert v == pytest.approx(2 * 1000.0 / 0.020)


def test_single_rank_helpers():
    import bench
    assert bench.reduce_max(3.0, None, "cpu") == 3.0
    assert bench.job_throughput(10.0, 1, 2.0) == 5.0


def _share_rank(rank: int, world: int, port: int, out):
    import torch.distributed as dist
    import bench
    from paper_2608_12574_gb300 import workloads as W
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    full = W.dynamic_requests(12)
    lo, hi = bench.request_share(full.batch, rank, world)
    mine = bench.share_of(full, lo, hi)
    strings = W.unpack(mine.set_bytes, mine.set_offsets)
    sets = {lo + i: strings[mine.set_index[i]:mine.set_index[i + 1]] for i in range(hi - lo)}
    got = [None] * world
    dist.all_gather_object(got, sets)
    dist.barrier()
    out.put((rank, got))
    dist.destroy_process_group()


def test_two_rank_request_partition():
    """The per-request workload split over two gloo ranks: every request is
    on exactly one rank, with exactly its own strings."""
    from paper_2608_12574_gb300 import workloads as W
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_share_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=300) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    full = W.dynamic_requests(12)
    strings = W.unpack(full.set_bytes, full.set_offsets)
    for _, got in res:
        ids = [i for part in got for i in part]
        assert sorted(ids) == list(range(12))
        for part in got:
            for i, st in part.items():
                assert st == strings[full.set_index[i]:full.set_index[i + 1]]


def test_request_share_covers_every_request():
    import bench
    for n in (1, 7, 256):
        for world in (1, 2, 3, 8):
            parts = [bench.request_share(n, r, world) for r in range(world)]
            assert parts[0][0] == 0 and parts[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(parts, parts[1:]))
            sizes = [hi - lo for lo, hi in parts]
            assert max(sizes) - min(sizes) <= 1
