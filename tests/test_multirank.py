"""N > 1 host logic of bench.py with world_size-2 gloo ranks on CPU.

The path needs no exchange between GPUs (replicas): the only cross-rank work
is the timing reduction (max over ranks) and the whole-job throughput.
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
