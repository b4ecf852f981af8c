"""Multi-rank host logic of bench.py on CPU (gloo, world size 2): each rank
draws its own batch, the timed region's duration is the slowest rank's, and
the reported value is every rank's steps over that time.  No GPU involved;
the benchmark's ranks exchange nothing else (requests are independent)."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 100.0 + 50.0 * rank          # rank 1 is the slow one
        dist.barrier()
        t = bench.slowest(local_ms, dist, "cpu")
        q.put((rank, bench.rank_seed(7, rank), t, bench.job_rate(20, world, t / 1e3)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_time_and_aggregate():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(world))
    assert res[0][1] != res[1][1]                       # independent batches per rank
    assert [r[2] for r in res] == [150.0, 150.0]        # max over ranks, seen by both
    assert res[0][3] == pytest.approx(2 * 20 / 0.150)   # whole-job steps/s


def test_single_process_has_no_collective():
    assert bench.slowest(12.5, None, "cpu") == 12.5
    assert bench.job_rate(10, 1, 0.5) == 20.0
    assert bench.rank_seed(3, 0) == 3
