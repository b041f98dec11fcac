"""The multi-GPU path of the benchmark runs independent replicas of the stage (the method shards
by layer range with no collective; a single job here runs on one GPU): the only cross-rank step
is the maximum of the replicas' step times.  Checked with two gloo ranks on the CPU."""
import multiprocessing as mp
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each replica reports its own time; the job's time is the slowest
        got = bench.max_over_ranks(1.5 + rank, dist, "cpu")
        dist.barrier()
        q.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_replica_time_is_the_max_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
    assert all(p.exitcode == 0 for p in procs)
    res = dict(q.get(timeout=5) for _ in procs)
    assert res == {0: 2.5, 1: 2.5}


def test_single_process_has_no_reduction():
    import bench
    assert bench.max_over_ranks(3.25, None, "cpu") == 3.25
