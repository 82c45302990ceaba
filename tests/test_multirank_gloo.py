"""Multi-rank path of bench.py on CPU: two gloo ranks (replicas) meet at the
barrier, agree on the slowest rank's time, and the whole-job rate counts the
work of every rank."""

import multiprocessing as mp
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch
    import torch.distributed as dist

    import bench
    r, w, _ = bench.init_dist(None)
    assert dist.get_backend() == "gloo"
    bench.barrier(w)
    ms_local = 100.0 + 50.0 * r  # rank 1 is the slow one
    ms_max = bench.max_over_ranks(ms_local, w, torch.device("cpu"))
    rate = bench.replica_throughput(1000.0, ms_max, w)
    out.put((r, ms_max, rate))
    dist.destroy_process_group()


def test_two_gloo_replicas_agree_on_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs)
    res = sorted(q.get(timeout=5) for _ in range(2))
    for r, ms_max, rate in res:
        assert ms_max == 150.0
        assert rate == pytest.approx(2 * 1000.0 / 0.150)


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5, 1, None) == 3.5
    assert bench.replica_throughput(10.0, 1000.0, 1) == pytest.approx(10.0)
