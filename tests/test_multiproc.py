"""Multi-process host logic of the bench on CPU (gloo, world size 2).

The transition only shards across independent transitions (replicas, no
exchange step); what the ranks share is the timing: a barrier on both sides
of the timed region and the slowest rank's time.  This runs that logic with
two gloo ranks on the CPU, including a rank that is slower than the other.
"""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, times, out_q):
    import time
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    os.environ["AVITS_BENCH_BACKEND"] = "gloo"
    w, r, local, pg = bench.dist_setup(world)
    assert (w, r) == (world, rank)
    bench.barrier(pg)
    t0 = time.perf_counter()
    time.sleep(times[rank])
    bench.barrier(pg)
    mine = time.perf_counter() - t0
    slowest = bench.max_over_ranks(pg, mine)
    value = bench.aggregate(100, w, slowest)
    out_q.put((rank, mine, slowest, value))
    pg.destroy_process_group()


def test_two_rank_timing_takes_the_slowest_rank():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    times = [0.05, 0.25]
    procs = [ctx.Process(target=_worker, args=(r, 2, port, times, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    slowest = [r[2] for r in res]
    assert abs(slowest[0] - slowest[1]) < 1e-12          # every rank agrees on the job time
    assert slowest[0] >= 0.25                              # barrier: the slow rank sets it
    assert abs(res[0][3] - 2 * 100 / slowest[0]) < 1e-6    # whole-job units / job time


def test_aggregate_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate(10, 1, 0.5) == 20.0
    assert bench.max_over_ranks(None, 3.0) == 3.0
