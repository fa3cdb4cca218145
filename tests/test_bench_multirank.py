"""The benchmark's multi-rank aggregation on CPU: two gloo ranks (127.0.0.1) with different
timings must both see the slowest rank's time, and the whole-job throughput must count every
rank's units over that time.  (On the GPU machine each rank is an independent replica of the workload;
there is no collective on the data path, only this timing reduction.)"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    w, r, _ = bench._dist()
    secs = [2.0, 3.5][rank]
    slowest = bench.max_over_ranks(secs, w)
    value = bench.whole_job_throughput(1000.0, secs, w)
    dist.barrier()
    dist.destroy_process_group()
    q.put((r, slowest, value))


def test_two_gloo_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs)
    got = sorted(q.get(timeout=5) for _ in range(2))
    for r, slowest, value in got:
        assert slowest == 3.5
        assert value == pytest.approx(2 * 1000.0 / 3.5)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(1.25, 1) == 1.25
    assert bench.whole_job_throughput(100.0, 0.5, 1) == 200.0
