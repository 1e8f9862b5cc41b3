"""The bench's multi-rank host logic on two gloo ranks (CPU).

The module shards by (batch, head) with no exchange, so N GPUs run N replica
layers; the only collectives are the bench's barrier and the max of the step
times.  Two CPU processes check that every rank agrees on the slowest rank's
time and on the whole-job throughput.
"""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    my_ms = [18.0, 19.5][rank]                 # rank 1 is the slower replica
    bench.barrier(world)
    worst = bench.reduce_max(my_ms, world)
    value = bench.job_throughput(75600, worst, world)
    out.put((rank, worst, value))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_agree_on_slowest_time_and_job_throughput():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    results = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in results] == [19.5, 19.5]
    assert results[0][2] == pytest.approx(2 * 75600 / 19.5e-3)
    assert results[0][2] == results[1][2]


def test_single_rank_is_the_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(3.5, 1) == 3.5
    assert bench.job_throughput(100, 10.0, 1) == pytest.approx(1e4)
