"""Multi-rank aggregation of bench.py on the CPU (gloo, world size 2).

The path runs replicas only: each rank executes the whole step on its own
GPU, with no collective on the data path.  The one collective is the
reduction of the step time in bench.py, which must take the slowest rank's
time and report the work of all ranks over it.  These tests drive that code
with two gloo processes on 127.0.0.1.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, step_ms, flops, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        assert (r, w, local) == (rank, world, rank)
        q.put((rank, bench.job_throughput(step_ms[rank], flops, world, dist, "cpu")))
    finally:
        dist.destroy_process_group()


def _run(world, step_ms, flops):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, step_ms, flops, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0, f"rank process exited with {p.exitcode}"
    out = {}
    while not q.empty():
        r, v = q.get()
        out[r] = v
    return out


def test_two_ranks_take_the_slowest_step_and_sum_the_work():
    flops = 3_000_000_000
    out = _run(2, [2.0, 5.0], flops)
    assert set(out) == {0, 1}
    for r in (0, 1):
        ms, gflops = out[r]
        assert ms == 5.0                                   # max over ranks, on every rank
        assert gflops == pytest.approx(2 * flops / 5e-3 / 1e9)  # both ranks' work over that time


def test_single_process_is_plain_throughput():
    ms, gflops = bench.job_throughput(4.0, 8_000_000_000, 1)
    assert ms == 4.0 and gflops == pytest.approx(2000.0)
