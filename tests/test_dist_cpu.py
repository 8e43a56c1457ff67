"""The multi-rank host logic of bench.py on two CPU ranks (gloo): the map has no exchange
step, so N GPUs run N replicas; what crosses ranks is the barrier around the timed region
and a MAX all-reduce of the elapsed time, from which rank 0 reports the whole-job rate.
The reference arm (the oracle) runs on rank 0 alone; the other ranks exit without work."""
import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(dist)
        ms = 100.0 + 37.5 * rank                     # a slower rank sets the job's time
        m = bench.max_over_ranks(ms, dist, torch.device("cpu"))
        rate = bench.job_rate(world, 32768, 10, m)
        # the reference arm returns before any work on ranks other than 0
        ref = bench.reference_arm(None, None, None) if rank != 0 else 0
        out.put((rank, m, rate, ref))
        bench.barrier(dist)
    finally:
        dist.destroy_process_group()


def test_two_rank_timing_and_rate():
    world = 2
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=240)
    alive = [p for p in procs if p.is_alive()]
    for p in alive:
        p.kill()
    assert not alive, "a rank did not finish"
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    res = sorted(out.get(timeout=10) for _ in range(world))
    slowest = 100.0 + 37.5 * (world - 1)
    for rank, m, rate, ref in res:
        assert m == slowest                         # every rank sees the slowest rank's time
        assert rate == pytest.approx(world * 32768 * 10 / (slowest / 1e3), rel=1e-12)
        assert ref == 0


def test_job_rate_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_rate(1, 32768, 300, 1000.0) == pytest.approx(32768 * 300)
    assert bench.job_rate(4, 1000, 2, 500.0) == pytest.approx(4 * 1000 * 2 / 0.5)
