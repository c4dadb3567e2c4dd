"""The multi-GPU host path of bench.py on CPU: two gloo ranks (world size 2).

Under weak scaling each rank compresses its own requests (same shapes and mix,
its own seed), the timed region is the slowest rank's, and the job value is the
units of all ranks over that time.  No data-path collective exists; the only
exchange is the max of the timings.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2608_24063_gb300 import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = bench.rank_workload(synth.scaled(synth.WORKLOADS[3], "tiny", L=2, Hq=4, Hkv=2, d=64,
                                               requests=[synth.Request(96, 8, 19, 100, 32)]), rank)
        # each rank's own request: same shapes, different values
        q = synth.make_q(wl, 0, "cpu")
        digest = float(q.double().abs().sum())
        sums = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(sums, torch.tensor([digest], dtype=torch.float64))
        # the timed region: the slowest rank's duration
        ms = bench.max_over_ranks(10.0 + 5.0 * rank, world, dist, "cpu")
        out[rank] = (tuple(q.shape), [float(x) for x in sums], ms,
                     bench.job_value(1000, world, ms))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_weak_scaling():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True,
                       start_method="spawn")
    r0, r1 = out[0], out[1]
    assert r0[0] == r1[0]                       # same request shapes on every rank
    assert r0[1] == r1[1] and r0[1][0] != r0[1][1]   # but each rank its own values
    assert r0[2] == r1[2] == 15.0               # max over ranks
    assert r0[3] == r1[3] == pytest.approx(2 * 1000 / 15e-3)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(3.5, 1, None, "cpu") == 3.5
    assert bench.job_value(50, 1, 2.0) == pytest.approx(25000.0)
    wl = synth.WORKLOADS[2]
    assert bench.rank_workload(wl, 0) is wl
    assert bench.rank_workload(wl, 3).seed != wl.seed
