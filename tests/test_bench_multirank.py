"""The multi-GPU host path on CPU: two gloo ranks (world size 2), and the partitions.

Under weak scaling the job is N copies of the workload's requests (each copy its
own seeded values), split over the ranks by the work-balanced request partition
that ``bench.py --gpus N`` uses (``bench.rank_requests`` ->
``shard.partition_requests``); each rank compresses its share with no data-path
collective, the timed region is the slowest rank's, and the job value is the
units of all ranks over that time.

Here each rank runs the fp64 oracle on its share (the CPU stand-in for its GPU)
and rank 0 reassembles the shares with ``shard.merge_requests``: the result must
equal the oracle on the unsharded job, request by request.  The KV-head split
(``shard.kv_head_ranges`` / ``merge_kv_heads``) is checked the same way on one
request.
"""
import os
import socket
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from oracle import plan as oplan
from oracle import prunekv as ok
from paper_2608_24063_gb300 import shard, synth

TINY = synth.scaled(synth.WORKLOADS[5], "tiny ragged batch", L=2, Hq=4, Hkv=2, d=32,
                    requests=[synth.Request(96, 8, 19, 100, 32), synth.Request(150, 5, 28, 100, 32),
                              synth.Request(64, 12, 23, 100, 32)])


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _oracle_request(wl, r):
    """The oracle's compressed cache of request r of wl: (idx, K_out, V_out) rows."""
    q = synth.make_q(wl, r)
    k, v = synth.make_kv(wl, r, q)
    req = wl.requests[r]
    B, Nq, _ = oplan.plan_budgets(wl.L, req.n, Fraction(req.rr_num, req.rr_den))
    out = ok.prunekv(q.double().numpy(), k.double().numpy(), v.double().numpy(), B, Nq)
    return out["idx_out"], out["K_out"], out["V_out"]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.set_num_threads(1)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        job, mine, view = bench.rank_requests(TINY, world, rank)
        assert [job.requests[i] for i in mine] == list(view.requests)
        res = [_oracle_request(job, i) for i in mine]
        rows = [len(x[0]) for x in res]
        cat = lambda j: np.concatenate([x[j] for x in res]) if res else np.zeros(0)
        share = (mine, rows, (cat(0), cat(1), cat(2)))
        gathered = [None] * world
        dist.all_gather_object(gathered, share)
        ms = bench.max_over_ranks(10.0 + 5.0 * rank, world, dist, "cpu")
        out[rank] = (gathered, ms, len(job.requests),
                     bench.job_value(sum(r.n * TINY.L for r in job.requests), ms))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_request_partition_equals_unsharded():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True,
                       start_method="spawn")
    g0, ms0, njob, val0 = out[0]
    g1, ms1, _, _ = out[1]
    assert ms0 == ms1 == 15.0                                   # max over ranks
    assert njob == world * len(TINY.requests)
    assert val0 == pytest.approx(sum(r.n * TINY.L for r in TINY.requests) * world / 15e-3)
    # the shares cover the job once; rank 0 reassembles them in request order
    assert sorted(i for m, _, _ in g0 for i in m) == list(range(njob))
    job = synth.replicated(TINY, world)
    for j in range(3):
        parts = [(m, rows, o[j]) for m, rows, o in g0]
        blocks = shard.merge_requests(parts, njob)
        for r in range(njob):
            assert np.array_equal(blocks[r], _oracle_request(job, r)[j]), "request %d part %d" % (r, j)
    # the copies differ in values, not in shapes
    a, b = _oracle_request(job, 0), _oracle_request(job, len(TINY.requests))
    assert a[1].shape == b[1].shape and not np.array_equal(a[1], b[1])


def test_partition_requests_properties():
    costs = [shard.request_cost(r.n, r.W, 28, 28) for r in synth.WORKLOADS[5].requests] * 3
    for world in (1, 2, 3, 4, 8, 30):
        parts = shard.partition_requests(costs, world)
        assert len(parts) == world
        assert sorted(i for p in parts for i in p) == list(range(len(costs)))
        assert all(p == sorted(p) for p in parts)
        loads = [sum(costs[i] for i in p) for p in parts]
        assert max(loads) - min(loads) <= max(costs)            # greedy bound
        assert parts == shard.partition_requests(costs, world)   # deterministic
    assert shard.partition_requests([5, 5, 5, 5], 2) == [[0, 2], [1, 3]]
    with pytest.raises(ValueError):
        shard.partition_requests([1], 0)
    with pytest.raises(ValueError):
        shard.merge_requests([([0], [1], [7]), ([0], [1], [8])], 1)


def test_bench_rank_requests_single_rank_is_the_workload():
    wl = synth.WORKLOADS[5]
    job, mine, view = bench.rank_requests(wl, 1, 0)
    assert mine == list(range(len(wl.requests)))
    assert tuple(view.requests) == tuple(wl.requests) and view.seed == wl.seed
    assert bench.max_over_ranks(3.5, 1, None, "cpu") == 3.5
    assert bench.job_value(50, 2.0) == pytest.approx(25000.0)


def test_kv_head_split_equals_unsharded():
    wl = TINY
    r = 1
    q = synth.make_q(wl, r)
    k, v = synth.make_kv(wl, r, q)
    req = wl.requests[r]
    B, Nq, _ = oplan.plan_budgets(wl.L, req.n, Fraction(req.rr_num, req.rr_den))
    Q, K, V = q.double().numpy(), k.double().numpy(), v.double().numpy()
    full = ok.prunekv(Q, K, V, B, Nq)
    G = wl.Hq // wl.Hkv
    for world in (1, 2):
        ranges = shard.kv_head_ranges(wl.Hkv, world)
        assert ranges[0][0] == 0 and ranges[-1][1] == wl.Hkv
        parts = [ok.prunekv(Q[:, g0 * G:g1 * G], K[:, g0:g1], V[:, g0:g1], B, Nq) for g0, g1 in ranges]
        for key in ("idx_out", "K_out", "V_out"):
            got = np.concatenate(shard.merge_kv_heads([p[key] for p in parts], B, ranges))
            assert np.array_equal(got, full[key]), (world, key)
    assert shard.kv_head_ranges(8, 3) == [(0, 3), (3, 6), (6, 8)]
    with pytest.raises(ValueError):
        shard.kv_head_ranges(2, 3)
