"""The collective-free splits on one GPU: each share is compressed with the ordinary
single-GPU call, one after the other, and the shares' outputs, put back together
with ``shard.merge_requests`` / ``shard.merge_kv_heads``, equal the unsharded
call bit for bit.

* by request: the ragged batch of 8 (7B shape) split over two ranks by the
  work-balanced partition that ``bench.py --gpus N`` uses;
* by KV head: the 7B shape at 12,544 tokens split into two halves of 2 KV heads
  (and the 14 query heads that read them), as two tensor-parallel GPUs would
  hold them.
"""
import pytest
import torch

from paper_2608_24063_gb300 import shard, synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _batch(reqs):
    return vc.Batch([r.n for r in reqs], [r.W for r in reqs], [(r.rr_num, r.rr_den) for r in reqs])


def _flat(ts):
    return torch.cat([t.flatten() for t in ts])


def test_request_partition_equals_one_launch():
    wl = synth.WORKLOADS[5]
    qs, ks, vs = synth.generate(wl, DEV)
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    full = vc.prunekv_compress(_batch(wl.requests), prm, _flat(qs), _flat(ks), _flat(vs))
    costs = [shard.request_cost(r.n, r.W, wl.L, wl.Hq) for r in wl.requests]
    parts = shard.partition_requests(costs, 2)
    assert all(parts)
    outs = []
    for mine in parts:
        reqs = [wl.requests[i] for i in mine]
        o = vc.prunekv_compress(_batch(reqs), prm, _flat([qs[i] for i in mine]), _flat([ks[i] for i in mine]),
                                _flat([vs[i] for i in mine]))
        rows = [vc.compressed_rows(_batch([r]), prm) for r in reqs]
        outs.append((mine, rows, o))
    torch.cuda.synchronize()
    for j in range(3):
        blocks = shard.merge_requests([(m, rows, o[j]) for m, rows, o in outs], len(wl.requests))
        assert torch.equal(torch.cat(blocks), full[j]), "output %d" % j


def test_kv_head_halves_equal_unsharded():
    wl = synth.WORKLOADS[3]
    req = wl.requests[0]
    qs, ks, vs = synth.generate(wl, DEV)
    Q, K, V = qs[0], ks[0], vs[0]
    batch = _batch([req])
    full = vc.prunekv_compress(batch, vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16), Q, K, V)
    B, _, _ = vc.viscache_plan_budgets(wl.L, req.n, req.rr_num, req.rr_den)
    ranges = shard.kv_head_ranges(wl.Hkv, 2)
    G = wl.G
    outs = []
    for g0, g1 in ranges:
        prm = vc.make_params(wl.L, (g1 - g0) * G, g1 - g0, wl.d, vc.VC_BF16)
        outs.append(vc.prunekv_compress(batch, prm, Q[:, g0 * G:g1 * G].contiguous(), K[:, g0:g1].contiguous(),
                                        V[:, g0:g1].contiguous()))
    torch.cuda.synchronize()
    for j in range(3):
        got = torch.cat(shard.merge_kv_heads([o[j] for o in outs], B, ranges))
        assert torch.equal(got, full[j]), "output %d" % j
