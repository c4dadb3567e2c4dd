"""The two workloads the oracle cannot finish whole: the 72B-shaped cache at full
size (80 layers x 8 KV heads x 32,768 tokens) and the ragged batch of 8 requests
in one fused launch.

Full-size 72B: the planner is compared bit-exactly; the scores are checked by the
softmax-mass invariant (every window row's softmax sums to 1, so a KV head's
shared score vector sums to G*W) and, on sampled (layer, KV head) slices, against
the fp64 oracle's per-layer column sums; the compacted cache is checked against
the GPU's own scores by the selection's defining property (every kept token ranks
above every other token under (-score, index)), K_out bit-exactly, and sampled
kept rows of V_out against the oracle's fusion on the GPU's drop list.

Ragged batch: the one-launch batch result equals, bit for bit, the same requests
run one at a time, and the two smallest requests match the oracle in full.
Repeated launches of the batch are bit-identical.
"""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import plan as oplan
from oracle import prunekv as ok
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc
from tests.parity import TOL, check_request, np64

DEV = "cuda:0"
pytestmark = pytest.mark.gpu


def _rows_of(B, Hkv):
    """First output row of each (layer, KV head) block in the dense varlen layout."""
    out, P = {}, 0
    for l, b in enumerate(B):
        for g in range(Hkv):
            out[(l, g)] = Hkv * P + g * b
        P += b
    return out


def _drops_of(B, Nq, Hkv):
    out, Qd = {}, 0
    for l, b in enumerate(B):
        D = Nq - b if b > 0 else 0
        for g in range(Hkv):
            out[(l, g)] = (Hkv * Qd + g * D, D)
        Qd += D
    return out


def test_workload4_72b_full_size():
    wl = synth.WORKLOADS[4]
    req = wl.requests[0]
    L, Hq, Hkv, d, n, W = wl.L, wl.Hq, wl.Hkv, wl.d, req.n, req.W
    G = Hq // Hkv
    qs, ks, vs = synth.generate(wl, DEV)
    Q, K, V = qs[0], ks[0], vs[0]
    B, Nq, h = vc.viscache_plan_budgets(L, n, req.rr_num, req.rr_den)
    assert (B, Nq, h) == oplan.plan_budgets(L, n, Fraction(req.rr_num, req.rr_den))

    # the fused entry point, as timed by the benchmark
    batch = vc.Batch([n], [W], [(req.rr_num, req.rr_den)])
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q, K, V)
    s = vc.prunekv_score(Q, K)                                     # [Hkv][n]
    s_layer = vc.prunekv_score(Q, K, rank_mode=vc.VC_RANK_PER_LAYER)  # [L][Hkv][n]
    rank, keep, drop = vc.prunekv_select(s, B, Nq)
    torch.cuda.synchronize()
    assert Ko.shape[0] == Hkv * sum(B)
    assert torch.equal(keep, idx)

    # scores: softmax mass of every KV head, shared and per layer
    s64 = np64(s)
    mass = s64.sum(axis=1)
    assert np.allclose(mass, G * W, rtol=1e-5), mass
    sl64 = np64(s_layer)
    assert np.allclose(sl64.sum(axis=2), G * W, rtol=1e-5)
    assert np.allclose(sl64.mean(axis=0), s64, rtol=1e-4, atol=1e-6 * G * W / n)

    # scores: sampled slices against the oracle (per-layer column sums)
    for (l, g) in [(0, 0), (L // 2, 3), (L - 1, Hkv - 1)]:
        Qs = np64(Q[l:l + 1, g * G:(g + 1) * G])
        Ks = np64(K[l:l + 1, g:g + 1])
        ref = ok.token_scores(Qs, Ks, None, "shared", None)[0]
        got = sl64[l, g]
        err = np.abs(got - ref) / np.maximum(np.abs(ref), 1e-30)
        assert float(err.max()) <= 2e-5, "layer %d head %d: score rel err %.3g" % (l, g, err.max())

    # selection: every kept token ranks above every other under (-score, index)
    idx_np = idx.cpu().numpy().astype(np.int64)
    rows = _rows_of(B, Hkv)
    for g in range(Hkv):
        order = np.lexsort((np.arange(n), -s64[g]))
        for l in range(L):
            b = B[l]
            kg = idx_np[rows[(l, g)]:rows[(l, g)] + b]
            assert np.array_equal(kg, np.sort(order[:b])), "keep l=%d g=%d" % (l, g)

    # K_out bit-exact and sampled V_out rows against the oracle fusion
    drops = _drops_of(B, Nq, Hkv)
    drop_np = drop.cpu().numpy().astype(np.int64)
    rng = np.random.default_rng(4)
    tol = TOL[torch.bfloat16]
    for (l, g) in [(0, 1), (h // 2, 2), (h - 1, 5), (L - 1, 7)]:
        b = B[l]
        if b == 0:
            continue
        r0 = rows[(l, g)]
        kg = idx_np[r0:r0 + b]
        assert torch.equal(Ko[r0:r0 + b].cpu(), K[l, g][torch.from_numpy(kg).to(DEV)].cpu())
        d0, D = drops[(l, g)]
        dg = drop_np[d0:d0 + D]
        pick = np.sort(rng.choice(b, size=min(b, 48), replace=False))
        Vn = np64(V[l, g])
        ref = ok.fuse_values(Vn, kg[pick], dg, 0.7, 1.0)
        got = np64(Vo[r0:r0 + b])[pick]
        diff = np.abs(got - ref)
        rms = float(np.sqrt((ref ** 2).mean()))
        assert float(diff.max()) <= tol * float(np.abs(ref).max()), "V_out l=%d g=%d" % (l, g)
        assert not (diff > tol * np.abs(ref) + tol * rms).any(), "V_out l=%d g=%d" % (l, g)


def test_workload5_ragged_batch_one_launch():
    wl = synth.WORKLOADS[5]
    qs, ks, vs = synth.generate(wl, DEV)
    Q = torch.cat([q.flatten() for q in qs])
    K = torch.cat([k.flatten() for k in ks])
    V = torch.cat([v.flatten() for v in vs])
    batch = vc.Batch([r.n for r in wl.requests], [r.W for r in wl.requests],
                     [(r.rr_num, r.rr_den) for r in wl.requests])
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q, K, V)
    torch.cuda.synchronize()
    off = 0
    for i, r in enumerate(wl.requests):
        one = vc.Batch([r.n], [r.W], [(r.rr_num, r.rr_den)])
        ko, vo, ix = vc.prunekv_compress(one, prm, qs[i], ks[i], vs[i])
        torch.cuda.synchronize()
        rows = vc.compressed_rows(one, prm)
        assert torch.equal(idx[off:off + rows], ix), "request %d idx" % i
        assert torch.equal(Ko[off:off + rows], ko), "request %d K_out" % i
        assert torch.equal(Vo[off:off + rows], vo), "request %d V_out" % i
        off += rows
    assert off == vc.compressed_rows(batch, prm)

    # the two smallest requests against the oracle, through the step API
    small = sorted(range(len(wl.requests)), key=lambda i: wl.requests[i].n * wl.requests[i].W)[:2]
    off = [0]
    for r in wl.requests:
        off.append(off[-1] + vc.compressed_rows(vc.Batch([r.n], [r.W], [(r.rr_num, r.rr_den)]), prm))
    for i in small:
        r = wl.requests[i]
        B, Nq, h = vc.viscache_plan_budgets(wl.L, r.n, r.rr_num, r.rr_den)
        s = vc.prunekv_score(qs[i], ks[i])
        rank, keep, drop = vc.prunekv_select(s, B, Nq)
        ko, vo = vc.prunekv_fuse_compact(ks[i], vs[i], B, Nq, keep, drop, 0.7, 1.0)
        torch.cuda.synchronize()
        out = dict(scores=s, rank=rank, keep=keep, drop=drop, K_out=ko, V_out=vo)
        log = check_request(qs[i].cpu(), ks[i].cpu(), vs[i].cpu(), B, Nq, out, 0.7, 1.0)
        print("request %d (n=%d, W=%d) near-tie swaps: %s" % (i, r.n, r.W, log))
        assert torch.equal(idx[off[i]:off[i + 1]], keep)
        assert torch.equal(Vo[off[i]:off[i + 1]], vo)


def test_repeated_launches_bit_identical():
    """The fused pass is deterministic: repeated launches on the ragged batch
    (8 requests, every CTA pair of the fusion racing its neighbours on the SMs)
    give bit-identical caches.  A barrier or ordering bug between the MMA
    issuer, the softmax warps and the epilogue shows up here as a rare
    difference in a few rows."""
    wl = synth.WORKLOADS[5]
    qs, ks, vs = synth.generate(wl, DEV)
    Q = torch.cat([q.flatten() for q in qs])
    K = torch.cat([k.flatten() for k in ks])
    V = torch.cat([v.flatten() for v in vs])
    batch = vc.Batch([r.n for r in wl.requests], [r.W for r in wl.requests],
                     [(r.rr_num, r.rr_den) for r in wl.requests])
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    Ko0, Vo0, idx0 = vc.prunekv_compress(batch, prm, Q, K, V)
    for rep in range(24):
        Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q, K, V)
        torch.cuda.synchronize()
        assert torch.equal(idx, idx0), "launch %d idx" % rep
        assert torch.equal(Ko, Ko0), "launch %d K_out" % rep
        assert torch.equal(Vo, Vo0), "launch %d V_out" % rep
