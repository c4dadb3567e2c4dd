"""Parity rules between the CUDA path and the fp64 oracle (used by the -m gpu tests).

* budgets and Nq: bit-exact;
* kept / dropped index sets: bit-exact, except swaps across a cut whose oracle
  scores differ by less than 1e-6 relative (logged, not failed);
* K_out: bit-exact copy of the rows the GPU kept;
* V_out: against the oracle's fusion run on the GPU's own keep/drop lists;
  bf16: max|d| <= 2e-2 max|ref| per (layer, head) and |d| <= 2e-2 |ref| + 2e-2 rms(ref)
  elementwise; fp32: the same forms with 1e-5.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import prunekv as ok

NEAR_TIE = 1e-6
TOL = {torch.bfloat16: 2e-2, torch.float32: 1e-5}


def np64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float64).numpy()


def check_v_rows(got, ref, tol, tag):
    """V_out rows of one (layer, KV head) against the oracle's fusion (both float64):
    max|d| <= tol max|ref| and |d| <= tol |ref| + tol rms(ref) elementwise."""
    diff = np.abs(got - ref)
    amax = float(np.abs(ref).max()) if ref.size else 0.0
    rms = float(np.sqrt((ref ** 2).mean())) if ref.size else 0.0
    assert float(diff.max(initial=0)) <= tol * amax + 1e-30, "V_out max %s: %g" % (tag, diff.max(initial=0))
    bad = diff > tol * np.abs(ref) + tol * rms
    assert not bad.any(), "V_out elementwise %s: %d bad" % (tag, int(bad.sum()))


def check_sets(gpu_keep, ref_rank, s_ref, cut, log, tag):
    """gpu_keep: the GPU's top-`cut` set (ascending ints); ref_rank: oracle rank per token."""
    ref_keep = np.sort(np.argsort(ref_rank, kind="stable")[:cut])
    g = np.asarray(gpu_keep, dtype=np.int64)
    if g.size != cut:
        raise AssertionError("%s: size %d != %d" % (tag, g.size, cut))
    if np.array_equal(g, ref_keep):
        return 0
    extra = np.setdiff1d(g, ref_keep)
    missing = np.setdiff1d(ref_keep, g)
    order = np.argsort(ref_rank, kind="stable")
    edge = [s_ref[order[cut - 1]]] + ([s_ref[order[cut]]] if cut < len(order) else [])
    ref_cut = max(edge)
    for t in np.concatenate([extra, missing]):
        if abs(s_ref[t] - ref_cut) > NEAR_TIE * max(s_ref[t], ref_cut):
            raise AssertionError("%s: token %d (score %.9g) swapped across cut %.9g" %
                                 (tag, t, s_ref[t], ref_cut))
    log.append((tag, extra.tolist(), missing.tolist()))
    return len(extra)


def check_request(Qw, K, V, B, Nq, gpu, mu, tau, rank_mode="shared", scale=None, row_lse=None,
                  score_rtol=2e-5, check_v=True):
    """Compare one request's GPU outputs (dict of torch tensors) with the oracle.

    gpu: scores [Hkv][n] or [L][Hkv][n] (optional), keep (flat, D8 layout),
         drop (flat), K_out, V_out.
    Returns the near-tie log.
    """
    Qn, Kn, Vn = np64(Qw), np64(K), np64(V)
    L, Hkv, n, d = Kn.shape
    s_ref = ok.token_scores(Qn, Kn, scale, rank_mode, row_lse)
    log = []
    if gpu.get("scores") is not None:
        sg = np64(gpu["scores"]).reshape(s_ref.shape)
        err = np.abs(sg - s_ref) / np.maximum(np.abs(s_ref), 1e-30)
        assert float(err.max()) <= score_rtol, "score rel err %.3g" % float(err.max())
    keep = gpu["keep"].cpu().numpy().astype(np.int64)
    drop = gpu["drop"].cpu().numpy().astype(np.int64)
    Kg = gpu["K_out"].cpu()
    Vg = np64(gpu["V_out"])
    tol = TOL[V.dtype]
    P = Qd = 0
    for l in range(L):
        b = B[l]
        D = Nq - b if b > 0 else 0
        for g in range(Hkv):
            sv = s_ref[l, g] if rank_mode == "per_layer" else s_ref[g]
            rank = np.empty(n, np.int64)
            rank[ok.ranking(sv)] = np.arange(n)
            r0 = Hkv * P + g * b
            kg = keep[r0:r0 + b]
            dg = drop[Hkv * Qd + g * D: Hkv * Qd + g * D + D]
            assert np.all(np.diff(kg) > 0) and np.all(np.diff(dg) > 0), "not ascending/unique"
            assert not set(kg.tolist()) & set(dg.tolist())
            if b == 0:
                continue
            check_sets(kg, rank, sv, b, log, "keep l=%d g=%d" % (l, g))
            check_sets(np.union1d(kg, dg), rank, sv, Nq, log, "survivors l=%d g=%d" % (l, g))
            # K_out: bit-exact rows
            assert torch.equal(Kg[r0:r0 + b], K[l, g].cpu()[torch.from_numpy(kg)]), "K_out l=%d g=%d" % (l, g)
            if check_v:
                ref = ok.fuse_values(Vn[l, g], kg, dg, mu, tau)
                check_v_rows(Vg[r0:r0 + b], ref, tol, "l=%d g=%d" % (l, g))
        P += b
        Qd += D
    return log
