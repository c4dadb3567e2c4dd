"""Oracle for PruneKV scoring, selection, key pruning and value fusion, in float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Inputs are numpy float64 arrays holding exactly the bf16/fp32 bits the GPU
reads (widened).  Shapes, per request:

    Qw [L][Hq][W][d]   observation-window queries (last W rows of prefill)
    K  [L][Hkv][n][d]  visual keys
    V  [L][Hkv][n][d]  visual values

GQA: query head j reads KV head j // G, G = Hq / Hkv.

Readings where the paper is silent or ambiguous:

* the query rows of Eq. (token_score) are the W window rows;
* the softmax of A^l runs over the n visual keys with scale 1/sqrt(d)
  (scaled dot-product attention, Sec. 3.2 "Asymmetric Key-Value Update"),
  unless a per-row log-sum-exp from prefill is supplied;
* one score vector per KV head, summed over the G query heads it serves;
* ties in the ranking go to the lower token index; kept and dropped tokens
  are listed in ascending position;
* the drop set of layer l is the survivors of the top-q step minus the keep
  set (Algorithm 1: "discard the rest" happens before the layer loop);
* Eq. (redistribution) normalises each row of Phi over the drop set; an empty
  drop set leaves V_k unchanged.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np


def _softmax_rows(x: np.ndarray) -> np.ndarray:
    m = x.max(axis=-1, keepdims=True)
    e = np.exp(x - m)
    return e / e.sum(axis=-1, keepdims=True)


def attention_weights(Qw_l: np.ndarray, K_l: np.ndarray, scale: float,
                      row_lse: Optional[np.ndarray] = None) -> np.ndarray:
    """A^l for one layer: [Hq][W][n] softmax(q.k * scale) over the visual keys.

    With ``row_lse`` ([Hq][W]), A = exp(q.k*scale - lse) instead (the
    normaliser a prefill attention kernel already computed).
    """
    Hq, W, d = Qw_l.shape
    Hkv = K_l.shape[0]
    G = Hq // Hkv
    out = np.empty((Hq, W, K_l.shape[1]))
    for j in range(Hq):
        x = (Qw_l[j] @ K_l[j // G].T) * scale
        out[j] = _softmax_rows(x) if row_lse is None else np.exp(x - row_lse[j][:, None])
    return out


def token_scores(Qw: np.ndarray, K: np.ndarray, scale: Optional[float] = None,
                 rank_mode: str = "shared", row_lse: Optional[np.ndarray] = None) -> np.ndarray:
    """Eq. (token_score) per KV head.

    shared    : s[g][v]    = (1/L) sum_l sum_{j in G(g)} sum_i A^l_{j,i,v}      -> [Hkv][n]
    per_layer : s[l][g][v] =       sum_{j in G(g)} sum_i A^l_{j,i,v}            -> [L][Hkv][n]
    (Sec. 4.4: shared global ranking vs. layer-specific ranking.)
    """
    L, Hq, W, d = Qw.shape
    _, Hkv, n, _ = K.shape
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    per_layer = np.zeros((L, Hkv, n))
    for l in range(L):
        A = attention_weights(Qw[l], K[l], scale, None if row_lse is None else row_lse[l])
        for g in range(Hkv):
            per_layer[l, g] = A[g * G:(g + 1) * G].sum(axis=(0, 1))
    if rank_mode == "per_layer":
        return per_layer
    return per_layer.sum(axis=0) / L


def ranking(s: np.ndarray) -> np.ndarray:
    """Token order for one score vector: descending score, lower index first on ties."""
    v = np.arange(s.shape[0])
    return np.lexsort((v, -s))


def select(s: np.ndarray, B: List[int], Nq: int, rank_mode: str = "shared"):
    """Keep/drop sets per (layer, KV head) (Algorithm 1 steps 1 and 3).

    survivors = first Nq of the ranking ("retain the q percent"); keep_l = first
    B_l; drop_l = survivors[B_l:Nq].  Lists are ascending token positions.
    Returns (keep, drop, rank) with keep[l][g], drop[l][g] int64 arrays and
    rank[g][v] (shared) or rank[l][g][v] (per_layer) the position in the order.
    """
    L = len(B)
    Hkv = s.shape[-2]
    keep = [[None] * Hkv for _ in range(L)]
    drop = [[None] * Hkv for _ in range(L)]
    rank = np.empty(s.shape, dtype=np.int64)
    for g in range(Hkv):
        for l in range(L):
            sv = s[l, g] if rank_mode == "per_layer" else s[g]
            order = ranking(sv)
            if rank_mode == "per_layer":
                rank[l, g, order] = np.arange(order.size)
            elif l == 0:
                rank[g, order] = np.arange(order.size)
            keep[l][g] = np.sort(order[:B[l]]) if B[l] > 0 else np.zeros(0, np.int64)
            drop[l][g] = np.sort(order[B[l]:Nq]) if B[l] > 0 else np.zeros(0, np.int64)
    return keep, drop, rank


def compact_keys(K_lg: np.ndarray, keep_lg: np.ndarray) -> np.ndarray:
    """K_new = key vectors of the keep set ("prune keys in C_d", Algorithm 1 step 3)."""
    return K_lg[keep_lg]


def fuse_values(V_lg: np.ndarray, keep_lg: np.ndarray, drop_lg: np.ndarray,
                mu: float, tau: float) -> np.ndarray:
    """V_new = mu V_k + (1-mu) Phi V_d, Phi = row-softmax(V_k V_d^T / tau).

    Eq. (redistribution) and Eq. (weight_fusion).  float64, unrounded.
    """
    Vk = V_lg[keep_lg]
    if drop_lg.size == 0:
        return Vk.copy()
    Vd = V_lg[drop_lg]
    Phi = _softmax_rows((Vk @ Vd.T) / tau)
    return mu * Vk + (1.0 - mu) * (Phi @ Vd)


def prunekv(Qw: np.ndarray, K: np.ndarray, V: np.ndarray, B: List[int], Nq: int,
            mu: float = 0.7, tau: float = 1.0, scale: Optional[float] = None,
            rank_mode: str = "shared", row_lse: Optional[np.ndarray] = None,
            fuse: bool = True) -> Dict[str, object]:
    """Algorithm 1 for one request.

    Output layout (dense varlen): layer l (0-based, B_l > 0) is a [Hkv][B_l][d]
    block at row offset Hkv * P_l, P_l = sum_{j<l} B_j; idx holds the kept
    positions in the same layout.  Returns a dict with the scores, ranks,
    keep/drop lists and the packed K_out / V_out (float64) / idx_out.
    """
    L, Hkv, n, d = K.shape
    s = token_scores(Qw, K, scale, rank_mode, row_lse)
    keep, drop, rank = select(s, B, Nq, rank_mode)
    tot = sum(B)
    K_out = np.zeros((Hkv * tot, d))
    V_out = np.zeros((Hkv * tot, d))
    idx_out = np.zeros(Hkv * tot, dtype=np.int64)
    P = 0
    for l in range(L):
        b = B[l]
        for g in range(Hkv):
            r0 = Hkv * P + g * b
            idx_out[r0:r0 + b] = keep[l][g]
            K_out[r0:r0 + b] = compact_keys(K[l, g], keep[l][g])
            if fuse:
                V_out[r0:r0 + b] = fuse_values(V[l, g], keep[l][g], drop[l][g], mu, tau)
        P += b
    return dict(scores=s, rank=rank, keep=keep, drop=drop, K_out=K_out, V_out=V_out,
                idx_out=idx_out)
