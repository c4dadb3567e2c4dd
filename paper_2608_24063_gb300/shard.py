"""Collective-free partitions of the compression pass across GPUs (host bookkeeping only).

The pass has no exchange step when it is split by request or by KV head: the
token scores, the ranking, the budgets and the fusion of Eq. (token_score) to
Eq. (weight_fusion) are all per (request, KV head), and a request's budgets do
not depend on its heads.  Each GPU therefore compresses its own share with the
ordinary single-GPU call, and the shares' outputs are plain slices of the
unsharded output:

* by request: rank r gets a subset of the batch's requests
  (``partition_requests``); its dense varlen output is the concatenation of its
  requests' outputs, and ``merge_requests`` puts the ranks' rows back into the
  batch order;
* by KV head: rank r gets a contiguous range of KV heads and the query heads
  that read them (``kv_head_ranges``; with G = Hq / Hkv, KV heads [g0, g1) and
  query heads [g0 G, g1 G)); layer l of the unsharded output is the ranks'
  [g1 - g0][B_l][d] blocks one after the other (``merge_kv_heads``).

Nothing here touches a device or computes any part of the method.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple


def request_cost(n: int, W: int, L: int, Hq: int) -> int:
    """Relative cost of one request: its logits (L * Hq * W * n), which dominate the
    score passes; the fusion and copies scale with n as well."""
    return L * Hq * W * n


def partition_requests(costs: Sequence[int], world: int) -> List[List[int]]:
    """Split requests over `world` ranks, balancing the summed cost.

    Longest-first greedy: requests in order of decreasing cost (ties: lower
    index first) each go to the rank with the smallest total so far (ties:
    lower rank).  Every request lands on exactly one rank; each rank's list is
    ascending.  A rank may get no request when world > len(costs).
    """
    if world < 1:
        raise ValueError("world must be >= 1")
    order = sorted(range(len(costs)), key=lambda i: (-costs[i], i))
    load = [0] * world
    out: List[List[int]] = [[] for _ in range(world)]
    for i in order:
        r = min(range(world), key=lambda k: (load[k], k))
        out[r].append(i)
        load[r] += costs[i]
    return [sorted(x) for x in out]


def merge_requests(parts: Sequence[Tuple[Sequence[int], Sequence[int], object]], n_req: int) -> list:
    """Reassemble per-rank outputs in batch order.

    parts: per rank, (its request indices, the row count of each of its
    requests, its output rows -- anything sliceable along the first axis, the
    requests' rows one after the other).  Returns the list of per-request row
    blocks in request order 0..n_req-1.
    """
    blocks = [None] * n_req
    for idx, rows, out in parts:
        off = 0
        for i, nr in zip(idx, rows):
            if blocks[i] is not None:
                raise ValueError("request %d assigned twice" % i)
            blocks[i] = out[off:off + nr]
            off += nr
    missing = [i for i, b in enumerate(blocks) if b is None]
    if missing:
        raise ValueError("requests without a rank: %s" % missing)
    return blocks


def kv_head_ranges(Hkv: int, world: int) -> List[Tuple[int, int]]:
    """Contiguous KV-head ranges [g0, g1) for `world` ranks, sizes differing by at most
    one (the larger first).  Requires world <= Hkv."""
    if world < 1 or world > Hkv:
        raise ValueError("need 1 <= world <= Hkv")
    base, extra = divmod(Hkv, world)
    out, g = [], 0
    for r in range(world):
        k = base + (1 if r < extra else 0)
        out.append((g, g + k))
        g += k
    return out


def merge_kv_heads(parts: Sequence[object], B: Sequence[int], ranges: Sequence[Tuple[int, int]]) -> list:
    """Rows of the unsharded dense varlen output (one request) from per-rank outputs.

    parts[r] holds rank r's output rows for its heads [g0, g1): layer l is a
    [(g1 - g0)][B_l] row block at row (g1 - g0) * P_l.  Returns the list of row
    blocks in the unsharded order (layer by layer, each layer's heads in order),
    to be concatenated by the caller.
    """
    blocks = []
    P = 0
    for b in B:
        for (g0, g1), out in zip(ranges, parts):
            h = g1 - g0
            blocks.append(out[h * P:h * (P + b)])
        P += b
    return blocks
