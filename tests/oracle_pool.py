"""The fp64 oracle over whole workloads, layer by layer on the host cores.

Test infrastructure for the full-size parity tests.  The oracle itself is
unchanged: each task regenerates one layer of one request from the seeded
generator (``synth`` draws any layer on its own), widens it to float64 and
calls ``oracle.prunekv`` on the (layer, KV head) slices -- the oracle's
per-(layer, head) quantities depend only on that slice, so the results are
the ones a single whole-request call would give.  Tasks run in worker
processes started with ``spawn`` (never forked from a process that has used
CUDA).  Workers only read the GPU's outputs handed to them; nothing here
touches a device.

Two kinds of task, both per (workload, request, layer):

* ``layer_scores``: the oracle's per-layer column sums of the softmax,
  sum_{j in G(g)} sum_i A^l_{j,i,v}, for every KV head g ([Hkv][n] float64);
  the shared score is then their sum over layers divided by L, exactly as
  ``oracle.prunekv.token_scores`` forms it.
* ``layer_outputs``: given the GPU's keep and drop lists and its K_out / V_out
  rows of that layer, checks K_out bit for bit against the cache rows and
  V_out against ``oracle.prunekv.fuse_values`` on the GPU's own lists (the
  parity rule for V), returning the failures as text.
"""
from __future__ import annotations

import multiprocessing as mp
import os
from typing import Dict, List, Optional, Tuple

import numpy as np

_Q: Dict[tuple, object] = {}


def _query(wl, r: int):
    """Request r's rounded Qw on the CPU (cached per worker)."""
    key = (wl, r)
    if key not in _Q:
        from paper_2608_24063_gb300 import synth
        if len(_Q) > 4:
            _Q.clear()
        _Q[key] = synth.make_q(wl, r, "cpu")
    return _Q[key]


def _layer_kv(wl, r: int, l: int):
    from paper_2608_24063_gb300 import synth
    q = _query(wl, r)
    K, V = synth.make_kv(wl, r, q, "cpu", layers=[l])
    return q[l], K[l].clone(), V[l].clone()


def layer_scores(task) -> Tuple[int, int, np.ndarray]:
    """(r, l, per-layer oracle scores [Hkv][n]) for task (workload, r, l)."""
    from oracle import prunekv as ok
    wl, r, l = task
    q, K, _ = _layer_kv(wl, r, l)
    G = wl.Hq // wl.Hkv
    Qn = q.double().numpy()
    Kn = K.double().numpy()
    out = np.empty((wl.Hkv, Kn.shape[1]))
    for g in range(wl.Hkv):
        out[g] = ok.token_scores(Qn[None, g * G:(g + 1) * G], Kn[None, g:g + 1], None,
                                 "per_layer", None)[0, 0]
    return r, l, out


def layer_outputs(task) -> Tuple[int, int, List[str]]:
    """Check one layer's K_out (bit-exact) and V_out (oracle fusion on the GPU's lists).

    task = (workload, r, l, keep [Hkv][B] int64, drop [Hkv][D] int64,
            K_out bits [Hkv*B][d] int16, V_out [Hkv*B][d] float64, mu, tau, tol)
    """
    import torch

    from oracle import prunekv as ok
    from tests.parity import check_v_rows
    wl, r, l, keep, drop, kbits, vout, mu, tau, tol = task
    _, K, V = _layer_kv(wl, r, l)
    kb = K.contiguous().view(torch.int16).numpy()
    Vn = V.double().numpy()
    fails = []
    B = keep.shape[1]
    for g in range(wl.Hkv):
        kg, dg = keep[g], drop[g]
        rows = slice(g * B, (g + 1) * B)
        if not np.array_equal(kbits[rows], kb[g][kg]):
            fails.append("K_out r=%d l=%d g=%d differs" % (r, l, g))
        ref = ok.fuse_values(Vn[g], kg, dg, mu, tau)
        try:
            check_v_rows(vout[rows], ref, tol, "r=%d l=%d g=%d" % (r, l, g))
        except AssertionError as e:
            fails.append(str(e))
    return r, l, fails


def workers() -> int:
    """Processes for the pool: the host cores, bounded by ~3 GB of free memory each."""
    try:
        cores = len(os.sched_getaffinity(0))
    except AttributeError:
        cores = os.cpu_count() or 1
    avail = None
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    avail = int(line.split()[1]) * 1024
    except OSError:
        pass
    n = min(cores, 16)
    if avail is not None:
        n = min(n, max(1, int(avail // (3 << 30))))
    return max(1, n)


def _init_worker() -> None:
    import torch
    torch.set_num_threads(1)


_ONE_THREAD = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def pool(processes: Optional[int] = None):
    """A spawn-started process pool (safe after the parent initialised CUDA); one
    BLAS and one torch thread per worker, so the workers do not oversubscribe."""
    saved = {k: os.environ.get(k) for k in _ONE_THREAD}
    try:
        for k in _ONE_THREAD:
            os.environ[k] = "1"          # read by the children's numpy at import
        return mp.get_context("spawn").Pool(processes or workers(), initializer=_init_worker)
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
