"""Python binding of libviscache (include/viscache.h): argument marshalling only.

Every function here has the name of the C entry point it calls.  torch is used
for device memory (outputs and workspaces) and for the current CUDA stream;
every step of the compression pass runs in the library's kernels.  There is no
fallback: if ``_lib/libviscache.so`` is missing or fails to load, importing
the functions raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence, Tuple

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libviscache.so")

VC_OK = 0
VC_ERR_INVALID_ARG = 1
VC_ERR_INFEASIBLE = 2
VC_ERR_WORKSPACE = 3
VC_ERR_CUDA = 4
VC_ERR_DEVICE_TIMEOUT = 5
VC_ERR_UNSUPPORTED = 6
VC_ERR_DEVICE_INDEX = 7
VC_BF16, VC_F32 = 0, 1
VC_RANK_SHARED, VC_RANK_PER_LAYER = 0, 1
VC_SCHED_PARABOLA, VC_SCHED_FIXED, VC_SCHED_ARITHMETIC, VC_SCHED_GEOMETRIC = 0, 1, 2, 3
VC_DROP_SURVIVORS, VC_DROP_ALL = 0, 1
VC_PATH_AUTO, VC_PATH_SIMT = 0, 1
VC_TEST_WAIT_SCORE_LSE, VC_TEST_WAIT_SCORE_COLSUM, VC_TEST_WAIT_FUSE = 1, 2, 4

_ERR_NAMES = {1: "VC_ERR_INVALID_ARG", 2: "VC_ERR_INFEASIBLE", 3: "VC_ERR_WORKSPACE",
              4: "VC_ERR_CUDA", 5: "VC_ERR_DEVICE_TIMEOUT", 6: "VC_ERR_UNSUPPORTED",
              7: "VC_ERR_DEVICE_INDEX"}

EXPORTED = ("viscache_plan_budgets", "viscache_plan_budgets_ex", "prunekv_score_workspace_size", "prunekv_score",
            "prunekv_select_workspace_size", "prunekv_select", "prunekv_fuse_workspace_size",
            "prunekv_fuse_compact", "prunekv_workspace_size", "prunekv_compress",
            "prunekv_get_status", "viscache_version", "viscache_profile_enable",
            "viscache_profile_read", "prunekv_score_static", "prunekv_score_static_capacity",
            "prunekv_score_static_status", "viscache_set_kernel_path", "viscache_set_dependent_launch",
            "viscache_test_inject_wait",
            "viscache_device_accessible", "viscache_scout_workspace_size", "viscache_scout_sizes", "viscache_scout_mmr",
            "viscache_decode_workspace_size", "viscache_decode_attention",
            "viscache_kv4_sizes", "viscache_kv4_quantize", "viscache_kv4_dequantize",
            "viscache_decode_attention_kv4")


class VisCacheError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__("%s failed: %s (%d)" % (fn, _ERR_NAMES.get(code, "unknown"), code))
        self.code = code


class vc_batch(ctypes.Structure):
    _fields_ = [("n_req", ctypes.c_int32), ("n_vis", ctypes.POINTER(ctypes.c_int32)),
                ("W", ctypes.POINTER(ctypes.c_int32)), ("rr_num", ctypes.POINTER(ctypes.c_uint32)),
                ("rr_den", ctypes.POINTER(ctypes.c_uint32))]


class vc_params(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32),
                ("d", ctypes.c_int32), ("dtype", ctypes.c_int32), ("h", ctypes.c_int32),
                ("m_num", ctypes.c_uint32), ("m_den", ctypes.c_uint32), ("mu", ctypes.c_float),
                ("tau", ctypes.c_float), ("scale", ctypes.c_float), ("rank_mode", ctypes.c_int32),
                ("schedule", ctypes.c_int32), ("drop_mode", ctypes.c_int32)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library (loads on first use; raises if it was never built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError("libviscache.so is not built (%s); run __graft_entry__.build()" % _LIB_PATH)
        L = ctypes.CDLL(_LIB_PATH)
        vp, i32, u32, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint32, ctypes.c_float, ctypes.c_size_t
        pi32 = ctypes.POINTER(ctypes.c_int32)
        L.viscache_plan_budgets.argtypes = [i32, i32, u32, u32, i32, u32, u32, pi32, pi32, pi32]
        L.viscache_plan_budgets_ex.argtypes = [i32, i32, u32, u32, i32, u32, u32, i32, i32, pi32, pi32,
                                               pi32]
        L.viscache_scout_workspace_size.argtypes = [i32, pi32, i32]
        L.viscache_scout_workspace_size.restype = sz
        L.viscache_scout_sizes.argtypes = [i32, pi32, u32, u32, pi32]
        L.viscache_scout_mmr.argtypes = [vp, vp, i32, pi32, i32, f32, u32, u32, vp, vp, vp, pi32, vp, sz, vp]
        L.viscache_kv4_sizes.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params),
                                         ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
        L.viscache_kv4_quantize.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params), vp, vp,
                                            vp, vp, vp, vp, vp]
        L.viscache_kv4_dequantize.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params), vp, vp,
                                              vp, vp, vp, vp, vp]
        L.viscache_decode_attention_kv4.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params), i32,
                                                    vp, vp, vp, vp, vp, vp, vp, pi32, vp, vp, sz, vp]
        L.viscache_decode_workspace_size.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params), pi32]
        L.viscache_decode_workspace_size.restype = sz
        L.viscache_decode_attention.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params), i32,
                                                vp, vp, vp, vp, vp, pi32, vp, vp, sz, vp]
        L.prunekv_score_workspace_size.argtypes = [i32, i32, i32]
        L.prunekv_score_workspace_size.restype = sz
        L.prunekv_score.argtypes = [vp, vp, i32, i32, i32, i32, i32, i32, i32, f32, i32, vp, vp,
                                    vp, sz, vp]
        L.prunekv_score_static.argtypes = [vp, vp, i32, i32, i32, i32, i32, i32, i32, f32, i32, vp,
                                           vp, vp]
        L.prunekv_score_static_capacity.argtypes = []
        L.prunekv_score_static_capacity.restype = sz
        L.prunekv_score_static_status.argtypes = [vp]
        L.prunekv_select_workspace_size.argtypes = [i32, i32, i32, i32]
        L.prunekv_select_workspace_size.restype = sz
        L.prunekv_select.argtypes = [vp, i32, i32, i32, pi32, i32, i32, vp, vp, vp, vp, sz, vp]
        L.prunekv_fuse_workspace_size.argtypes = [pi32, i32, i32, i32, i32, i32]
        L.prunekv_fuse_workspace_size.restype = sz
        L.prunekv_fuse_compact.argtypes = [vp, vp, i32, i32, i32, i32, i32, pi32, i32, vp, vp, f32,
                                           f32, vp, vp, vp, sz, vp]
        L.prunekv_workspace_size.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params)]
        L.prunekv_workspace_size.restype = sz
        L.prunekv_compress.argtypes = [ctypes.POINTER(vc_batch), ctypes.POINTER(vc_params), vp, vp,
                                       vp, vp, vp, vp, vp, sz, vp]
        L.prunekv_get_status.argtypes = [vp, vp]
        L.viscache_version.restype = ctypes.c_char_p
        L.viscache_profile_enable.argtypes = [i32]
        L.viscache_set_kernel_path.argtypes = [i32]
        L.viscache_set_dependent_launch.argtypes = [i32]
        L.viscache_test_inject_wait.argtypes = [i32]
        L.viscache_device_accessible.argtypes = [vp]
        L.viscache_profile_read.argtypes = [ctypes.c_char_p, i32, ctypes.POINTER(ctypes.c_float),
                                            pi32, i32]
        _lib = L
    return _lib


def _check(fn: str, rc: int) -> None:
    if rc != VC_OK:
        raise VisCacheError(fn, rc)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return VC_BF16
    if t.dtype == torch.float32:
        return VC_F32
    raise TypeError("unsupported dtype %s (bf16 or fp32)" % t.dtype)


def _workspace(nbytes: int, device, ws: Optional[torch.Tensor]) -> torch.Tensor:
    if ws is not None:
        return ws
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)


def _i32(seq):
    arr = (ctypes.c_int32 * len(seq))(*[int(x) for x in seq])
    return arr


# ---------------------------------------------------------------------------

def viscache_version() -> str:
    return lib().viscache_version().decode()


def viscache_device_accessible(t: torch.Tensor) -> bool:
    """True if the current CUDA device can read the tensor's memory directly."""
    rc = lib().viscache_device_accessible(ctypes.c_void_p(t.data_ptr()))
    if rc < 0:
        raise VisCacheError("viscache_device_accessible", -rc)
    return rc == 1


def viscache_plan_budgets(L: int, n_vis: int, rr_num: int, rr_den: int, h: int = 0,
                          m_num: int = 3, m_den: int = 4) -> Tuple[List[int], int, int]:
    """Host planner (Eq. parabolic): returns (B[L], Nq, h)."""
    B = (ctypes.c_int32 * L)()
    nq, hh = ctypes.c_int32(), ctypes.c_int32()
    _check("viscache_plan_budgets",
           lib().viscache_plan_budgets(L, n_vis, rr_num, rr_den, h, m_num, m_den, B,
                                       ctypes.byref(nq), ctypes.byref(hh)))
    return list(B), nq.value, hh.value


def viscache_plan_budgets_ex(L: int, n_vis: int, rr_num: int, rr_den: int, h: int = 0,
                             m_num: int = 3, m_den: int = 4, schedule: int = VC_SCHED_PARABOLA,
                             drop_mode: int = VC_DROP_SURVIVORS) -> Tuple[List[int], int, int]:
    """Host planner with a budget schedule and drop-set choice: returns (B[L], Nq, h)."""
    B = (ctypes.c_int32 * L)()
    nq, hh = ctypes.c_int32(), ctypes.c_int32()
    _check("viscache_plan_budgets_ex",
           lib().viscache_plan_budgets_ex(L, n_vis, rr_num, rr_den, h, m_num, m_den, schedule,
                                          drop_mode, B, ctypes.byref(nq), ctypes.byref(hh)))
    return list(B), nq.value, hh.value


def viscache_scout_mmr(H: torch.Tensor, prompt: torch.Tensor, n_frames: Sequence[int], lam: float = 0.7,
                       p: Tuple[int, int] = (3, 4), with_gains: bool = True, stream=None,
                       out: Optional[Tuple[torch.Tensor, torch.Tensor, Optional[torch.Tensor]]] = None,
                       ws: Optional[torch.Tensor] = None):
    """Keyframe selection, Eq. (mmr): returns (order, keyframes, gains, k per video).

    H: device fp32 [sum F][D], prompt: device fp32 [n_req][D].  ``out`` may
    hold preallocated (order, keyframes, gains) int32/int32/fp32 [sum k]
    tensors and ``ws`` a workspace, so repeated calls allocate nothing.
    """
    n_req = len(n_frames)
    D = H.shape[1]
    nf = (ctypes.c_int32 * n_req)(*n_frames)
    need = lib().viscache_scout_workspace_size(n_req, nf, D)
    if need == 0:
        raise VisCacheError("viscache_scout_workspace_size", VC_ERR_INVALID_ARG)
    kk = (ctypes.c_int32 * n_req)()
    _check("viscache_scout_sizes", lib().viscache_scout_sizes(n_req, nf, p[0], p[1], kk))
    ks = list(kk)
    dev = H.device
    if out is not None:
        order, keys, gains = out
    else:
        order = torch.empty(sum(ks), dtype=torch.int32, device=dev)
        keys = torch.empty(sum(ks), dtype=torch.int32, device=dev)
        gains = torch.empty(sum(ks), dtype=torch.float32, device=dev) if with_gains else None
    ws = _workspace(need, dev, ws)
    k_out = (ctypes.c_int32 * n_req)()
    if H.dtype != torch.float32 or prompt.dtype != torch.float32 or not H.is_contiguous() \
            or not prompt.is_contiguous() or prompt.shape != (n_req, D) or H.shape[0] != sum(n_frames):
        raise VisCacheError("viscache_scout_mmr", VC_ERR_INVALID_ARG)
    _check("viscache_scout_mmr", lib().viscache_scout_mmr(
        _ptr(H), _ptr(prompt), n_req, nf, D, float(lam), p[0], p[1], _ptr(order), _ptr(keys),
        _ptr(gains), k_out, _ptr(ws), ws.numel(), _stream(stream)))
    assert list(k_out) == ks
    return order, keys, gains, ks


def prunekv_score_workspace_size(L: int, Hq: int, W: int) -> int:
    return lib().prunekv_score_workspace_size(L, Hq, W)


def prunekv_score(Qw: torch.Tensor, K: torch.Tensor, scale: float = 0.0,
                  rank_mode: int = VC_RANK_SHARED, row_lse: Optional[torch.Tensor] = None,
                  scores: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                  stream=None) -> torch.Tensor:
    """Eq. (token_score): scores [Hkv][n] (shared) or [L][Hkv][n] (per layer), fp32."""
    L, Hq, W, d = Qw.shape
    _, Hkv, n, _ = K.shape
    if scores is None:
        shape = (Hkv, n) if rank_mode == VC_RANK_SHARED else (L, Hkv, n)
        scores = torch.empty(shape, dtype=torch.float32, device=K.device)
    ws = _workspace(prunekv_score_workspace_size(L, Hq, W), K.device, ws)
    _check("prunekv_score", lib().prunekv_score(
        _ptr(Qw), _ptr(K), _dtype_code(K), L, Hq, Hkv, d, n, W, float(scale), rank_mode,
        _ptr(row_lse), _ptr(scores), _ptr(ws), ws.numel(), _stream(stream)))
    return scores


def prunekv_score_static_capacity() -> int:
    """Bytes of the library's fixed scratch array (VC_STATIC_SCRATCH_BYTES)."""
    return lib().prunekv_score_static_capacity()


def prunekv_score_static_status(stream=None) -> int:
    """Device status of the last prunekv_score_static call (synchronises `stream`)."""
    return lib().prunekv_score_static_status(_stream(stream))


def prunekv_score_static(Qw: torch.Tensor, K: torch.Tensor, scale: float = 0.0,
                         rank_mode: int = VC_RANK_SHARED, row_lse: Optional[torch.Tensor] = None,
                         scores: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """prunekv_score with the library's fixed scratch array instead of a workspace.

    For callers that cannot allocate device memory: the C entry point
    allocates nothing (pass ``scores`` to keep this wrapper allocation-free
    too).  Calls overlapping on the GPU race on the shared scratch.
    """
    L, Hq, W, d = Qw.shape
    _, Hkv, n, _ = K.shape
    if scores is None:
        shape = (Hkv, n) if rank_mode == VC_RANK_SHARED else (L, Hkv, n)
        scores = torch.empty(shape, dtype=torch.float32, device=K.device)
    _check("prunekv_score_static", lib().prunekv_score_static(
        _ptr(Qw), _ptr(K), _dtype_code(K), L, Hq, Hkv, d, n, W, float(scale), rank_mode,
        _ptr(row_lse), _ptr(scores), _stream(stream)))
    return scores


def prunekv_select_workspace_size(L: int, Hkv: int, n_vis: int, rank_mode: int = VC_RANK_SHARED) -> int:
    return lib().prunekv_select_workspace_size(L, Hkv, n_vis, rank_mode)


def drop_rows(B: Sequence[int], Nq: int, Hkv: int) -> int:
    return Hkv * sum(Nq - b for b in B if b > 0)


def prunekv_select(scores: torch.Tensor, B: Sequence[int], Nq: int, rank_mode: int = VC_RANK_SHARED,
                   ws: Optional[torch.Tensor] = None, stream=None):
    """Ranking and keep/drop lists: returns (rank, keep_idx, drop_idx), int32 device tensors."""
    L = len(B)
    Hkv, n = scores.shape[-2], scores.shape[-1]
    dev = scores.device
    rank = torch.empty(scores.shape, dtype=torch.int32, device=dev)
    keep = torch.empty(max(1, Hkv * sum(B)), dtype=torch.int32, device=dev)
    drop = torch.empty(max(1, drop_rows(B, Nq, Hkv)), dtype=torch.int32, device=dev)
    ws = _workspace(prunekv_select_workspace_size(L, Hkv, n, rank_mode), dev, ws)
    _check("prunekv_select", lib().prunekv_select(
        _ptr(scores), L, Hkv, n, _i32(B), Nq, rank_mode, _ptr(rank), _ptr(keep), _ptr(drop),
        _ptr(ws), ws.numel(), _stream(stream)))
    return rank, keep[:Hkv * sum(B)], drop[:drop_rows(B, Nq, Hkv)]


def prunekv_fuse_workspace_size(B: Sequence[int], Hkv: int, d: int, n_vis: int, Nq: int) -> int:
    return lib().prunekv_fuse_workspace_size(_i32(B), len(B), Hkv, d, n_vis, Nq)


def prunekv_fuse_compact(K: torch.Tensor, V: torch.Tensor, B: Sequence[int], Nq: int,
                         keep_idx: torch.Tensor, drop_idx: torch.Tensor, mu: float = 0.7,
                         tau: float = 1.0, K_out: Optional[torch.Tensor] = None,
                         V_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                         stream=None):
    """Prune keys / fuse values (Eq. redistribution, Eq. weight_fusion): returns (K_out, V_out)."""
    L, Hkv, n, d = K.shape
    rows = Hkv * sum(B)
    if K_out is None:
        K_out = torch.empty((max(rows, 1), d), dtype=K.dtype, device=K.device)
    if V_out is None:
        V_out = torch.empty((max(rows, 1), d), dtype=V.dtype, device=V.device)
    keep_idx = keep_idx if keep_idx.numel() else torch.zeros(1, dtype=torch.int32, device=K.device)
    drop_idx = drop_idx if drop_idx.numel() else torch.zeros(1, dtype=torch.int32, device=K.device)
    ws = _workspace(prunekv_fuse_workspace_size(B, Hkv, d, n, Nq), K.device, ws)
    _check("prunekv_fuse_compact", lib().prunekv_fuse_compact(
        _ptr(K), _ptr(V), _dtype_code(K), L, Hkv, d, n, _i32(B), Nq, _ptr(keep_idx),
        _ptr(drop_idx), float(mu), float(tau), _ptr(K_out), _ptr(V_out), _ptr(ws), ws.numel(),
        _stream(stream)))
    return K_out[:rows], V_out[:rows]


class Batch:
    """Host description of a batch (vc_batch) kept alive with its arrays."""

    def __init__(self, n_vis: Sequence[int], W: Sequence[int], rr: Sequence[Tuple[int, int]]):
        k = len(n_vis)
        self._n = (ctypes.c_int32 * k)(*n_vis)
        self._w = (ctypes.c_int32 * k)(*W)
        self._a = (ctypes.c_uint32 * k)(*[a for a, _ in rr])
        self._b = (ctypes.c_uint32 * k)(*[b for _, b in rr])
        self.c = vc_batch(k, self._n, self._w, self._a, self._b)
        self.n_vis, self.W, self.rr = list(n_vis), list(W), list(rr)


def make_params(L: int, Hq: int, Hkv: int, d: int, dtype: int, h: int = 0, m=(3, 4),
                mu: float = 0.7, tau: float = 1.0, scale: float = 0.0,
                rank_mode: int = VC_RANK_SHARED, schedule: int = VC_SCHED_PARABOLA,
                drop_mode: int = VC_DROP_SURVIVORS) -> vc_params:
    return vc_params(L, Hq, Hkv, d, dtype, h, m[0], m[1], mu, tau, scale, rank_mode, schedule,
                     drop_mode)


def prunekv_workspace_size(batch: Batch, params: vc_params) -> int:
    return lib().prunekv_workspace_size(ctypes.byref(batch.c), ctypes.byref(params))


def compressed_rows(batch: Batch, params: vc_params) -> int:
    rows = 0
    for n, (a, b) in zip(batch.n_vis, batch.rr):
        B, _, _ = viscache_plan_budgets_ex(params.L, n, a, b, params.h, params.m_num, params.m_den,
                                           params.schedule, params.drop_mode)
        rows += params.Hkv * sum(B)
    return rows


def prunekv_compress(batch: Batch, params: vc_params, Qw: torch.Tensor, K: torch.Tensor,
                     V: torch.Tensor, K_out: Optional[torch.Tensor] = None,
                     V_out: Optional[torch.Tensor] = None, idx_out: Optional[torch.Tensor] = None,
                     ws: Optional[torch.Tensor] = None, stream=None):
    """The whole pass over a packed batch: returns (K_out, V_out, idx_out)."""
    rows = compressed_rows(batch, params)
    dev = K.device
    if K_out is None:
        K_out = torch.empty((max(rows, 1), params.d), dtype=K.dtype, device=dev)
    if V_out is None:
        V_out = torch.empty((max(rows, 1), params.d), dtype=V.dtype, device=dev)
    if idx_out is None:
        idx_out = torch.empty(max(rows, 1), dtype=torch.int32, device=dev)
    ws = _workspace(prunekv_workspace_size(batch, params), dev, ws)
    _check("prunekv_compress", lib().prunekv_compress(
        ctypes.byref(batch.c), ctypes.byref(params), _ptr(Qw), _ptr(K), _ptr(V), _ptr(K_out),
        _ptr(V_out), _ptr(idx_out), _ptr(ws), ws.numel(), _stream(stream)))
    return K_out[:rows], V_out[:rows], idx_out[:rows]


def viscache_decode_workspace_size(batch: Batch, params: vc_params,
                                   n_text: Optional[Sequence[int]] = None) -> int:
    return lib().viscache_decode_workspace_size(ctypes.byref(batch.c), ctypes.byref(params),
                                                _i32(n_text) if n_text is not None else None)


def viscache_decode_attention(batch: Batch, params: vc_params, layer: int, q: torch.Tensor,
                              K_out: torch.Tensor, V_out: torch.Tensor,
                              K_text: Optional[torch.Tensor] = None, V_text: Optional[torch.Tensor] = None,
                              n_text: Optional[Sequence[int]] = None, out: Optional[torch.Tensor] = None,
                              ws: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """One decode step's attention in `layer` over the compressed cache: q [n_req][Hq][d] -> out."""
    if out is None:
        out = torch.empty_like(q)
    nt = _i32(n_text) if n_text is not None else None
    if ws is None:
        need = lib().viscache_decode_workspace_size(ctypes.byref(batch.c), ctypes.byref(params), nt)
        if need == 0:
            raise VisCacheError("viscache_decode_workspace_size", VC_ERR_INVALID_ARG)
        ws = _workspace(need, q.device, None)
    _check("viscache_decode_attention", lib().viscache_decode_attention(
        ctypes.byref(batch.c), ctypes.byref(params), int(layer), _ptr(q), _ptr(K_out), _ptr(V_out),
        _ptr(K_text), _ptr(V_text), nt, _ptr(out), _ptr(ws), ws.numel(), _stream(stream)))
    return out


def viscache_decode_attention_kv4(batch: Batch, params: vc_params, layer: int, q: torch.Tensor,
                                  kv4, K_text: Optional[torch.Tensor] = None,
                                  V_text: Optional[torch.Tensor] = None, n_text: Optional[Sequence[int]] = None,
                                  out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                                  stream=None) -> torch.Tensor:
    """Decode step in `layer` over the 4-bit cache kv4 = (K_codes, V_codes, K_params, V_params)."""
    if out is None:
        out = torch.empty_like(q)
    nt = _i32(n_text) if n_text is not None else None
    if ws is None:
        need = lib().viscache_decode_workspace_size(ctypes.byref(batch.c), ctypes.byref(params), nt)
        if need == 0:
            raise VisCacheError("viscache_decode_workspace_size", VC_ERR_INVALID_ARG)
        ws = _workspace(need, q.device, None)
    kc, vc_, kp, vp_ = kv4
    _check("viscache_decode_attention_kv4", lib().viscache_decode_attention_kv4(
        ctypes.byref(batch.c), ctypes.byref(params), int(layer), _ptr(q), _ptr(kc), _ptr(vc_), _ptr(kp),
        _ptr(vp_), _ptr(K_text), _ptr(V_text), nt, _ptr(out), _ptr(ws), ws.numel(), _stream(stream)))
    return out


def viscache_kv4_sizes(batch: Batch, params: vc_params) -> Tuple[int, int]:
    """(rows, key groups) of the compacted cache's 4-bit form."""
    rows, groups = ctypes.c_int64(0), ctypes.c_int64(0)
    _check("viscache_kv4_sizes", lib().viscache_kv4_sizes(ctypes.byref(batch.c), ctypes.byref(params),
                                                          ctypes.byref(rows), ctypes.byref(groups)))
    return rows.value, groups.value


def viscache_kv4_quantize(batch: Batch, params: vc_params, K_out: torch.Tensor, V_out: torch.Tensor,
                          out=None, stream=None):
    """4-bit codes and (scale, min) parameters of the compacted cache:
    returns (K_codes [rows][d/2], V_codes [rows][d/2], K_params [groups][d][2], V_params [rows][d/32][2])."""
    rows, groups = viscache_kv4_sizes(batch, params)
    d, dev = params.d, K_out.device
    if out is None:
        out = (torch.empty((max(rows, 1), d // 2), dtype=torch.uint8, device=dev),
               torch.empty((max(rows, 1), d // 2), dtype=torch.uint8, device=dev),
               torch.empty((max(groups, 1), d, 2), dtype=torch.float32, device=dev),
               torch.empty((max(rows, 1), d // 32, 2), dtype=torch.float32, device=dev))
    kc, vc_, kp, vp_ = out
    _check("viscache_kv4_quantize", lib().viscache_kv4_quantize(
        ctypes.byref(batch.c), ctypes.byref(params), _ptr(K_out), _ptr(V_out), _ptr(kc), _ptr(vc_),
        _ptr(kp), _ptr(vp_), _stream(stream)))
    return kc[:rows], vc_[:rows], kp[:groups], vp_[:rows]


def viscache_kv4_dequantize(batch: Batch, params: vc_params, K_codes: torch.Tensor, V_codes: torch.Tensor,
                            K_params: torch.Tensor, V_params: torch.Tensor, dtype=torch.bfloat16,
                            out=None, stream=None):
    """Reconstruction (K_hat, V_hat) [rows][d] of the 4-bit cache in `dtype`."""
    rows = K_codes.shape[0]
    if out is None:
        out = (torch.empty((max(rows, 1), params.d), dtype=dtype, device=K_codes.device),
               torch.empty((max(rows, 1), params.d), dtype=dtype, device=K_codes.device))
    kh, vh = out
    _check("viscache_kv4_dequantize", lib().viscache_kv4_dequantize(
        ctypes.byref(batch.c), ctypes.byref(params), _ptr(K_codes), _ptr(V_codes), _ptr(K_params),
        _ptr(V_params), _ptr(kh), _ptr(vh), _stream(stream)))
    return kh[:rows], vh[:rows]


def viscache_set_kernel_path(path: int) -> None:
    """VC_PATH_AUTO (tensor cores for bf16, d=128) or VC_PATH_SIMT (CUDA cores everywhere)."""
    _check("viscache_set_kernel_path", lib().viscache_set_kernel_path(path))


def viscache_set_dependent_launch(on: bool) -> None:
    """True (default): kernels after a call's first are dependent launches; False: ordinary launches."""
    _check("viscache_set_dependent_launch", lib().viscache_set_dependent_launch(1 if on else 0))


def viscache_test_inject_wait(kernel_mask: int) -> None:
    """Test support: the named tensor-core kernels add one wait that gives up (0 = off)."""
    _check("viscache_test_inject_wait", lib().viscache_test_inject_wait(kernel_mask))


def viscache_profile_enable(on: bool) -> None:
    _check("viscache_profile_enable", lib().viscache_profile_enable(1 if on else 0))


def viscache_profile_read(max_kernels: int = 32):
    """{kernel name: (total ms, launches)} recorded since profiling was enabled / last read."""
    names = ctypes.create_string_buffer(4096)
    ms = (ctypes.c_float * max_kernels)()
    cnt = (ctypes.c_int32 * max_kernels)()
    k = lib().viscache_profile_read(names, 4096, ms, cnt, max_kernels)
    if k < 0:
        raise VisCacheError("viscache_profile_read", -k)
    keys = names.value.decode().split("\n")[:k]
    return {keys[i]: (ms[i], cnt[i]) for i in range(k)}


def prunekv_get_status(ws: torch.Tensor, stream=None) -> int:
    return lib().prunekv_get_status(_ptr(ws), _stream(stream))
