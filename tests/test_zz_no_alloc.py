"""prunekv_score_static: scoring for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc -- an allocator or memory-pool hook (a
device allocation from inside it would re-enter the allocator), a host that
replays frozen CUDA graphs (new allocations would not be part of the captured
memory), an embedding runtime that hands out no workspace.  The fixed-scratch
entry point serves them from a device array inside the library.  These checks
call it through the C ABI and compare it with the workspace entry point,
twice in a row with different shapes so that the second call runs on scratch
the first one left behind.  This file is named to be collected last.
"""
import ctypes

import pytest
import torch

from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
RTOL = 2e-5          # the score tolerance of the parity tests


def _inputs(L, Hq, Hkv, d, n, W, key):
    q = synth._round(synth.normal(key, 0, L * Hq * W * d, "cpu").view(L, Hq, W, d), torch.bfloat16)
    k = synth._round(synth.normal(key + 1, 0, L * Hkv * n * d, "cpu").view(L, Hkv, n, d), torch.bfloat16)
    return q.to(DEV), k.to(DEV)


def _static_scores(Q, K, rank_mode):
    L, Hq, W, d = Q.shape
    _, Hkv, n, _ = K.shape
    shape = (Hkv, n) if rank_mode == vc.VC_RANK_SHARED else (L, Hkv, n)
    out = torch.full(shape, float("nan"), dtype=torch.float32, device=DEV)
    rc = vc.lib().prunekv_score_static(
        ctypes.c_void_p(Q.data_ptr()), ctypes.c_void_p(K.data_ptr()), vc.VC_BF16, L, Hq, Hkv, d, n,
        W, 0.0, rank_mode, None, ctypes.c_void_p(out.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == vc.VC_OK
    return out


def test_static_scratch_matches_workspace_entry_point_twice():
    cases = [((4, 8, 2, 128, 1500, 32), vc.VC_RANK_SHARED, 31),
             ((3, 7, 1, 128, 777, 20), vc.VC_RANK_PER_LAYER, 57)]
    for shape, mode, key in cases:
        Q, K = _inputs(*shape, key)
        got = _static_scores(Q, K, mode)
        ref = vc.prunekv_score(Q, K, rank_mode=mode)
        torch.cuda.synchronize()
        assert torch.isfinite(got).all()
        assert torch.allclose(got, ref, rtol=RTOL, atol=0), float(((got - ref).abs() / ref).max())


def test_static_scratch_rejects_oversized_problems():
    p = ctypes.c_void_p(256)
    # L*Hq*W window rows far beyond the fixed scratch: refused before any device work
    rc = vc.lib().prunekv_score_static(p, p, vc.VC_BF16, 256, 64, 8, 128, 100, 4096, 0.0,
                                       vc.VC_RANK_SHARED, None, p, None)
    assert rc == vc.VC_ERR_WORKSPACE
    assert vc.prunekv_score_workspace_size(256, 64, 4096) > vc.STATIC_SCRATCH_BYTES
