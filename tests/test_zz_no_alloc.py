"""prunekv_score_static: scoring for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc -- an allocator or memory-pool hook (a
device allocation from inside it would re-enter the allocator), a host that
replays frozen CUDA graphs (new allocations would not be part of the captured
memory), an embedding runtime that hands out no workspace.  The fixed-scratch
entry point serves them from a device array inside the library.  These checks
call it through the C ABI, several times in a row, each call needing more
scratch than the one before (so every call runs on scratch the previous one
left behind, and reads past the previous call's layout), on both kernel paths
(tcgen05 for bf16 at d = 128, CUDA cores for fp32 and d = 64).  Each result
must equal the workspace entry point's bit for bit -- both run the same
kernels on the same plan -- and its device status must read VC_OK.  One case
is also compared with the fp64 oracle.  This file is named to be collected
last.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import prunekv as ok
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
SCORE_RTOL = 2e-5    # the score tolerance of the oracle parity tests


def _inputs(L, Hq, Hkv, d, n, W, key, dtype):
    q = synth._round(synth.normal(key, 0, L * Hq * W * d, "cpu").view(L, Hq, W, d), dtype)
    k = synth._round(synth.normal(key + 1, 0, L * Hkv * n * d, "cpu").view(L, Hkv, n, d), dtype)
    return q.to(DEV), k.to(DEV)


def _static_scores(Q, K, rank_mode):
    L, Hq, W, d = Q.shape
    _, Hkv, n, _ = K.shape
    shape = (Hkv, n) if rank_mode == vc.VC_RANK_SHARED else (L, Hkv, n)
    out = torch.full(shape, float("nan"), dtype=torch.float32, device=DEV)
    code = vc.VC_BF16 if Q.dtype == torch.bfloat16 else vc.VC_F32
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = vc.lib().prunekv_score_static(
        ctypes.c_void_p(Q.data_ptr()), ctypes.c_void_p(K.data_ptr()), code, L, Hq, Hkv, d, n,
        W, 0.0, rank_mode, None, ctypes.c_void_p(out.data_ptr()), stream)
    assert rc == vc.VC_OK
    assert vc.lib().prunekv_score_static_status(stream) == vc.VC_OK
    return out


# (L, Hq, Hkv, d, n, W), ranking, stream key, dtype; each needs more scratch than the last
CASES = [((3, 7, 1, 128, 777, 20), vc.VC_RANK_SHARED, 57, torch.bfloat16),
         ((2, 8, 4, 64, 1024, 40), vc.VC_RANK_SHARED, 71, torch.float32),
         ((4, 8, 2, 128, 1500, 32), vc.VC_RANK_PER_LAYER, 31, torch.bfloat16),
         ((5, 8, 2, 64, 900, 48), vc.VC_RANK_PER_LAYER, 93, torch.bfloat16)]


def test_static_scratch_equals_workspace_entry_point_call_after_call():
    need = [vc.prunekv_score_workspace_size(s[0], s[1], s[5]) for s, _, _, _ in CASES]
    assert need == sorted(need) and len(set(need)) == len(need)
    for i, (shape, mode, key, dtype) in enumerate(CASES):
        Q, K = _inputs(*shape, key, dtype)
        got = _static_scores(Q, K, mode)
        ref = vc.prunekv_score(Q, K, rank_mode=mode)
        torch.cuda.synchronize()
        assert torch.isfinite(got).all(), "case %d" % i
        assert torch.equal(got, ref), "case %d: max rel diff %g" % (
            i, float(((got - ref).abs() / ref.abs()).max()))
        if i == 0:
            # and against the fp64 oracle (same inputs, widened)
            s_ref = ok.token_scores(Q.cpu().double().numpy(), K.cpu().double().numpy())
            g = got.cpu().double().numpy()
            err = np.abs(g - s_ref) / np.maximum(np.abs(s_ref), 1e-30)
            assert float(err.max()) <= SCORE_RTOL, float(err.max())


def test_static_scratch_rejects_oversized_problems():
    p = ctypes.c_void_p(256)
    cap = vc.prunekv_score_static_capacity()
    assert vc.prunekv_score_workspace_size(256, 64, 4096) > cap
    # L*Hq*W window rows far beyond the fixed scratch: refused before any device work
    rc = vc.lib().prunekv_score_static(p, p, vc.VC_BF16, 256, 64, 8, 128, 100, 4096, 0.0,
                                       vc.VC_RANK_SHARED, None, p, None)
    assert rc == vc.VC_ERR_WORKSPACE
