"""Failure detection on the GPU without a fault: bounded device waits that give up.

Every wait of the tensor-core kernels (score_lse_tc, score_colsum_tc, fuse_v_tc)
is bounded and records VC_ERR_DEVICE_TIMEOUT in the workspace status word when
it gives up.  viscache_test_inject_wait makes one consumer warp of the chosen
kernel wait on an mbarrier that nothing ever completes (a flag that nothing
sets), with a short limit; the wait must give up, the host must read the
timeout through prunekv_get_status (or prunekv_score_static_status for the
fixed-scratch entry point), and the context must stay usable: the same calls
without the injected wait then return VC_OK and match the fp64 oracle.  The
injected wait touches none of the kernel's own barriers or copies, so the
timed-out launch still completes its work (its outputs equal the clean
launch's bit for bit).
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc
from tests.parity import check_request

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
L, Hq, Hkv, d, n, W = 3, 14, 2, 128, 2049, 20
RR = (23, 100)


def _inputs():
    mk = lambda shape, k: synth._round(synth.normal(4100 + k, 0, int(np.prod(shape)), "cpu").view(*shape),
                                        torch.bfloat16)
    return mk((L, Hq, W, d), 1), mk((L, Hkv, n, d), 2), mk((L, Hkv, n, d), 3)


@pytest.fixture
def inject():
    yield vc.viscache_test_inject_wait
    vc.viscache_test_inject_wait(0)


def _steps(Q, K, V, B, Nq):
    ws_s = torch.empty(vc.prunekv_score_workspace_size(L, Hq, W), dtype=torch.uint8, device=DEV)
    s = vc.prunekv_score(Q, K, ws=ws_s)
    st_s = vc.prunekv_get_status(ws_s)
    _, keep, drop = vc.prunekv_select(s, B, Nq)
    ws_f = torch.empty(vc.prunekv_fuse_workspace_size(B, Hkv, d, n, Nq), dtype=torch.uint8, device=DEV)
    Ko, Vo = vc.prunekv_fuse_compact(K, V, B, Nq, keep, drop, 0.7, 1.0, ws=ws_f)
    st_f = vc.prunekv_get_status(ws_f)
    return dict(scores=s, keep=keep, drop=drop, K_out=Ko, V_out=Vo), st_s, st_f


@pytest.mark.parametrize("mask,where", [(vc.VC_TEST_WAIT_SCORE_LSE, "score"),
                                        (vc.VC_TEST_WAIT_SCORE_COLSUM, "score"),
                                        (vc.VC_TEST_WAIT_FUSE, "fuse")])
def test_wait_gives_up_reports_timeout_and_context_stays_usable(mask, where, inject):
    q, k, v = _inputs()
    Q, K, V = q.to(DEV), k.to(DEV), v.to(DEV)
    B, Nq, _ = vc.viscache_plan_budgets(L, n, *RR)
    inject(mask)
    bad, st_s, st_f = _steps(Q, K, V, B, Nq)
    torch.cuda.synchronize()
    assert (st_s, st_f) == ((vc.VC_ERR_DEVICE_TIMEOUT, vc.VC_OK) if where == "score"
                            else (vc.VC_OK, vc.VC_ERR_DEVICE_TIMEOUT))
    inject(0)
    good, st_s, st_f = _steps(Q, K, V, B, Nq)
    torch.cuda.synchronize()
    assert (st_s, st_f) == (vc.VC_OK, vc.VC_OK)
    check_request(q, k, v, B, Nq, good, 0.7, 1.0)
    for key in good:
        assert torch.equal(bad[key], good[key]), key


def test_fused_pass_and_static_scoring_report_timeouts(inject):
    q, k, v = _inputs()
    Q, K, V = q.to(DEV), k.to(DEV), v.to(DEV)
    batch = vc.Batch([n], [W], [RR])
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    ws = torch.empty(vc.prunekv_workspace_size(batch, prm), dtype=torch.uint8, device=DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    s_static = torch.empty((Hkv, n), dtype=torch.float32, device=DEV)

    def static_call():
        rc = vc.lib().prunekv_score_static(ctypes.c_void_p(Q.data_ptr()), ctypes.c_void_p(K.data_ptr()),
                                           vc.VC_BF16, L, Hq, Hkv, d, n, W, 0.0, vc.VC_RANK_SHARED, None,
                                           ctypes.c_void_p(s_static.data_ptr()), stream)
        assert rc == vc.VC_OK
        return vc.lib().prunekv_score_static_status(stream)

    inject(vc.VC_TEST_WAIT_SCORE_LSE | vc.VC_TEST_WAIT_SCORE_COLSUM | vc.VC_TEST_WAIT_FUSE)
    out_bad = vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_ERR_DEVICE_TIMEOUT
    assert static_call() == vc.VC_ERR_DEVICE_TIMEOUT
    inject(0)
    out = vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_OK
    assert static_call() == vc.VC_OK
    torch.cuda.synchronize()
    for a, b in zip(out_bad, out):
        assert torch.equal(a, b)
    assert torch.equal(s_static, vc.prunekv_score(Q, K))

