"""Failure detection on the GPU without a fault: bounded device waits that give up.

Every wait of the tensor-core kernels (score_lse_tc, score_colsum_tc, fuse_v_tc)
is bounded and records VC_ERR_DEVICE_TIMEOUT in the workspace status word when
it gives up.  viscache_test_inject_wait makes one consumer warp of every CTA of
the chosen kernel wait on an mbarrier that nothing ever completes (a flag that
nothing sets), with a short limit; when that wait gives up the warp records the
timeout and raises the CTA's abort flag, exactly as a real give-up does.  The
rest of the CTA pair then takes the abort path: waits stop, the MMA issuer
stops issuing, warps that gave up keep meeting their named barriers without
working, the even CTA drains the pair's copies with the odd CTA's fill counts,
both CTAs wait for the pair's last MMA, and only then is tensor memory freed.

The checks: the launch returns (well inside the device wait limits), the host
reads the timeout through prunekv_get_status (or prunekv_score_static_status
for the fixed-scratch entry point), and the context stays usable: the same
calls without the injected wait return VC_OK and match the fp64 oracle.  The
aborted launch's outputs are incomplete by design and are not compared.
"""
import ctypes
import time

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
# An aborted launch ends within a few device wait limits (each about a second)
# even when one CTA of a pair gives up long before the other; with every CTA
# aborting at once it ends in milliseconds.
ABORT_SECONDS = 30.0


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
    t0 = time.perf_counter()
    _, st_s, st_f = _steps(Q, K, V, B, Nq)
    torch.cuda.synchronize()
    assert time.perf_counter() - t0 < ABORT_SECONDS
    assert (st_s, st_f) == ((vc.VC_ERR_DEVICE_TIMEOUT, vc.VC_OK) if where == "score"
                            else (vc.VC_OK, vc.VC_ERR_DEVICE_TIMEOUT))
    inject(0)
    good, st_s, st_f = _steps(Q, K, V, B, Nq)
    torch.cuda.synchronize()
    assert (st_s, st_f) == (vc.VC_OK, vc.VC_OK)
    check_request(q, k, v, B, Nq, good, 0.7, 1.0)


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
    t0 = time.perf_counter()
    vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_ERR_DEVICE_TIMEOUT
    assert static_call() == vc.VC_ERR_DEVICE_TIMEOUT
    assert time.perf_counter() - t0 < 2 * ABORT_SECONDS
    inject(0)
    out = vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_OK
    assert static_call() == vc.VC_OK
    torch.cuda.synchronize()
    B, Nq, _ = vc.viscache_plan_budgets(L, n, *RR)
    check_request(q, k, v, B, Nq, _steps(Q, K, V, B, Nq)[0], 0.7, 1.0)
    assert torch.equal(s_static, vc.prunekv_score(Q, K))
    Ko, Vo, _ = out
    assert not bool(torch.isnan(Ko.float()).any()) and not bool(torch.isnan(Vo.float()).any())



def test_abort_with_several_units_per_fusion_pair(inject):
    # a shape whose fusion deals two to four units to every CTA pair and whose
    # score passes run tens of tiles per unit: the injected give-ups then abort
    # pairs in the middle of later units; the call returns, reports the
    # timeout, and the context stays usable
    L2, Hq2, Hkv2, n2, W2 = 8, 28, 4, 8192, 20
    mk = lambda shape, k: synth._round(synth.normal(4200 + k, 0, int(np.prod(shape)), "cpu").view(*shape),
                                        torch.bfloat16)
    q, k, v = mk((L2, Hq2, W2, d), 1), mk((L2, Hkv2, n2, d), 2), mk((L2, Hkv2, n2, d), 3)
    Q, K, V = q.to(DEV), k.to(DEV), v.to(DEV)
    B, Nq, _ = vc.viscache_plan_budgets(L2, n2, *RR)
    units = sum(Hkv2 * ((b + 255) // 256) for b in B if b > 0)
    assert units > 2 * (torch.cuda.get_device_properties(0).multi_processor_count // 2), units
    batch = vc.Batch([n2], [W2], [RR])
    prm = vc.make_params(L2, Hq2, Hkv2, d, vc.VC_BF16)
    ws = torch.empty(vc.prunekv_workspace_size(batch, prm), dtype=torch.uint8, device=DEV)
    for mask in (vc.VC_TEST_WAIT_FUSE,
                 vc.VC_TEST_WAIT_SCORE_LSE | vc.VC_TEST_WAIT_SCORE_COLSUM | vc.VC_TEST_WAIT_FUSE):
        inject(mask)
        t0 = time.perf_counter()
        vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
        assert vc.prunekv_get_status(ws) == vc.VC_ERR_DEVICE_TIMEOUT
        assert time.perf_counter() - t0 < ABORT_SECONDS
    inject(0)
    vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_OK
    s = vc.prunekv_score(Q, K)
    _, keep, drop = vc.prunekv_select(s, B, Nq)
    Ko, Vo = vc.prunekv_fuse_compact(K, V, B, Nq, keep, drop, 0.7, 1.0)
    torch.cuda.synchronize()
    check_request(q, k, v, B, Nq, dict(scores=s, keep=keep, drop=drop, K_out=Ko, V_out=Vo), 0.7, 1.0)
