"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the same seeded inputs."""
import numpy as np
import pytest
import torch

from oracle import plan as oplan
from oracle import prunekv as ok
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc
from tests.parity import check_request, np64

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _rand(shape, key, dtype):
    x = synth.normal(key, 0, int(np.prod(shape)), "cpu").view(*shape)
    return synth._round(x, dtype)


@pytest.fixture(params=[vc.VC_PATH_AUTO, vc.VC_PATH_SIMT], ids=["auto", "simt"])
def kernel_path(request):
    vc.viscache_set_kernel_path(request.param)
    yield request.param
    vc.viscache_set_kernel_path(vc.VC_PATH_AUTO)


def run_steps(Q, K, V, B, Nq, mu=0.7, tau=1.0, rank_mode=vc.VC_RANK_SHARED, row_lse=None):
    s = vc.prunekv_score(Q, K, rank_mode=rank_mode, row_lse=row_lse)
    rank, keep, drop = vc.prunekv_select(s, B, Nq, rank_mode)
    Ko, Vo = vc.prunekv_fuse_compact(K, V, B, Nq, keep, drop, mu, tau)
    torch.cuda.synchronize()
    return dict(scores=s, rank=rank, keep=keep, drop=drop, K_out=Ko, V_out=Vo)


SMALL = [
    # L, Hq, Hkv, d, n, W, dtype, rr
    (1, 2, 1, 64, 1, 1, torch.float32, (1, 1)),
    (2, 4, 2, 64, 63, 3, torch.bfloat16, (1, 2)),
    (3, 7, 1, 128, 129, 5, torch.bfloat16, (1, 4)),
    (4, 8, 1, 128, 1000, 64, torch.bfloat16, (19, 100)),
    (2, 8, 4, 64, 257, 32, torch.float32, (25, 100)),
    (1, 1, 1, 128, 64, 1, torch.bfloat16, (1, 1)),
    (5, 6, 2, 128, 700, 17, torch.float32, (28, 100)),
]


@pytest.mark.parametrize("case", SMALL)
def test_small_shapes_step_api(case, kernel_path):
    L, Hq, Hkv, d, n, W, dt, rr = case
    key = hash(case[:6]) & 0xFFFFFFFF
    Q = _rand((L, Hq, W, d), key + 1, dt)
    K = _rand((L, Hkv, n, d), key + 2, dt)
    V = _rand((L, Hkv, n, d), key + 3, dt)
    B, Nq, h = vc.viscache_plan_budgets(L, n, *rr)
    from fractions import Fraction
    assert (B, Nq, h) == oplan.plan_budgets(L, n, Fraction(*rr))
    out = run_steps(Q.to(DEV), K.to(DEV), V.to(DEV), B, Nq)
    log = check_request(Q, K, V, B, Nq, out, 0.7, 1.0)
    assert len(log) <= 2, log


@pytest.mark.parametrize("case", SMALL[1:5])
def test_compress_equals_step_api(case):
    L, Hq, Hkv, d, n, W, dt, rr = case
    key = hash(case[:6]) & 0xFFFFFFFF
    Q, K, V = (_rand(s, key + i, dt).to(DEV) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)], 1))
    B, Nq, h = vc.viscache_plan_budgets(L, n, *rr)
    ref = run_steps(Q, K, V, B, Nq)
    batch = vc.Batch([n], [W], [rr])
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_F32 if dt == torch.float32 else vc.VC_BF16)
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q, K, V)
    torch.cuda.synchronize()
    assert torch.equal(idx, ref["keep"]) and torch.equal(Ko, ref["K_out"]) and torch.equal(Vo, ref["V_out"])


def test_maximum_visual_tokens(kernel_path):
    # n at its limit (65,536 visual tokens): scores, ranking, both lists, K_out
    # and V_out against the oracle; the fused call equals the steps bit for bit
    L, Hq, Hkv, d, n, W, rr = 2, 4, 2, 128, 65536, 16, (1, 10)
    Q = _rand((L, Hq, W, d), 9301, torch.bfloat16)
    K = _rand((L, Hkv, n, d), 9302, torch.bfloat16)
    V = _rand((L, Hkv, n, d), 9303, torch.bfloat16)
    B, Nq, h = vc.viscache_plan_budgets(L, n, *rr)
    gpu = run_steps(Q.to(DEV), K.to(DEV), V.to(DEV), B, Nq)
    check_request(Q, K, V, B, Nq, gpu, 0.7, 1.0)
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    Ko, Vo, idx = vc.prunekv_compress(vc.Batch([n], [W], [rr]), prm, Q.to(DEV), K.to(DEV), V.to(DEV))
    torch.cuda.synchronize()
    assert torch.equal(idx, gpu["keep"]) and torch.equal(Ko, gpu["K_out"]) and torch.equal(Vo, gpu["V_out"])


def test_mu_one_is_plain_pruning_bit_exact():
    L, Hq, Hkv, d, n, W = 3, 4, 2, 128, 300, 8
    Q, K, V = (_rand(s, 700 + i, torch.bfloat16).to(DEV) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)]))
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 1, 4)
    out = run_steps(Q, K, V, B, Nq, mu=1.0)
    keep = out["keep"].long().cpu()
    P = 0
    for l in range(L):
        for g in range(Hkv):
            r0 = Hkv * P + g * B[l]
            rows = V[l, g].cpu()[keep[r0:r0 + B[l]]]
            assert torch.equal(out["V_out"][r0:r0 + B[l]].cpu(), rows)
        P += B[l]


def test_empty_drop_set_keeps_values():
    # L = 1, m = 1: Nq = B_1, nothing to fuse.
    L, Hq, Hkv, d, n, W = 1, 2, 1, 64, 200, 4
    Q, K, V = (_rand(s, 800 + i, torch.float32).to(DEV) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)]))
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 1, 4, 0, 1, 1)
    assert Nq == B[0]
    out = run_steps(Q, K, V, B, Nq)
    assert out["drop"].numel() == 0
    assert torch.equal(out["V_out"].cpu(), V[0, 0].cpu()[out["keep"].long().cpu()])


def test_zero_queries_keep_first_positions(kernel_path):
    L, Hq, Hkv, d, n, W = 2, 4, 2, 128, 500, 16
    Q = torch.zeros((L, Hq, W, d), dtype=torch.bfloat16, device=DEV)
    K, V = (_rand((L, Hkv, n, d), 900 + i, torch.bfloat16).to(DEV) for i in range(2))
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 1, 4)
    out = run_steps(Q, K, V, B, Nq)
    keep = out["keep"].cpu()
    for g in range(Hkv):
        assert keep[g * B[0]:(g + 1) * B[0]].tolist() == list(range(B[0]))
    assert torch.allclose(out["scores"].cpu(), torch.full((Hkv, n), 2.0 * W / n), rtol=1e-6)


def test_per_layer_ranking(kernel_path):
    L, Hq, Hkv, d, n, W = 3, 6, 2, 128, 333, 9
    Q, K, V = (_rand(s, 1000 + i, torch.bfloat16) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)]))
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 3, 10)
    out = run_steps(Q.to(DEV), K.to(DEV), V.to(DEV), B, Nq, rank_mode=vc.VC_RANK_PER_LAYER)
    assert out["scores"].shape == (L, Hkv, n)
    check_request(Q, K, V, B, Nq, out, 0.7, 1.0, rank_mode="per_layer")


def test_row_lse_input(kernel_path):
    L, Hq, Hkv, d, n, W = 2, 4, 2, 64, 190, 6
    Q, K, V = (_rand(s, 1100 + i, torch.float32) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)]))
    Qn, Kn = np64(Q), np64(K)
    lse = np.empty((L, Hq, W))
    for l in range(L):
        for j in range(Hq):
            x = (Qn[l, j] @ Kn[l, j // 2].T) / np.sqrt(d)
            lse[l, j] = np.log(np.exp(x).sum(axis=1)) + 0.25    # a wider softmax domain
    lse32 = torch.from_numpy(lse).float()
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 1, 4)
    out = run_steps(Q.to(DEV), K.to(DEV), V.to(DEV), B, Nq, row_lse=lse32.to(DEV))
    check_request(Q, K, V, B, Nq, out, 0.7, 1.0, row_lse=lse32.double().numpy())


def test_bad_index_sets_device_status():
    # A keep list with an out-of-range position: the kernels skip it and record
    # VC_ERR_DEVICE_INDEX; the context stays usable.
    L, Hkv, d, n = 1, 1, 64, 50
    K, V = (_rand((L, Hkv, n, d), 1200 + i, torch.float32).to(DEV) for i in range(2))
    B, Nq = [4], 6
    keep = torch.tensor([1, 2, 3, 999], dtype=torch.int32, device=DEV)
    drop = torch.tensor([5, 6], dtype=torch.int32, device=DEV)
    ws = torch.empty(vc.prunekv_fuse_workspace_size(B, Hkv, d, n, Nq), dtype=torch.uint8, device=DEV)
    vc.prunekv_fuse_compact(K, V, B, Nq, keep, drop, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_ERR_DEVICE_INDEX
    keep[3] = 4
    vc.prunekv_fuse_compact(K, V, B, Nq, keep, drop, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_OK


TC_SHAPES = [
    # L, Hq, Hkv, n, W  (bf16, d = 128: the tensor-core score path)
    (1, 1, 1, 1, 1),
    (2, 7, 1, 127, 5),
    (2, 8, 1, 129, 16),
    (1, 2, 1, 128, 64),
    (3, 14, 2, 1000, 19),     # 7*19 = 133 rows: two row blocks, ragged
    (2, 28, 4, 300, 64),      # 448 rows per group
    (1, 8, 1, 2049, 40),      # 320 rows: two 256-row blocks
    (2, 4, 4, 513, 3),        # G = 1
]


@pytest.mark.parametrize("shape", TC_SHAPES)
@pytest.mark.parametrize("mode", [vc.VC_RANK_SHARED, vc.VC_RANK_PER_LAYER], ids=["shared", "layer"])
def test_tensor_core_scores_match_oracle_and_cuda_cores(shape, mode):
    L, Hq, Hkv, n, W = shape
    d = 128
    key = 5000 + 13 * sum(shape)
    Q = _rand((L, Hq, W, d), key, torch.bfloat16)
    K = _rand((L, Hkv, n, d), key + 1, torch.bfloat16)
    Qd, Kd = Q.to(DEV), K.to(DEV)
    s_tc = vc.prunekv_score(Qd, Kd, rank_mode=mode)
    vc.viscache_set_kernel_path(vc.VC_PATH_SIMT)
    try:
        s_simt = vc.prunekv_score(Qd, Kd, rank_mode=mode)
    finally:
        vc.viscache_set_kernel_path(vc.VC_PATH_AUTO)
    torch.cuda.synchronize()
    ref = ok.token_scores(np64(Q), np64(K), rank_mode="per_layer" if mode else "shared")
    for got in (s_tc, s_simt):
        err = np.abs(np64(got) - ref) / np.maximum(np.abs(ref), 1e-30)
        assert float(err.max()) < 2e-5, float(err.max())


FUSE_CASES = [
    # n, B, D, mu, tau
    (300, 1, 1, 0.7, 1.0),
    (300, 129, 127, 0.7, 1.0),
    (600, 128, 129, 0.0, 0.5),
    (1000, 300, 500, 0.7, 4.0),
    (2000, 257, 1500, 0.3, 1.0),
    (500, 200, 0, 0.7, 1.0),
    (700, 130, 260, 1.0, 1.0),
]


@pytest.mark.parametrize("case", FUSE_CASES)
def test_tensor_core_fusion_matches_oracle(case, kernel_path):
    n, b, D, mu, tau = case
    L, Hkv, d = 1, 2, 128
    K = _rand((L, Hkv, n, d), 7000 + n + b, torch.bfloat16)
    V = _rand((L, Hkv, n, d), 7100 + n + D, torch.bfloat16)
    rng = np.random.default_rng(n * 7 + b)
    keep, drop = [], []
    for g in range(Hkv):
        perm = rng.permutation(n)
        keep.append(np.sort(perm[:b]))
        drop.append(np.sort(perm[b:b + D]))
    keep_t = torch.tensor(np.concatenate(keep), dtype=torch.int32, device=DEV)
    drop_t = torch.tensor(np.concatenate(drop), dtype=torch.int32, device=DEV)
    Ko, Vo = vc.prunekv_fuse_compact(K.to(DEV), V.to(DEV), [b], b + D, keep_t, drop_t, mu, tau)
    torch.cuda.synchronize()
    Vn = np64(V)
    got = np64(Vo)
    for g in range(Hkv):
        ref = ok.fuse_values(Vn[0, g], keep[g], drop[g], mu, tau)
        sl = got[g * b:(g + 1) * b]
        diff = np.abs(sl - ref)
        rms = float(np.sqrt((ref ** 2).mean()))
        assert float(diff.max()) <= 2e-2 * float(np.abs(ref).max())
        assert not (diff > 2e-2 * np.abs(ref) + 2e-2 * rms).any()
        if mu == 1.0 or D == 0:
            assert np.array_equal(sl, Vn[0, g][keep[g]])
        assert torch.equal(Ko[g * b:(g + 1) * b].cpu(), K[0, g][torch.from_numpy(keep[g])])


# ---------------------------------------------------------------------------
# The workloads at full size.

def _workload_inputs(wid, device="cpu"):
    wl = synth.WORKLOADS[wid]
    qs, ks, vs = synth.generate(wl, device)
    return wl, qs[0], ks[0], vs[0]


@pytest.mark.parametrize("wid", [1, 2, 3])
def test_workload_full_parity(wid, kernel_path):
    if wid == 1 and kernel_path == vc.VC_PATH_SIMT:
        pytest.skip("fp32 workload runs on CUDA cores under both settings")
    wl, Q, K, V = _workload_inputs(wid)
    req = wl.requests[0]
    B, Nq, h = vc.viscache_plan_budgets(wl.L, req.n, req.rr_num, req.rr_den)
    out = run_steps(Q.to(DEV), K.to(DEV), V.to(DEV), B, Nq)
    log = check_request(Q, K, V, B, Nq, out, 0.7, 1.0)
    print("workload %d near-tie swaps: %s" % (wid, log))
    # the fused entry point gives the same bits
    batch = vc.Batch([req.n], [req.W], [(req.rr_num, req.rr_den)])
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_F32 if wl.dtype == "f32" else vc.VC_BF16)
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q.to(DEV), K.to(DEV), V.to(DEV))
    torch.cuda.synchronize()
    assert torch.equal(idx, out["keep"]) and torch.equal(Ko, out["K_out"]) and torch.equal(Vo, out["V_out"])


def test_values_in_host_memory(kernel_path):
    # V may stay in pinned host memory the device can read: same bits as from HBM
    L, Hq, Hkv, d, n, W = 4, 8, 2, 128, 1000, 32
    Q = _rand((L, Hq, W, d), 9101, torch.bfloat16).to(DEV)
    K = _rand((L, Hkv, n, d), 9102, torch.bfloat16).to(DEV)
    V = _rand((L, Hkv, n, d), 9103, torch.bfloat16)
    hV = V.pin_memory()
    if not vc.viscache_device_accessible(hV):
        pytest.skip("pinned host memory is not mapped into the device's address space here")
    assert vc.viscache_device_accessible(K)
    batch = vc.Batch([n], [W], [(19, 100)])
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    Ko1, Vo1, i1 = vc.prunekv_compress(batch, prm, Q, K, V.to(DEV))
    Ko2, Vo2, i2 = vc.prunekv_compress(batch, prm, Q, K, hV)
    torch.cuda.synchronize()
    assert torch.equal(i1, i2) and torch.equal(Ko1, Ko2) and torch.equal(Vo1, Vo2)


def test_keys_and_values_in_host_memory(kernel_path):
    # the fusion step with K and V in pinned host memory: the kept keys are then
    # copied by the gather (the tensor-core fusion copies them itself only from
    # device memory); same bits as from HBM
    L, Hq, Hkv, d, n, W = 3, 8, 2, 128, 1500, 16
    Q = _rand((L, Hq, W, d), 9201, torch.bfloat16).to(DEV)
    K = _rand((L, Hkv, n, d), 9202, torch.bfloat16)
    V = _rand((L, Hkv, n, d), 9203, torch.bfloat16)
    hK, hV = K.pin_memory(), V.pin_memory()
    if not (vc.viscache_device_accessible(hK) and vc.viscache_device_accessible(hV)):
        pytest.skip("pinned host memory is not mapped into the device's address space here")
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 23, 100)
    s = vc.prunekv_score(Q, K.to(DEV))
    _, keep, drop = vc.prunekv_select(s, B, Nq)
    Ko1, Vo1 = vc.prunekv_fuse_compact(K.to(DEV), V.to(DEV), B, Nq, keep, drop, 0.7, 1.0)
    # outputs and workspace on the device (the binding would put them beside K)
    Ko2 = torch.empty_like(Ko1)
    Vo2 = torch.empty_like(Vo1)
    ws = torch.empty(vc.prunekv_fuse_workspace_size(B, Hkv, d, n, Nq), dtype=torch.uint8, device=DEV)
    vc.prunekv_fuse_compact(hK, hV, B, Nq, keep, drop, 0.7, 1.0, K_out=Ko2, V_out=Vo2, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_OK
    torch.cuda.synchronize()
    assert torch.equal(Ko1, Ko2) and torch.equal(Vo1, Vo2)


def test_generator_same_bits_on_device():
    wl = synth.scaled(synth.WORKLOADS[3], "slice", L=2)
    q_cpu = synth.make_q(wl, 0, "cpu")
    q_dev = synth.make_q(wl, 0, DEV)
    assert torch.equal(q_cpu, q_dev.cpu())
    k_cpu, v_cpu = synth.make_kv(wl, 0, q_cpu, "cpu", layers=[1])
    k_dev, v_dev = synth.make_kv(wl, 0, q_cpu, DEV, layers=[1])
    assert torch.equal(k_cpu[1], k_dev[1].cpu()) and torch.equal(v_cpu[1], v_dev[1].cpu())


@pytest.mark.parametrize("n", [1, 31, 1023, 1025, 16384, 32768, 65535, 65536])
@pytest.mark.parametrize("mode", [vc.VC_RANK_SHARED, vc.VC_RANK_PER_LAYER], ids=["shared", "layer"])
def test_select_matches_oracle_ranking(n, mode):
    # chunked ranking (1024-key chunks, full and ragged last chunk); exact ties
    # (scores drawn from a small set) must go to the lower index.
    L, Hkv = 3, 2
    rng = np.random.default_rng(n + 7 * mode)
    shape = (Hkv, n) if mode == vc.VC_RANK_SHARED else (L, Hkv, n)
    s = rng.integers(0, max(2, n // 3), size=shape).astype(np.float32) / 7.0
    B, Nq, _ = vc.viscache_plan_budgets(L, n, 1, 3)
    rank, keep, drop = vc.prunekv_select(torch.from_numpy(s).to(DEV), B, Nq, mode)
    torch.cuda.synchronize()
    keep_ref, drop_ref, rank_ref = ok.select(s.astype(np.float64), B, Nq,
                                             "per_layer" if mode else "shared")
    assert np.array_equal(rank.cpu().numpy(), rank_ref)
    keep, drop = keep.cpu().numpy(), drop.cpu().numpy()
    P = Qd = 0
    for l in range(L):
        D = Nq - B[l] if B[l] > 0 else 0
        for g in range(Hkv):
            assert np.array_equal(keep[Hkv * P + g * B[l]:Hkv * P + (g + 1) * B[l]], keep_ref[l][g])
            assert np.array_equal(drop[Hkv * Qd + g * D:Hkv * Qd + (g + 1) * D], drop_ref[l][g])
        P += B[l]
        Qd += D


SCHEDULES = [(vc.VC_SCHED_PARABOLA, "parabola"), (vc.VC_SCHED_FIXED, "fixed"),
             (vc.VC_SCHED_ARITHMETIC, "arithmetic"), (vc.VC_SCHED_GEOMETRIC, "geometric")]


@pytest.mark.parametrize("drop_code,drop", [(vc.VC_DROP_SURVIVORS, "survivors"), (vc.VC_DROP_ALL, "all")],
                         ids=["survivors", "drop_all"])
@pytest.mark.parametrize("code,name", SCHEDULES, ids=[s for _, s in SCHEDULES])
def test_budget_schedules_match_oracle(code, name, drop_code, drop, kernel_path):
    """The ablation schedules and the drop-all reading: same kernels, other plans."""
    from fractions import Fraction
    L, Hq, Hkv, d, n, W, rr = 6, 8, 2, 128, 1000, 16, (28, 100)
    Q, K, V = (_rand(s, 900 + i, torch.bfloat16) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)], 1))
    B, Nq, h = vc.viscache_plan_budgets_ex(L, n, *rr, 0, 3, 4, code, drop_code)
    assert (B, Nq, h) == oplan.plan_budgets(L, n, Fraction(*rr), schedule=name, drop=drop)
    out = run_steps(Q.to(DEV), K.to(DEV), V.to(DEV), B, Nq)
    log = check_request(Q, K, V, B, Nq, out, 0.7, 1.0)
    assert len(log) <= 2, log
    # the fused entry point with the same plan choices
    batch = vc.Batch([n], [W], [rr])
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16, schedule=code, drop_mode=drop_code)
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q.to(DEV), K.to(DEV), V.to(DEV))
    torch.cuda.synchronize()
    assert torch.equal(idx, out["keep"]) and torch.equal(Ko, out["K_out"])
    assert torch.equal(Vo, out["V_out"])


def test_compress_per_layer_equals_step_api(kernel_path):
    """Per-layer ranking in the fused pass (which scores and ranks only the
    layers the budgets keep) gives the step API's result bit for bit."""
    L, Hq, Hkv, d, n, W, rr = 6, 8, 2, 128, 1500, 16, (28, 100)
    Q, K, V = (_rand(s, 950 + i, torch.bfloat16).to(DEV) for i, s in
               enumerate([(L, Hq, W, d), (L, Hkv, n, d), (L, Hkv, n, d)], 1))
    B, Nq, h = vc.viscache_plan_budgets(L, n, *rr)
    assert B[-1] == 0                                    # an evicted layer
    ref = run_steps(Q, K, V, B, Nq, rank_mode=vc.VC_RANK_PER_LAYER)
    batch = vc.Batch([n], [W], [rr])
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16, rank_mode=vc.VC_RANK_PER_LAYER)
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q, K, V)
    torch.cuda.synchronize()
    assert torch.equal(idx, ref["keep"]) and torch.equal(Ko, ref["K_out"])
    assert torch.equal(Vo, ref["V_out"])


def test_batch_with_tables_beyond_the_parameter_image(kernel_path):
    """40 requests of 28 layers: every (request, layer) adds at least 36 bytes of
    plan tables, so the image (> 40 KB) no longer travels as the upload kernel's
    24 KB parameter; the call copies it with a memcpy and then clears the status
    word with an upload of no bytes, and the kernels after it are ordered behind
    that.  The batch equals every request compressed alone, bit for bit, and
    three requests match the oracle."""
    L, Hq, Hkv, d, nreq = 28, 8, 2, 128, 40
    rng = np.random.default_rng(2608)
    ns = [int(x) for x in rng.integers(200, 700, nreq)]
    Ws = [int(x) for x in rng.integers(4, 17, nreq)]
    rrs = [[(19, 100), (23, 100), (28, 100)][i % 3] for i in range(nreq)]
    qs = [_rand((L, Hq, Ws[i], d), 7100 + 3 * i, torch.bfloat16) for i in range(nreq)]
    ks = [_rand((L, Hkv, ns[i], d), 7101 + 3 * i, torch.bfloat16) for i in range(nreq)]
    vs = [_rand((L, Hkv, ns[i], d), 7102 + 3 * i, torch.bfloat16) for i in range(nreq)]
    Q = torch.cat([q.flatten() for q in qs]).to(DEV)
    K = torch.cat([k.flatten() for k in ks]).to(DEV)
    V = torch.cat([v.flatten() for v in vs]).to(DEV)
    batch = vc.Batch(ns, Ws, rrs)
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    ws = torch.empty(vc.prunekv_workspace_size(batch, prm), dtype=torch.uint8, device=DEV)
    ws.fill_(0xff)                       # a stale status word must be cleared by the call
    Ko, Vo, idx = vc.prunekv_compress(batch, prm, Q, K, V, ws=ws)
    assert vc.prunekv_get_status(ws) == vc.VC_OK
    off = 0
    for i in range(nreq):
        one = vc.Batch([ns[i]], [Ws[i]], [rrs[i]])
        rows = vc.compressed_rows(one, prm)
        ko, vo, ix = vc.prunekv_compress(one, prm, qs[i].to(DEV), ks[i].to(DEV), vs[i].to(DEV))
        torch.cuda.synchronize()
        assert torch.equal(idx[off:off + rows], ix), "request %d idx" % i
        assert torch.equal(Ko[off:off + rows], ko), "request %d K_out" % i
        assert torch.equal(Vo[off:off + rows], vo), "request %d V_out" % i
        if i in (0, nreq // 2, nreq - 1):
            B, Nq, _ = vc.viscache_plan_budgets(L, ns[i], *rrs[i])
            out = run_steps(qs[i].to(DEV), ks[i].to(DEV), vs[i].to(DEV), B, Nq)
            assert torch.equal(out["keep"], ix) and torch.equal(out["K_out"], ko)
            log = check_request(qs[i], ks[i], vs[i], B, Nq, out, 0.7, 1.0)
            assert len(log) <= 2, log
        off += rows
    assert off == Ko.shape[0]


@pytest.mark.parametrize("rise", [40.0, 300.0])
def test_fusion_rescale_after_a_large_rise(rise):
    """A dropped row in the fifth tile whose logit with kept row 5 exceeds that
    row's maximum over the first four tiles by `rise` (log2 units, above the
    fusion's 2^32 threshold) makes the softmax rescale the row's O and row sum;
    without the rescale the earlier tiles' terms would outweigh it by 2^rise.
    V_out of every kept row matches the oracle's fusion; K_out is exact."""
    from oracle import prunekv as okp
    from tests.parity import TOL, check_v_rows
    L, Hkv, d, n, tau, mu = 1, 1, 128, 1200, 1.0, 0.3
    B, Nq = [256], 1000                                   # 744 dropped rows: 6 tiles of 128
    K = _rand((L, Hkv, n, d), 9101, torch.bfloat16)
    V = _rand((L, Hkv, n, d), 9102, torch.bfloat16)
    keep = np.arange(0, 256)
    drop = np.arange(256, Nq)
    r0, j_plant = 5, 256 + 4 * 128 + 17                   # kept row, planted token (tile 4)
    v = V[0, 0].double().numpy()
    m_prev = float((v[drop[:512]] @ v[r0]).max()) / tau * np.log2(np.e)
    alpha = (m_prev + rise) * tau / (float(v[r0] @ v[r0]) * np.log2(np.e))
    V[0, 0, j_plant] = (alpha * V[0, 0, r0].double()).to(torch.bfloat16)
    v = V[0, 0].double().numpy()
    got_rise = float(v[j_plant] @ v[r0]) / tau * np.log2(np.e) - m_prev
    assert got_rise > 35.0, got_rise
    ki = torch.tensor(keep, dtype=torch.int32, device=DEV)
    di = torch.tensor(drop, dtype=torch.int32, device=DEV)
    Ko, Vo = vc.prunekv_fuse_compact(K.to(DEV), V.to(DEV), B, Nq, ki, di, mu, tau)
    torch.cuda.synchronize()
    assert torch.equal(Ko.cpu(), K[0, 0][torch.from_numpy(keep)])
    ref = okp.fuse_values(v, keep, drop, mu, tau)
    check_v_rows(np64(Vo), ref, TOL[torch.bfloat16], "rise %g" % rise)
    # the planted row dominates kept row 5's fused value
    assert np.allclose(ref[r0], mu * v[r0] + (1 - mu) * v[j_plant], rtol=1e-6, atol=1e-6 * np.abs(v[j_plant]).max())


def test_concurrent_calls_on_two_streams():
    """Calls on two streams with their own workspaces run at the same time (their
    kernels are dependent launches within each stream, not across streams) and
    give, bit for bit, what the same calls give one after the other; repeated
    three times so the two streams' kernels interleave differently."""
    wl = synth.scaled(synth.WORKLOADS[3], "7B shape, 8 layers, 4000 tokens", L=8,
                      requests=[synth.Request(4000, 64, 19, 100, 100)])
    wl2 = synth.scaled(synth.WORKLOADS[3], "7B shape, 8 layers, 2500 tokens", L=8,
                       requests=[synth.Request(2500, 48, 28, 100, 101)])
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    inputs = []
    for w in (wl, wl2):
        q = synth.make_q(w, 0)
        k, v = synth.make_kv(w, 0, q)
        r = w.requests[0]
        batch = vc.Batch([r.n], [r.W], [(r.rr_num, r.rr_den)])
        inputs.append((batch, q.to(DEV), k.to(DEV), v.to(DEV)))
    ref = []
    for batch, Q, K, V in inputs:
        ref.append(vc.prunekv_compress(batch, prm, Q, K, V))
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    wss = [torch.empty(vc.prunekv_workspace_size(b, prm), dtype=torch.uint8, device=DEV) for b, _, _, _ in inputs]
    for rep in range(3):
        outs = [None, None]
        torch.cuda.synchronize()
        for i in (0, 1) if rep % 2 == 0 else (1, 0):
            batch, Q, K, V = inputs[i]
            with torch.cuda.stream(streams[i]):
                outs[i] = vc.prunekv_compress(batch, prm, Q, K, V, ws=wss[i], stream=streams[i])
        torch.cuda.synchronize()
        for i in (0, 1):
            assert vc.prunekv_get_status(wss[i]) == vc.VC_OK
            for a, b in zip(outs[i], ref[i]):
                assert torch.equal(a, b), "rep %d stream %d" % (rep, i)


@pytest.fixture
def dependent_launch():
    yield vc.viscache_set_dependent_launch
    vc.viscache_set_dependent_launch(True)


@pytest.mark.parametrize("wid", [3, 5])
def test_dependent_launches_give_the_same_bits(wid, dependent_launch):
    """The whole pass (and the step API) with the kernels of a call launched as
    dependent launches and as ordinary launches: equal bit for bit (workload 3,
    the 7B shape at 12,544 tokens, and the ragged 8-request batch)."""
    wl = synth.WORKLOADS[wid]
    qs, ks, vs = synth.generate(wl, DEV)
    Q = torch.cat([q.flatten() for q in qs])
    K = torch.cat([k.flatten() for k in ks])
    V = torch.cat([v.flatten() for v in vs])
    batch = vc.Batch([r.n for r in wl.requests], [r.W for r in wl.requests],
                     [(r.rr_num, r.rr_den) for r in wl.requests])
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    outs = {}
    for on in (True, False, True):
        dependent_launch(on)
        res = vc.prunekv_compress(batch, prm, Q, K, V)
        s = vc.prunekv_score(qs[0], ks[0])
        torch.cuda.synchronize()
        outs.setdefault(on, []).append(tuple(t.clone() for t in res) + (s.clone(),))
    ref = outs[True][0]
    for got in outs[True][1:] + outs[False]:
        for a, b in zip(got, ref):
            assert torch.equal(a, b)
