"""GPU parity of the 4-bit quantisation of the compacted cache against the
oracle (codes and parameters bit for bit: the oracle decides each code in
float32 with the kernel's operation order; reconstructions within one
rounding of the output type)."""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import plan as oplan
from oracle import quant as oq
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _rand(shape, key, dtype, scale=1.0):
    x = synth.normal(key, 0, int(np.prod(shape)), "cpu").view(*shape) * scale
    return synth._round(x, dtype)


def check(batch, params, K, V, Bs):
    """Quantise on the GPU and compare every array with the oracle."""
    kc, vcodes, kp, vp = vc.viscache_kv4_quantize(batch, params, K.to(DEV), V.to(DEV))
    torch.cuda.synchronize()
    K32, V32 = K.float().numpy(), V.float().numpy()
    rkc, rvc, rkp, rvp = oq.quantize_cache(K32, V32, Bs, params.Hkv)
    np.testing.assert_array_equal(kc.cpu().numpy(), rkc)
    np.testing.assert_array_equal(vcodes.cpu().numpy(), rvc)
    # parameters equal as values (a zero minimum may carry either sign)
    assert (kp.cpu().numpy() == rkp).all()
    assert (vp.cpu().numpy() == rvp).all()
    # reconstruction: the oracle's float32 result rounded to the output type
    kh, vh = vc.viscache_kv4_dequantize(batch, params, kc, vcodes, kp, vp, dtype=K.dtype)
    torch.cuda.synchronize()
    ref_k = np.zeros_like(K32)
    for row0, b in oq.segments(Bs, params.Hkv):
        if b:
            c = oq.unpack(rkc[row0:row0 + b])
            c_s, c_m = oq.quantize_keys(K32[row0:row0 + b])[1:]
            ref_k[row0:row0 + b] = oq.dequantize_keys(c, c_s, c_m)
    ref_v = oq.dequantize_values(oq.unpack(rvc), rvp[..., 0], rvp[..., 1])
    rk = torch.from_numpy(ref_k).to(K.dtype)
    rv = torch.from_numpy(ref_v).to(K.dtype)
    assert torch.equal(kh.cpu(), rk) and torch.equal(vh.cpu(), rv)
    return kc, vcodes, kp, vp


@pytest.mark.parametrize("dtype,d", [(torch.bfloat16, 128), (torch.bfloat16, 64), (torch.float32, 64),
                                     (torch.float32, 128)], ids=["bf16-128", "bf16-64", "f32-64", "f32-128"])
def test_ragged_batch_matches_oracle(dtype, d):
    # three requests, L = 4 (layer 3 evicted), segments of 1..>100 rows with ragged last groups
    ns, rrs, L, Hkv = [1500, 40, 333], [(25, 100), (50, 100), (19, 100)], 4, 2
    batch = vc.Batch(ns, [8] * 3, rrs)
    params = vc.make_params(L, 4, Hkv, d, vc.VC_BF16 if dtype == torch.bfloat16 else vc.VC_F32)
    Bs = [oplan.plan_budgets(L, n, Fraction(*rr))[0] for n, rr in zip(ns, rrs)]
    rows = Hkv * sum(sum(b) for b in Bs)
    K = _rand((rows, d), 101 + d, dtype, 2.0)
    V = _rand((rows, d), 202 + d, dtype, 2.0)
    check(batch, params, K, V, Bs)


def test_outlier_channels_and_constant_groups():
    # channel 3 scaled by 100 (keys are per channel, so only its groups widen);
    # a constant value row and a constant key block give scale 0 and exact values
    L, Hkv, d, n = 2, 2, 128, 300
    batch = vc.Batch([n], [8], [(1, 1)])
    params = vc.make_params(L, 8, Hkv, d, vc.VC_BF16, h=L, m=(1, 1), schedule=vc.VC_SCHED_FIXED)
    Bs = [[n] * L]
    rows = Hkv * n * L
    K = _rand((rows, d), 303, torch.bfloat16)
    V = _rand((rows, d), 304, torch.bfloat16)
    K[:, 3] *= 100
    K[32:64] = 0.5
    V[7] = -1.25
    kc, vcodes, kp, vp = check(batch, params, K, V, Bs)
    assert (kp[1, :, 0] == 0).all().item() and (vp[7, :, 0] == 0).all().item()


def test_many_entries_split_into_launches():
    # 72 requests x 30 kept layers of 40 > the 1792 (request, layer) entries of one launch
    ns = [64 + (7 * i) % 90 for i in range(72)]
    rrs = [(25, 100)] * 72
    L, Hkv, d = 40, 1, 64
    batch = vc.Batch(ns, [8] * 72, rrs)
    params = vc.make_params(L, 2, Hkv, d, vc.VC_BF16)
    Bs = [oplan.plan_budgets(L, n, Fraction(*rr))[0] for n, rr in zip(ns, rrs)]
    assert sum(1 for B in Bs for b in B if b) > 1792
    rows = Hkv * sum(sum(b) for b in Bs)
    K = _rand((rows, d), 405, torch.bfloat16)
    V = _rand((rows, d), 406, torch.bfloat16)
    check(batch, params, K, V, Bs)


def test_quantizes_the_compressed_pass_output():
    wl = synth.scaled(synth.WORKLOADS[2], "kv4-e2e", L=4,
                      requests=[synth.Request(700, 16, 25, 100, 196), synth.Request(300, 16, 50, 100, 196)])
    qs, ks, vs = synth.generate(wl, "cpu")
    batch = vc.Batch([r.n for r in wl.requests], [r.W for r in wl.requests],
                     [(r.rr_num, r.rr_den) for r in wl.requests])
    params = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    Qw = torch.cat([x.reshape(-1, wl.d) for x in qs]).to(DEV)
    K = torch.cat([x.reshape(-1, wl.d) for x in ks]).to(DEV)
    V = torch.cat([x.reshape(-1, wl.d) for x in vs]).to(DEV)
    K_out, V_out, _ = vc.prunekv_compress(batch, params, Qw, K, V)
    Bs = [oplan.plan_budgets(wl.L, r.n, Fraction(r.rr_num, r.rr_den))[0] for r in wl.requests]
    check(batch, params, K_out.cpu(), V_out.cpu(), Bs)


def test_repeated_calls_bit_identical():
    batch = vc.Batch([2000], [8], [(19, 100)])
    params = vc.make_params(3, 8, 2, 128, vc.VC_BF16)
    rows, _ = vc.viscache_kv4_sizes(batch, params)
    K = _rand((rows, 128), 507, torch.bfloat16).to(DEV)
    V = _rand((rows, 128), 508, torch.bfloat16).to(DEV)
    a = vc.viscache_kv4_quantize(batch, params, K, V)
    for _ in range(2):
        b = vc.viscache_kv4_quantize(batch, params, K, V)
        assert all(torch.equal(x, y) for x, y in zip(a, b))
