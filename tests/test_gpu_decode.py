"""GPU parity of decode attention over the compressed cache (Sec. 2 decoding
after the Sec. 3.2 compression) against the fp64 oracle.

The cache rows are seeded synthetic values laid out as the compressed pass
leaves them; the test finds each request's and layer's rows from the oracle
planner's budgets, independently of the library's table code."""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import decode as odec
from oracle import plan as oplan
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
SCHED = {vc.VC_SCHED_PARABOLA: "parabola", vc.VC_SCHED_FIXED: "fixed"}


def _rand(shape, key, dtype):
    x = synth.normal(key, 0, int(np.prod(shape)), "cpu").view(*shape)
    return synth._round(x, dtype)


def budgets(L, n, rr, schedule=vc.VC_SCHED_PARABOLA, h=None, m=Fraction(3, 4)):
    return oplan.plan_budgets(L, n, Fraction(*rr), h=h, m=m, schedule=SCHED[schedule])[0]


def tolerance(dtype, ref, vmax):
    # fp32 logits and sums: relative error of the weights ~1e-6 per term;
    # 1e-4 * max|V| bounds the accumulated effect with margin.  A bf16 output
    # adds one rounding: half an ulp, 2^-9 relative.
    base = 1e-4 * vmax
    return base + (2.0 ** -8) * np.abs(ref) if dtype == torch.bfloat16 else base + 1e-6 * np.abs(ref)


def run_case(L, Hq, Hkv, d, dtype, ns, rrs, texts, schedule=vc.VC_SCHED_PARABOLA, h=0,
             m=(3, 4), seed=1, layers=None, scale=0.0):
    code = vc.VC_BF16 if dtype == torch.bfloat16 else vc.VC_F32
    batch = vc.Batch(ns, [8] * len(ns), rrs)
    params = vc.make_params(L, Hq, Hkv, d, code, h=h, m=m, schedule=schedule, scale=scale)
    Bs = [budgets(L, n, rr, schedule, h or None, Fraction(*m)) for n, rr in zip(ns, rrs)]
    rows = sum(Hkv * sum(B) for B in Bs)
    K = _rand((max(rows, 1), d), synth.stream_key(seed, 1), dtype)
    V = _rand((max(rows, 1), d), synth.stream_key(seed, 2), dtype)
    trows = sum(Hkv * t for t in texts)
    Kt = _rand((max(trows, 1), d), synth.stream_key(seed, 3), dtype)
    Vt = _rand((max(trows, 1), d), synth.stream_key(seed, 4), dtype)
    Kd, Vd, Ktd, Vtd = (x.to(DEV) for x in (K, V, Kt, Vt))
    K64, V64, Kt64, Vt64 = (x.double().numpy() for x in (K, V, Kt, Vt))
    sc = scale if scale > 0 else 1.0 / np.sqrt(d)
    for l in (range(L) if layers is None else layers):
        q = _rand((len(ns), Hq, d), synth.stream_key(seed, 10 + l), dtype)
        out = vc.viscache_decode_attention(batch, params, l, q.to(DEV), Kd, Vd, Ktd, Vtd, texts)
        got = out.float().cpu().numpy()
        r0, t0 = 0, 0
        for r, B in enumerate(Bs):
            v0 = r0 + Hkv * sum(B[:l])
            Kv = K64[v0:v0 + Hkv * B[l]].reshape(Hkv, B[l], d)
            Vv = V64[v0:v0 + Hkv * B[l]].reshape(Hkv, B[l], d)
            T = texts[r]
            Ktr = Kt64[t0:t0 + Hkv * T].reshape(Hkv, T, d)
            Vtr = Vt64[t0:t0 + Hkv * T].reshape(Hkv, T, d)
            ref = odec.decode_attention(q[r].double().numpy(), Kv, Vv, Ktr, Vtr, scale=sc)
            vmax = max(np.abs(Vv).max(initial=0.0), np.abs(Vtr).max(initial=0.0), 1.0)
            err = np.abs(got[r] - ref)
            tol = tolerance(dtype, ref, vmax)
            assert (err <= tol).all(), "layer %d request %d: max err %.3g" % (l, r, err.max())
            if B[l] + T == 0:
                assert not got[r].any()
            r0 += Hkv * sum(B)
            t0 += Hkv * T


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32], ids=["bf16", "f32"])
@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("Hq,Hkv", [(4, 4), (28, 4), (16, 2)])
def test_ragged_batch_matches_oracle(dtype, d, Hq, Hkv):
    # three requests: two 512-key splits with the visual/text boundary inside
    # the second (request 0) or the first (request 2), a small request with
    # no text, and an evicted last layer (B = 0): text only, or no keys at all
    run_case(4, Hq, Hkv, d, dtype, ns=[1500, 40, 333], rrs=[(25, 100), (50, 100), (19, 100)],
             texts=[37, 0, 700], seed=Hq * 131 + d)


def test_text_only_and_empty_requests():
    # layer 3 of L = 4 is evicted (h = 3): text only, or no keys at all -> zeros
    run_case(4, 8, 2, 128, torch.bfloat16, ns=[600, 600], rrs=[(25, 100), (25, 100)],
             texts=[513, 0], layers=[3], seed=7)


def test_no_text_pointer():
    code = vc.VC_BF16
    batch = vc.Batch([700], [8], [(25, 100)])
    params = vc.make_params(2, 8, 2, 128, code)
    B = budgets(2, 700, (25, 100))
    rows = 2 * sum(B)
    K = _rand((rows, 128), 11, torch.bfloat16)
    V = _rand((rows, 128), 12, torch.bfloat16)
    q = _rand((1, 8, 128), 13, torch.bfloat16)
    out = vc.viscache_decode_attention(batch, params, 0, q.to(DEV), K.to(DEV), V.to(DEV))
    ref = odec.decode_attention(q[0].double().numpy(), K[:2 * B[0]].double().numpy().reshape(2, B[0], 128),
                                V[:2 * B[0]].double().numpy().reshape(2, B[0], 128))
    err = np.abs(out[0].float().cpu().numpy() - ref)
    assert (err <= tolerance(torch.bfloat16, ref, float(V.abs().max()))).all()


def test_full_cache_layout_is_the_uncompressed_cache():
    # with every B_l = n (fixed schedule, RR = 1, h = L, m = 1) the compressed
    # layout is the input cache [L][Hkv][n][d]: decoding it is plain attention
    # over all n visual rows of the layer
    L, Hkv, G, d, n = 3, 2, 4, 128, 900
    assert budgets(L, n, (1, 1), vc.VC_SCHED_FIXED, h=L, m=Fraction(1)) == [n] * L
    K = _rand((L, Hkv, n, d), 21, torch.bfloat16)
    V = _rand((L, Hkv, n, d), 22, torch.bfloat16)
    batch = vc.Batch([n], [8], [(1, 1)])
    params = vc.make_params(L, G * Hkv, Hkv, d, vc.VC_BF16, h=L, m=(1, 1), schedule=vc.VC_SCHED_FIXED)
    Kd, Vd = K.reshape(-1, d).to(DEV), V.reshape(-1, d).to(DEV)
    for l in range(L):
        q = _rand((1, G * Hkv, d), 30 + l, torch.bfloat16)
        out = vc.viscache_decode_attention(batch, params, l, q.to(DEV), Kd, Vd)
        ref = odec.decode_attention(q[0].double().numpy(), K[l].double().numpy(), V[l].double().numpy())
        err = np.abs(out[0].float().cpu().numpy() - ref)
        assert (err <= tolerance(torch.bfloat16, ref, float(V.abs().max()))).all()


def test_decodes_the_compressed_pass_output():
    # the pass's own outputs feed the decode step unchanged
    wl = synth.scaled(synth.WORKLOADS[2], "decode-e2e", L=4,
                      requests=[synth.Request(700, 16, 25, 100, 196), synth.Request(300, 16, 50, 100, 196)])
    qs, ks, vs = synth.generate(wl, "cpu")
    batch = vc.Batch([r.n for r in wl.requests], [r.W for r in wl.requests],
                     [(r.rr_num, r.rr_den) for r in wl.requests])
    params = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16)
    Qw = torch.cat([x.reshape(-1, wl.d) for x in qs]).to(DEV)
    K = torch.cat([x.reshape(-1, wl.d) for x in ks]).to(DEV)
    V = torch.cat([x.reshape(-1, wl.d) for x in vs]).to(DEV)
    K_out, V_out, _ = vc.prunekv_compress(batch, params, Qw, K, V)
    Bs = [budgets(wl.L, r.n, (r.rr_num, r.rr_den)) for r in wl.requests]
    Kc, Vc = K_out.double().cpu().numpy(), V_out.double().cpu().numpy()
    for l in range(wl.L):
        q = _rand((2, wl.Hq, wl.d), 40 + l, torch.bfloat16)
        out = vc.viscache_decode_attention(batch, params, l, q.to(DEV), K_out, V_out).float().cpu().numpy()
        r0 = 0
        for r, B in enumerate(Bs):
            v0 = r0 + wl.Hkv * sum(B[:l])
            Kv = Kc[v0:v0 + wl.Hkv * B[l]].reshape(wl.Hkv, B[l], wl.d)
            Vv = Vc[v0:v0 + wl.Hkv * B[l]].reshape(wl.Hkv, B[l], wl.d)
            ref = odec.decode_attention(q[r].double().numpy(), Kv, Vv)
            err = np.abs(out[r] - ref)
            assert (err <= tolerance(torch.bfloat16, ref, max(np.abs(Vv).max(initial=0.0), 1.0))).all()
            r0 += wl.Hkv * sum(B)


def test_repeated_calls_bit_identical():
    batch = vc.Batch([2000, 900], [8, 8], [(19, 100), (28, 100)])
    params = vc.make_params(2, 28, 4, 128, vc.VC_BF16)
    rows = vc.compressed_rows(batch, params)
    K = _rand((rows, 128), 51, torch.bfloat16).to(DEV)
    V = _rand((rows, 128), 52, torch.bfloat16).to(DEV)
    Kt = _rand((4 * 300, 128), 53, torch.bfloat16).to(DEV)
    Vt = _rand((4 * 300, 128), 54, torch.bfloat16).to(DEV)
    q = _rand((2, 28, 128), 55, torch.bfloat16).to(DEV)
    a = vc.viscache_decode_attention(batch, params, 0, q, K, V, Kt, Vt, [150, 150])
    for _ in range(3):
        b = vc.viscache_decode_attention(batch, params, 0, q, K, V, Kt, Vt, [150, 150])
        assert torch.equal(a, b)


def test_rejects_bad_arguments():
    batch = vc.Batch([100], [8], [(25, 100)])
    q = torch.zeros((1, 8, 128), dtype=torch.bfloat16, device=DEV)
    K = torch.zeros((1000, 128), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(vc.VisCacheError):
        vc.viscache_decode_attention(batch, vc.make_params(2, 8, 2, 128, vc.VC_BF16), 2, q, K, K)
    with pytest.raises(vc.VisCacheError):       # 16 query heads per KV head
        vc.viscache_decode_attention(batch, vc.make_params(2, 16, 1, 128, vc.VC_BF16), 0,
                                     torch.zeros((1, 16, 128), dtype=torch.bfloat16, device=DEV), K, K)
    with pytest.raises(vc.VisCacheError):       # text lengths without text rows
        vc.viscache_decode_attention(batch, vc.make_params(2, 8, 2, 128, vc.VC_BF16), 0, q, K, K,
                                     n_text=[3])


def test_many_splits_merge():
    # 9000 + 300 keys per KV head: more than 32 splits of the tensor-core
    # path, so the merge takes its split states 32 at a time
    L, Hkv, G, d, n, T = 2, 2, 7, 128, 9000, 300
    K = _rand((L, Hkv, n, d), 61, torch.bfloat16)
    V = _rand((L, Hkv, n, d), 62, torch.bfloat16)
    Kt = _rand((Hkv * T, d), 63, torch.bfloat16)
    Vt = _rand((Hkv * T, d), 64, torch.bfloat16)
    batch = vc.Batch([n], [8], [(1, 1)])
    params = vc.make_params(L, G * Hkv, Hkv, d, vc.VC_BF16, h=L, m=(1, 1), schedule=vc.VC_SCHED_FIXED)
    q = _rand((1, G * Hkv, d), 65, torch.bfloat16)
    out = vc.viscache_decode_attention(batch, params, 1, q.to(DEV), K.reshape(-1, d).to(DEV),
                                       V.reshape(-1, d).to(DEV), Kt.to(DEV), Vt.to(DEV), [T])
    ref = odec.decode_attention(q[0].double().numpy(), K[1].double().numpy(), V[1].double().numpy(),
                                Kt.double().numpy().reshape(Hkv, T, d), Vt.double().numpy().reshape(Hkv, T, d))
    err = np.abs(out[0].float().cpu().numpy() - ref)
    assert (err <= tolerance(torch.bfloat16, ref, float(V.abs().max()))).all()


def _oracle_reconstruction(K, V, Bs, Hkv):
    """The oracle's 4-bit reconstruction of a compacted cache, rounded to bf16."""
    from oracle import quant as oq
    K32, V32 = K.float().numpy(), V.float().numpy()
    kc, vcodes, kp, vp = oq.quantize_cache(K32, V32, Bs, Hkv)
    Kh = np.zeros_like(K32)
    for row0, b in oq.segments(Bs, Hkv):
        if b:
            c, s, m = oq.quantize_keys(K32[row0:row0 + b])
            Kh[row0:row0 + b] = oq.dequantize_keys(c, s, m)
    Vh = oq.dequantize_values(oq.unpack(vcodes), vp[..., 0], vp[..., 1])
    return torch.from_numpy(Kh).to(torch.bfloat16), torch.from_numpy(Vh).to(torch.bfloat16)


@pytest.mark.parametrize("d", [128, 64])
def test_decode_over_4bit_cache_matches_oracle(d):
    # the ragged batch of the bf16 test, its visual rows in 4-bit form
    ns, rrs, texts, L, Hkv, Hq = [1500, 40, 333], [(25, 100), (50, 100), (19, 100)], [37, 0, 700], 4, 4, 28
    batch = vc.Batch(ns, [8] * 3, rrs)
    params = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    Bs = [budgets(L, n, rr) for n, rr in zip(ns, rrs)]
    rows = sum(Hkv * sum(B) for B in Bs)
    K = _rand((rows, d), 71, torch.bfloat16)
    V = _rand((rows, d), 72, torch.bfloat16)
    trows = sum(Hkv * t for t in texts)
    Kt = _rand((trows, d), 73, torch.bfloat16)
    Vt = _rand((trows, d), 74, torch.bfloat16)
    kv4 = vc.viscache_kv4_quantize(batch, params, K.to(DEV), V.to(DEV))
    Kh, Vh = _oracle_reconstruction(K, V, Bs, Hkv)
    Kh64, Vh64 = Kh.double().numpy(), Vh.double().numpy()
    Kt64, Vt64 = Kt.double().numpy(), Vt.double().numpy()
    Ktd, Vtd = Kt.to(DEV), Vt.to(DEV)
    gKh, gVh = vc.viscache_kv4_dequantize(batch, params, *kv4)
    for l in range(L):
        q = _rand((3, Hq, d), 80 + l, torch.bfloat16)
        out = vc.viscache_decode_attention_kv4(batch, params, l, q.to(DEV), kv4, Ktd, Vtd, texts)
        # same rows in bf16 through the bf16 kernel: identical arithmetic
        ref_gpu = vc.viscache_decode_attention(batch, params, l, q.to(DEV), gKh, gVh, Ktd, Vtd, texts)
        assert torch.equal(out, ref_gpu)
        got = out.float().cpu().numpy()
        r0, t0 = 0, 0
        for r, B in enumerate(Bs):
            v0 = r0 + Hkv * sum(B[:l])
            Kv = Kh64[v0:v0 + Hkv * B[l]].reshape(Hkv, B[l], d)
            Vv = Vh64[v0:v0 + Hkv * B[l]].reshape(Hkv, B[l], d)
            T = texts[r]
            Ktr = Kt64[t0:t0 + Hkv * T].reshape(Hkv, T, d)
            Vtr = Vt64[t0:t0 + Hkv * T].reshape(Hkv, T, d)
            ref = odec.decode_attention(q[r].double().numpy(), Kv, Vv, Ktr, Vtr)
            vmax = max(np.abs(Vv).max(initial=0.0), np.abs(Vtr).max(initial=0.0), 1.0)
            err = np.abs(got[r] - ref)
            assert (err <= tolerance(torch.bfloat16, ref, vmax)).all(), "layer %d request %d" % (l, r)
            r0 += Hkv * sum(B)
            t0 += Hkv * T


def test_decode_over_4bit_cache_rejects_fp32():
    batch = vc.Batch([100], [8], [(25, 100)])
    params = vc.make_params(2, 8, 2, 64, vc.VC_F32)
    z = torch.zeros(4096, dtype=torch.uint8, device=DEV)
    zf = torch.zeros(4096, dtype=torch.float32, device=DEV)
    with pytest.raises(vc.VisCacheError):
        vc.viscache_decode_attention_kv4(batch, params, 0, torch.zeros((1, 8, 64), device=DEV), (z, z, zf, zf))


def test_full_table_of_256_requests():
    # the decode table's limit: 256 requests, mixed budgets, text lengths
    # (some zero) and an evicted layer; also through the 4-bit path
    n_req, L, Hkv, Hq, d = 256, 4, 2, 8, 64
    ns = [24 + (37 * i) % 200 for i in range(n_req)]
    rrs = [(25 + (i % 3) * 10, 100) for i in range(n_req)]
    texts = [(11 * i) % 40 if i % 5 else 0 for i in range(n_req)]
    batch = vc.Batch(ns, [8] * n_req, rrs)
    params = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    Bs = [budgets(L, n, rr) for n, rr in zip(ns, rrs)]
    rows = sum(Hkv * sum(B) for B in Bs)
    K = _rand((rows, d), 91, torch.bfloat16)
    V = _rand((rows, d), 92, torch.bfloat16)
    trows = sum(Hkv * t for t in texts)
    Kt = _rand((trows, d), 93, torch.bfloat16)
    Vt = _rand((trows, d), 94, torch.bfloat16)
    Kd, Vd, Ktd, Vtd = (x.to(DEV) for x in (K, V, Kt, Vt))
    kv4 = vc.viscache_kv4_quantize(batch, params, Kd, Vd)
    Kh, Vh = vc.viscache_kv4_dequantize(batch, params, *kv4)
    K64, V64, Kt64, Vt64 = (x.double().numpy() for x in (K, V, Kt, Vt))
    for l in (0, L - 1):
        q = _rand((n_req, Hq, d), 95 + l, torch.bfloat16)
        out = vc.viscache_decode_attention(batch, params, l, q.to(DEV), Kd, Vd, Ktd, Vtd, texts)
        out4 = vc.viscache_decode_attention_kv4(batch, params, l, q.to(DEV), kv4, Ktd, Vtd, texts)
        assert torch.equal(out4, vc.viscache_decode_attention(batch, params, l, q.to(DEV), Kh, Vh, Ktd, Vtd, texts))
        got = out.float().cpu().numpy()
        r0, t0 = 0, 0
        for r, B in enumerate(Bs):
            v0 = r0 + Hkv * sum(B[:l])
            Kv = K64[v0:v0 + Hkv * B[l]].reshape(Hkv, B[l], d)
            Vv = V64[v0:v0 + Hkv * B[l]].reshape(Hkv, B[l], d)
            T = texts[r]
            Ktr = Kt64[t0:t0 + Hkv * T].reshape(Hkv, T, d)
            Vtr = Vt64[t0:t0 + Hkv * T].reshape(Hkv, T, d)
            ref = odec.decode_attention(q[r].double().numpy(), Kv, Vv, Ktr, Vtr)
            vmax = max(np.abs(Vv).max(initial=0.0), np.abs(Vtr).max(initial=0.0), 1.0)
            assert (np.abs(got[r] - ref) <= tolerance(torch.bfloat16, ref, vmax)).all(), "layer %d request %d" % (l, r)
            if B[l] + T == 0:
                assert not got[r].any()
            r0 += Hkv * sum(B)
            t0 += Hkv * T
