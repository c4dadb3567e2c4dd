"""Guard regions and poisoned outputs: no kernel writes outside its output rows, and
every output row is written.

compute-sanitizer is closed on this machine, so out-of-bounds stores are caught the
plain way: every caller buffer the library writes (K_out, V_out, idx, scores,
ranks, keep and drop lists, decode outputs, 4-bit codes and parameters, and the
workspace itself) sits between a 4 KB head and a 4 KB tail filled with the byte
0xA5, and its body is poisoned (NaN for floats, -7 for indices).  After each call
on the workloads' shapes (the 7B shape at 12,544 tokens, the ragged batch of 8,
small and ragged shapes on both kernel paths, the fp32 single-layer workload) the
guards must be intact byte for byte, no NaN may remain in a float output, and
every index must lie in [0, n).  For byte outputs that can hold any value (the
4-bit codes), the call runs twice with the bodies pre-filled with 0x00 and with
0xFF: equal results mean every byte was written.
"""
import numpy as np
import pytest
import torch

from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
GUARD = 4096
SENTINEL = 0xA5


class Guarded:
    """A device buffer of `numel` elements between two 4 KB sentinel regions."""

    def __init__(self, numel, dtype, poison=None):
        es = torch.empty(0, dtype=dtype).element_size()
        self.g = GUARD // es
        self.numel = max(int(numel), 1)
        self.buf = torch.empty(self.numel + 2 * self.g, dtype=dtype, device=DEV)
        self.buf.view(torch.uint8).fill_(SENTINEL)
        self.body = self.buf[self.g:self.g + self.numel]
        if poison is None:
            poison = float("nan") if dtype.is_floating_point else -7
        self.body.fill_(poison)

    def view(self, *shape):
        return self.body.view(*shape)

    def check(self, tag):
        torch.cuda.synchronize()
        head = self.buf[:self.g].view(torch.uint8)
        tail = self.buf[self.g + self.numel:].view(torch.uint8)
        assert bool((head == SENTINEL).all()), "%s: write before the buffer" % tag
        assert bool((tail == SENTINEL).all()), "%s: write past the buffer" % tag


def _no_nan(t, tag):
    assert not bool(torch.isnan(t.float()).any()), "%s: unwritten (NaN) elements remain" % tag


def _batch(reqs):
    return vc.Batch([r.n for r in reqs], [r.W for r in reqs], [(r.rr_num, r.rr_den) for r in reqs])


def _inputs(wl):
    qs, ks, vs = synth.generate(wl, DEV)
    cat = lambda ts: torch.cat([t.flatten() for t in ts])
    return qs, ks, vs, cat(qs), cat(ks), cat(vs)


def _compress_guarded(wl, Q, K, V):
    batch = _batch(wl.requests)
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16 if wl.dtype == "bf16" else vc.VC_F32)
    rows = vc.compressed_rows(batch, prm)
    Ko = Guarded(rows * wl.d, K.dtype)
    Vo = Guarded(rows * wl.d, V.dtype)
    ix = Guarded(rows, torch.int32)
    ws = Guarded(vc.prunekv_workspace_size(batch, prm), torch.uint8, poison=0)
    vc.prunekv_compress(batch, prm, Q, K, V, Ko.view(rows, wl.d), Vo.view(rows, wl.d), ix.view(rows),
                        ws.body)
    assert vc.prunekv_get_status(ws.body) == vc.VC_OK
    for b, tag in ((Ko, "K_out"), (Vo, "V_out"), (ix, "idx"), (ws, "workspace")):
        b.check("%s %s" % (wl.name, tag))
    _no_nan(Ko.body, wl.name + " K_out")
    _no_nan(Vo.body, wl.name + " V_out")
    # indices in range, request by request
    off = 0
    for r in wl.requests:
        n_rows = vc.compressed_rows(_batch([r]), prm)
        seg = ix.body[off:off + n_rows]
        assert bool(((seg >= 0) & (seg < r.n)).all()), "%s idx out of range" % wl.name
        off += n_rows
    return batch, prm, Ko.view(rows, wl.d), Vo.view(rows, wl.d)


@pytest.mark.parametrize("wid", [1, 2, 3, 5])
def test_compress_writes_only_its_rows(wid):
    wl = synth.WORKLOADS[wid]
    _, _, _, Q, K, V = _inputs(wl)
    _compress_guarded(wl, Q, K, V)


SMALL = [
    # L, Hq, Hkv, d, n, W, dtype, rr
    (1, 2, 1, 64, 1, 1, torch.float32, (1, 1)),
    (2, 4, 2, 64, 63, 3, torch.bfloat16, (1, 2)),
    (3, 7, 1, 128, 129, 5, torch.bfloat16, (1, 4)),
    (4, 8, 1, 128, 1000, 64, torch.bfloat16, (19, 100)),
    (2, 8, 4, 64, 257, 32, torch.float32, (25, 100)),
    (5, 6, 2, 128, 700, 17, torch.float32, (28, 100)),
    (3, 14, 2, 128, 2049, 100, torch.bfloat16, (23, 100)),
]


@pytest.mark.parametrize("path", [vc.VC_PATH_AUTO, vc.VC_PATH_SIMT], ids=["auto", "simt"])
@pytest.mark.parametrize("case", SMALL)
def test_step_api_writes_only_its_rows(case, path):
    L, Hq, Hkv, d, n, W, dt, rr = case
    key = 9000 + 17 * SMALL.index(case)
    mk = lambda shape, k: synth._round(synth.normal(key + k, 0, int(np.prod(shape)), "cpu").view(*shape),
                                        dt).to(DEV)
    Q, K, V = mk((L, Hq, W, d), 1), mk((L, Hkv, n, d), 2), mk((L, Hkv, n, d), 3)
    B, Nq, _ = vc.viscache_plan_budgets(L, n, *rr)
    vc.viscache_set_kernel_path(path)
    try:
        for mode in (vc.VC_RANK_SHARED, vc.VC_RANK_PER_LAYER):
            shape = (Hkv, n) if mode == vc.VC_RANK_SHARED else (L, Hkv, n)
            sc = Guarded(int(np.prod(shape)), torch.float32)
            ws = Guarded(vc.prunekv_score_workspace_size(L, Hq, W), torch.uint8, poison=0)
            vc.prunekv_score(Q, K, rank_mode=mode, scores=sc.view(*shape), ws=ws.body)
            assert vc.prunekv_get_status(ws.body) == vc.VC_OK
            sc.check("scores"); ws.check("score workspace")
            _no_nan(sc.body, "scores")
            # selection through the C ABI with guarded outputs
            T, Dr = Hkv * sum(B), vc.drop_rows(B, Nq, Hkv)
            rk = Guarded(int(np.prod(shape)), torch.int32)
            kp = Guarded(T, torch.int32)
            dp = Guarded(Dr, torch.int32)
            ws2 = Guarded(vc.prunekv_select_workspace_size(L, Hkv, n, mode), torch.uint8, poison=0)
            import ctypes
            rc = vc.lib().prunekv_select(
                ctypes.c_void_p(sc.body.data_ptr()), L, Hkv, n, vc._i32(B), Nq, mode,
                ctypes.c_void_p(rk.body.data_ptr()), ctypes.c_void_p(kp.body.data_ptr()),
                ctypes.c_void_p(dp.body.data_ptr()), ctypes.c_void_p(ws2.body.data_ptr()),
                ws2.body.numel(), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
            assert rc == vc.VC_OK
            assert vc.prunekv_get_status(ws2.body) == vc.VC_OK
            for b, tag in ((rk, "rank"), (kp, "keep"), (dp, "drop"), (ws2, "select workspace")):
                b.check(tag)
            assert bool(((rk.body >= 0) & (rk.body < n)).all())
            if T:
                assert bool(((kp.body[:T] >= 0) & (kp.body[:T] < n)).all())
            if Dr:
                assert bool(((dp.body[:Dr] >= 0) & (dp.body[:Dr] < n)).all())
            if mode == vc.VC_RANK_PER_LAYER:
                continue
            # fusion with guarded outputs and workspace
            Ko = Guarded(max(T, 1) * d, dt)
            Vo = Guarded(max(T, 1) * d, dt)
            ws3 = Guarded(vc.prunekv_fuse_workspace_size(B, Hkv, d, n, Nq), torch.uint8, poison=0)
            vc.prunekv_fuse_compact(K, V, B, Nq, kp.body[:max(T, 1)], dp.body[:max(Dr, 1)], 0.7, 1.0,
                                    K_out=Ko.view(max(T, 1), d), V_out=Vo.view(max(T, 1), d), ws=ws3.body)
            assert vc.prunekv_get_status(ws3.body) == vc.VC_OK
            for b, tag in ((Ko, "K_out"), (Vo, "V_out"), (ws3, "fuse workspace")):
                b.check(tag)
            if T:
                _no_nan(Ko.body[:T * d], "K_out")
                _no_nan(Vo.body[:T * d], "V_out")
    finally:
        vc.viscache_set_kernel_path(vc.VC_PATH_AUTO)


def test_decode_and_4bit_cache_write_only_their_rows():
    wl = synth.scaled(synth.WORKLOADS[5], "guards: 3 ragged requests, 8 layers",
                      L=8, requests=synth.WORKLOADS[5].requests[:3])
    qs, ks, vs, Q, K, V = _inputs(wl)
    batch, prm, Ko, Vo = _compress_guarded(wl, Q, K, V)
    n_req, Hq, Hkv, d = len(wl.requests), wl.Hq, wl.Hkv, wl.d
    n_text = [40, 0, 300]
    kt = synth._round(synth.normal(71, 0, Hkv * sum(n_text) * d, "cpu"), torch.bfloat16).view(-1, d).to(DEV)
    vt = synth._round(synth.normal(72, 0, Hkv * sum(n_text) * d, "cpu"), torch.bfloat16).view(-1, d).to(DEV)
    q = synth._round(synth.normal(73, 0, n_req * Hq * d, "cpu"), torch.bfloat16).view(n_req, Hq, d).to(DEV)
    for layer in (0, wl.L - 1):
        out = Guarded(n_req * Hq * d, torch.bfloat16)
        need = vc.viscache_decode_workspace_size(batch, prm, n_text)
        ws = Guarded(need, torch.uint8, poison=0)
        vc.viscache_decode_attention(batch, prm, layer, q, Ko, Vo, kt, vt, n_text,
                                     out=out.view(n_req, Hq, d), ws=ws.body)
        out.check("decode out"); ws.check("decode workspace")
        _no_nan(out.body, "decode out")
    # 4-bit form: codes written everywhere (two prefills agree), parameters finite
    rows, groups = vc.viscache_kv4_sizes(batch, prm)
    results = []
    for fill in (0x00, 0xFF):
        kc = Guarded(rows * d // 2, torch.uint8, poison=fill)
        vcc = Guarded(rows * d // 2, torch.uint8, poison=fill)
        kpp = Guarded(groups * d * 2, torch.float32)
        vpp = Guarded(rows * (d // 32) * 2, torch.float32)
        vc.viscache_kv4_quantize(batch, prm, Ko, Vo, out=(kc.view(rows, d // 2), vcc.view(rows, d // 2),
                                                          kpp.view(groups, d, 2), vpp.view(rows, d // 32, 2)))
        for b, tag in ((kc, "K codes"), (vcc, "V codes"), (kpp, "K params"), (vpp, "V params")):
            b.check(tag)
        _no_nan(kpp.body, "K params")
        _no_nan(vpp.body, "V params")
        results.append((kc.body.clone(), vcc.body.clone()))
        kh = Guarded(rows * d, torch.bfloat16)
        vh = Guarded(rows * d, torch.bfloat16)
        vc.viscache_kv4_dequantize(batch, prm, kc.view(rows, d // 2), vcc.view(rows, d // 2),
                                   kpp.view(groups, d, 2), vpp.view(rows, d // 32, 2),
                                   out=(kh.view(rows, d), vh.view(rows, d)))
        kh.check("K_hat"); vh.check("V_hat")
        _no_nan(kh.body, "K_hat")
        _no_nan(vh.body, "V_hat")
    assert torch.equal(results[0][0], results[1][0]), "K codes: some bytes unwritten"
    assert torch.equal(results[0][1], results[1][1]), "V codes: some bytes unwritten"
