"""CPU checks of the C-ABI library: it loads, exports every declared symbol, the host
planner matches the oracle planner bit-exactly, and argument errors come back as codes."""
import ctypes
import os
import re
from fractions import Fraction

import pytest

from oracle import plan
from paper_2608_24063_gb300 import viscache as vc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "viscache.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:int|size_t|const char\*)\s+(\w+)\s*\(", src, flags=re.M)))


def test_library_exports_every_declared_symbol():
    names = _declared()
    assert "prunekv_compress" in names and "viscache_plan_budgets" in names
    lib = vc.lib()
    for name in names:
        assert hasattr(lib, name), name
    assert set(vc.EXPORTED) == set(names)


def test_version():
    assert "sm_103a" in vc.viscache_version()


def test_device_accessible_null_pointer():
    assert vc.lib().viscache_device_accessible(None) == 0


@pytest.mark.parametrize("rr", [(19, 100), (22, 100), (23, 100), (28, 100), (1, 3), (56, 100)])
def test_planner_matches_oracle_exhaustive_L(rr):
    for L in range(1, 129):
        for n in (1, 7, 1000, 3136, 12544, 32768):
            try:
                ref = plan.plan_budgets(L, n, Fraction(*rr))
            except plan.Infeasible:
                with pytest.raises(vc.VisCacheError) as ei:
                    vc.viscache_plan_budgets(L, n, *rr)
                assert ei.value.code == vc.VC_ERR_INFEASIBLE
                continue
            got = vc.viscache_plan_budgets(L, n, *rr)
            assert got == (ref[0], ref[1], ref[2]), (L, n, rr)


SCHED = [(vc.VC_SCHED_PARABOLA, "parabola"), (vc.VC_SCHED_FIXED, "fixed"),
         (vc.VC_SCHED_ARITHMETIC, "arithmetic"), (vc.VC_SCHED_GEOMETRIC, "geometric")]


@pytest.mark.parametrize("code,name", SCHED)
@pytest.mark.parametrize("drop_code,drop", [(vc.VC_DROP_SURVIVORS, "survivors"), (vc.VC_DROP_ALL, "all")])
def test_schedule_planner_matches_oracle(code, name, drop_code, drop):
    for L in list(range(1, 41)) + [64, 80, 128]:
        for n in (1, 7, 1000, 12544):
            for rr in ((19, 100), (28, 100), (1, 3)):
                try:
                    ref = plan.plan_budgets(L, n, Fraction(*rr), schedule=name, drop=drop)
                except plan.Infeasible:
                    with pytest.raises(vc.VisCacheError) as ei:
                        vc.viscache_plan_budgets_ex(L, n, *rr, 0, 3, 4, code, drop_code)
                    assert ei.value.code == vc.VC_ERR_INFEASIBLE
                    continue
                got = vc.viscache_plan_budgets_ex(L, n, *rr, 0, 3, 4, code, drop_code)
                assert got == (ref[0], ref[1], ref[2]), (L, n, rr, name, drop)


def test_schedule_planner_rejects_unknown_choices():
    for sched, drop in [(-1, 0), (4, 0), (0, 2), (0, -1)]:
        with pytest.raises(vc.VisCacheError) as ei:
            vc.viscache_plan_budgets_ex(28, 1000, 1, 5, 0, 3, 4, sched, drop)
        assert ei.value.code == vc.VC_ERR_INVALID_ARG


def test_planner_explicit_h_and_m():
    for L, h, m in [(28, 14, (1, 2)), (80, 80, (1, 1)), (5, 1, (3, 4)), (64, 48, (3, 4))]:
        ref = plan.plan_budgets(L, 5000, Fraction(1, 5), h=h, m=Fraction(*m))
        assert vc.viscache_plan_budgets(L, 5000, 1, 5, h, *m) == ref


def test_planner_argument_errors():
    for args in [(0, 10, 1, 2), (3, 0, 1, 2), (3, 10, 0, 2), (3, 10, 3, 2), (3, 10, 1, 0)]:
        with pytest.raises(vc.VisCacheError) as ei:
            vc.viscache_plan_budgets(*args)
        assert ei.value.code == vc.VC_ERR_INVALID_ARG
    with pytest.raises(vc.VisCacheError):
        vc.viscache_plan_budgets(4, 10, 1, 2, 5)          # h > L


def test_entry_points_reject_bad_arguments_without_touching_the_device():
    lib = vc.lib()
    p = ctypes.c_void_p(256)
    # d not in {64, 128}
    assert lib.prunekv_score(p, p, 0, 1, 2, 1, 96, 10, 4, 0.0, 0, None, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    # Hq % Hkv != 0
    assert lib.prunekv_score(p, p, 0, 1, 3, 2, 64, 10, 4, 0.0, 0, None, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    # misaligned pointer
    q = ctypes.c_void_p(258)
    assert lib.prunekv_score(q, p, 0, 1, 2, 1, 64, 10, 4, 0.0, 0, None, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    # workspace too small / misaligned
    assert lib.prunekv_score(p, p, 0, 1, 2, 1, 64, 10, 4, 0.0, 0, None, p, p, 16, None) == vc.VC_ERR_WORKSPACE
    assert lib.prunekv_score(p, p, 0, 1, 2, 1, 64, 10, 4, 0.0, 0, None, p, ctypes.c_void_p(272), 1 << 20, None) == vc.VC_ERR_WORKSPACE
    # more tokens than the documented maximum
    B1 = (ctypes.c_int32 * 1)(3)
    assert lib.prunekv_select(p, 1, 1, 65537, B1, 4, 0, p, p, p, p, 1 << 30, None) == vc.VC_ERR_INVALID_ARG
    # B_l > Nq, Nq > n
    B = (ctypes.c_int32 * 2)(5, 3)
    assert lib.prunekv_select(p, 2, 1, 10, B, 4, 0, p, p, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    assert lib.prunekv_select(p, 2, 1, 10, B, 11, 0, p, p, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    # mu out of range, tau <= 0
    B2 = (ctypes.c_int32 * 1)(2)
    assert lib.prunekv_fuse_compact(p, p, 0, 1, 1, 64, 10, B2, 4, p, p, 1.5, 1.0, p, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    assert lib.prunekv_fuse_compact(p, p, 0, 1, 1, 64, 10, B2, 4, p, p, 0.5, 0.0, p, p, p, 1 << 20, None) == vc.VC_ERR_INVALID_ARG
    # batch: infeasible retention surfaces as VC_ERR_INFEASIBLE
    b = vc.Batch([10], [4], [(1, 1)])
    prm = vc.make_params(4, 2, 1, 64, vc.VC_BF16, h=2, m=(1, 2))
    assert lib.prunekv_compress(ctypes.byref(b.c), ctypes.byref(prm), p, p, p, p, p, p, p, 1 << 30, None) == vc.VC_ERR_INFEASIBLE


def test_workspace_sizes_are_positive_and_aligned():
    assert vc.prunekv_score_workspace_size(28, 28, 64) % 256 == 0
    assert vc.prunekv_score_workspace_size(28, 28, 64) >= 28 * 28 * 64 * 4
    # sorted 1024-key chunks (8-byte keys) for every ranking problem
    assert vc.prunekv_select_workspace_size(28, 4, 12544) >= 8 * 1024 * 4 * 13
    assert vc.prunekv_select_workspace_size(28, 4, 12544, vc.VC_RANK_PER_LAYER) >= 8 * 1024 * 28 * 4 * 13
    assert vc.prunekv_select_workspace_size(2, 2, 65536) >= 8 * 65536 * 2
    assert vc.prunekv_fuse_workspace_size([3833, 1916], 4, 128, 12544, 4237) > 4 * 4237 * 2 * 256
    b = vc.Batch([12544], [64], [(19, 100)])
    prm = vc.make_params(28, 28, 4, 128, vc.VC_BF16)
    assert vc.prunekv_workspace_size(b, prm) > vc.prunekv_score_workspace_size(28, 28, 64)
    assert vc.compressed_rows(b, prm) == 4 * 66734


def test_decode_entry_rejects_bad_arguments_without_touching_the_device():
    lib = vc.lib()
    p = ctypes.c_void_p(256)
    b = vc.Batch([100, 50], [8, 8], [(25, 100), (25, 100)])
    prm = vc.make_params(4, 8, 2, 128, vc.VC_BF16)
    call = lambda prm, layer, q=p, nt=None, ws=p, wsb=1 << 30: lib.viscache_decode_attention(
        ctypes.byref(b.c), ctypes.byref(prm), layer, q, p, p, None, None, nt, p, ws, wsb, None)
    assert call(prm, 4) == vc.VC_ERR_INVALID_ARG                           # layer out of range
    assert call(prm, -1) == vc.VC_ERR_INVALID_ARG
    assert call(prm, 0, q=ctypes.c_void_p(264)) == vc.VC_ERR_INVALID_ARG   # misaligned q
    nt = (ctypes.c_int32 * 2)(3, 0)
    assert call(prm, 0, nt=nt) == vc.VC_ERR_INVALID_ARG                    # text lengths, no text rows
    assert call(prm, 0, wsb=16) == vc.VC_ERR_WORKSPACE
    assert call(prm, 0, ws=ctypes.c_void_p(272)) == vc.VC_ERR_WORKSPACE
    wide = vc.make_params(4, 32, 2, 128, vc.VC_BF16)                     # 16 query heads per KV head
    assert call(wide, 0) == vc.VC_ERR_INVALID_ARG
    assert vc.viscache_decode_workspace_size(b, wide) == 0


def test_decode_workspace_covers_every_layer():
    # the largest layer budget, split into 512-key pieces per KV head, bounds
    # the partial states (8 query slots x d floats + 8 (max, sum) pairs each)
    b = vc.Batch([12544], [64], [(19, 100)])
    prm = vc.make_params(28, 28, 4, 128, vc.VC_BF16)
    B, _, _ = vc.viscache_plan_budgets(28, 12544, 19, 100)
    units = 4 * -(-(max(B) + 300) // 512)
    got = vc.viscache_decode_workspace_size(b, prm, [300])
    assert got % 256 == 0 and got >= units * 8 * (128 * 4 + 8)
    assert vc.viscache_decode_workspace_size(b, prm) <= got
    assert vc.viscache_decode_workspace_size(vc.Batch([100] * 257, [8] * 257, [(1, 4)] * 257), prm) == 0


def test_kv4_sizes_match_the_oracle_layout():
    from oracle import quant as oq
    ns, rrs, L, Hkv = [12544, 700, 33], [(19, 100), (25, 100), (50, 100)], 28, 4
    b = vc.Batch(ns, [64] * 3, rrs)
    prm = vc.make_params(L, 28, Hkv, 128, vc.VC_BF16)
    Bs = [plan.plan_budgets(L, n, Fraction(*rr))[0] for n, rr in zip(ns, rrs)]
    rows, groups = vc.viscache_kv4_sizes(b, prm)
    segs = oq.segments(Bs, Hkv)
    assert rows == sum(n for _, n in segs)
    assert groups == sum(-(-n // oq.GROUP) for _, n in segs)


def test_kv4_entries_reject_bad_arguments_without_touching_the_device():
    lib = vc.lib()
    p = ctypes.c_void_p(256)
    b = vc.Batch([100], [8], [(25, 100)])
    prm = vc.make_params(4, 8, 2, 128, vc.VC_BF16)
    args = lambda *x: (ctypes.byref(b.c), ctypes.byref(prm)) + x
    assert lib.viscache_kv4_quantize(*args(p, p, None, p, p, p, None)) == vc.VC_ERR_INVALID_ARG
    assert lib.viscache_kv4_quantize(*args(p, p, p, p, ctypes.c_void_p(260), p, None)) == vc.VC_ERR_INVALID_ARG
    assert lib.viscache_kv4_dequantize(*args(p, p, p, p, None, p, None)) == vc.VC_ERR_INVALID_ARG
    bad = vc.make_params(4, 8, 2, 96, vc.VC_BF16)
    assert lib.viscache_kv4_sizes(ctypes.byref(b.c), ctypes.byref(bad), None, None) == vc.VC_ERR_INVALID_ARG


def test_repeated_batches_reuse_plans_and_changes_replan():
    # the batch entry points plan once per distinct (batch, parameters); any
    # change of either must give the new plan, alternating calls included
    b1 = vc.Batch([12544, 700], [64, 8], [(19, 100), (25, 100)])
    b2 = vc.Batch([12544, 701], [64, 8], [(19, 100), (25, 100)])
    p1 = vc.make_params(28, 28, 4, 128, vc.VC_BF16)
    p2 = vc.make_params(28, 28, 4, 128, vc.VC_BF16, schedule=vc.VC_SCHED_FIXED)

    def expect(b, p):
        rows = groups = 0
        for n, (a, d) in zip(b.n_vis, b.rr):
            B = plan.plan_budgets(28, n, Fraction(a, d), schedule="fixed" if p.schedule else "parabola")[0]
            rows += 4 * sum(B)
            groups += 4 * sum(-(-x // 32) for x in B)
        return rows, groups

    for b, p in [(b1, p1), (b1, p1), (b2, p1), (b1, p1), (b1, p2), (b1, p1), (b2, p2)]:
        assert vc.viscache_kv4_sizes(b, p) == expect(b, p)


def test_static_scratch_capacity_matches_header():
    """The no-allocation scoring entry point's array size, as the library reports it,
    is the header's VC_STATIC_SCRATCH_BYTES (the binding reads it from the library)."""
    src = open(os.path.join(ROOT, "include", "viscache.h")).read()
    m = re.search(r"#define\s+VC_STATIC_SCRATCH_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", src)
    assert m, "VC_STATIC_SCRATCH_BYTES not found"
    assert vc.prunekv_score_static_capacity() == int(m.group(1)) << int(m.group(2))
    # the 7B shape fits with up to 512 window rows; the 72B shape with 128 does not
    assert vc.prunekv_score_workspace_size(28, 28, 512) <= vc.prunekv_score_static_capacity()
    assert vc.prunekv_score_workspace_size(80, 64, 128) > vc.prunekv_score_static_capacity()


def test_scout_sizes_match_oracle_keyframe_count():
    """The C sizing call the binding uses for the scout's outputs gives the oracle's
    k = ceil(p F) for every video; bad arguments come back as codes."""
    from oracle import scout as osc
    frames = [1, 2, 3, 7, 64, 100, 333, 4096]
    for p in [(1, 1), (3, 4), (1, 3), (2, 7), (1, 4096)]:
        kk = (ctypes.c_int32 * len(frames))()
        arr = (ctypes.c_int32 * len(frames))(*frames)
        assert vc.lib().viscache_scout_sizes(len(frames), arr, p[0], p[1], kk) == vc.VC_OK
        assert list(kk) == [osc.keyframe_count(F, Fraction(*p)) for F in frames], p
    one = (ctypes.c_int32 * 1)(5)
    out = (ctypes.c_int32 * 1)()
    assert vc.lib().viscache_scout_sizes(1, one, 0, 4, out) == vc.VC_ERR_INVALID_ARG
    assert vc.lib().viscache_scout_sizes(1, one, 5, 4, out) == vc.VC_ERR_INVALID_ARG
    assert vc.lib().viscache_scout_sizes(1, (ctypes.c_int32 * 1)(0), 3, 4, out) == vc.VC_ERR_INVALID_ARG
    assert vc.lib().viscache_scout_sizes(1, one, 3, 4, None) == vc.VC_ERR_INVALID_ARG


def test_test_wait_switch_rejects_unknown_bits():
    assert vc.lib().viscache_test_inject_wait(8) == vc.VC_ERR_INVALID_ARG
    assert vc.lib().viscache_test_inject_wait(-1) == vc.VC_ERR_INVALID_ARG
    assert vc.lib().viscache_test_inject_wait(0) == vc.VC_OK
