"""Planted mistakes in the oracle: every one must be caught by the pins.

Each case replaces one oracle function (on the CPU, for this test only) with
a copy that carries a single plausible mistake -- a dropped term, a wrong
sign, index or axis, a transposed or swapped operand, an off-by-one -- and
runs the pin tests of that part of the oracle (test_oracle_plan,
test_oracle_scores, test_oracle_select_fuse, test_oracle_scout,
test_oracle_decode, test_oracle_quant).  At least one pin must fail.

The pins used here check the oracle against things other than itself: values
and closed forms from the paper, brute force on tiny inputs, invariants, and
library routines (torch softmax / SDPA).  The stored golden budgets are left
out on purpose: they were written by the oracle, so they would catch a change
but prove nothing about correctness.
"""
import inspect
import itertools
from fractions import Fraction
from math import floor

import numpy as np
import pytest

from oracle import plan
from oracle import prunekv as ok
from oracle import decode as odec
from oracle import quant as oq
from oracle import scout as osc
from tests import test_oracle_decode as pins_decode
from tests import test_oracle_plan as pins_plan
from tests import test_oracle_quant as pins_quant
from tests import test_oracle_scout as pins_scout
from tests import test_oracle_scores as pins_scores
from tests import test_oracle_select_fuse as pins_select_fuse

SELF_PINS = {"test_golden_budgets_match_oracle"}


def _pin_calls(module):
    """Every test function of a pin module with its parametrize grid expanded."""
    for name, fn in inspect.getmembers(module, inspect.isfunction):
        if not name.startswith("test_") or name in SELF_PINS or fn.__module__ != module.__name__:
            continue
        grids = []
        for mark in getattr(fn, "pytestmark", []):
            if mark.name != "parametrize":
                continue
            names = mark.args[0]
            names = [s.strip() for s in names.split(",")] if isinstance(names, str) else list(names)
            combos = []
            for v in mark.args[1]:
                v = v.values if hasattr(v, "values") else v
                v = tuple(v) if len(names) > 1 else (v,)
                combos.append(dict(zip(names, v)))
            grids.append(combos)
        for combo in itertools.product(*grids) if grids else [()]:
            kw = {}
            for part in combo:
                kw.update(part)
            yield name, fn, kw


def _failing_pins(modules):
    failed = []
    for mod in modules:
        for name, fn, kw in _pin_calls(mod):
            try:
                fn(**kw)
            except Exception:      # an assertion, or a crash a real run would report
                failed.append(name)
    return sorted(set(failed))


# ---------------------------------------------------------------------------
# mutated copies of oracle functions (one planted mistake each)

def _softmax_rows(x):
    m = x.max(axis=-1, keepdims=True)
    e = np.exp(x - m)
    return e / e.sum(axis=-1, keepdims=True)


def _attention(Qw_l, K_l, scale, row_lse=None, kv=lambda j, G, Hkv: j // G, use_scale=True,
               axis_rows=False, lse_sign=-1.0):
    Hq, W, d = Qw_l.shape
    Hkv = K_l.shape[0]
    G = Hq // Hkv
    out = np.empty((Hq, W, K_l.shape[1]))
    for j in range(Hq):
        x = Qw_l[j] @ K_l[kv(j, G, Hkv)].T
        if use_scale:
            x = x * scale
        if row_lse is not None:
            out[j] = np.exp(x + lse_sign * row_lse[j][:, None])
        elif axis_rows:
            out[j] = _softmax_rows(x.T).T
        else:
            out[j] = _softmax_rows(x)
    return out


def _scores(Qw, K, scale=None, rank_mode="shared", row_lse=None, mean=True, heads=None):
    L, Hq, W, d = Qw.shape
    _, Hkv, n, _ = K.shape
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    per_layer = np.zeros((L, Hkv, n))
    for l in range(L):
        A = ok.attention_weights(Qw[l], K[l], scale, None if row_lse is None else row_lse[l])
        for g in range(Hkv):
            hi = (g + 1) * G if heads is None else g * G + heads
            per_layer[l, g] = A[g * G:hi].sum(axis=(0, 1))
    if rank_mode == "per_layer":
        return per_layer
    return per_layer.sum(axis=0) / (L if mean else 1)


def _select(s, B, Nq, rank_mode="shared", order_fn=None, drop_from=0, drop_to=0, sort_keep=True):
    L = len(B)
    Hkv = s.shape[-2]
    keep = [[None] * Hkv for _ in range(L)]
    drop = [[None] * Hkv for _ in range(L)]
    rank = np.empty(s.shape, dtype=np.int64)
    rank_fn = order_fn or ok.ranking
    for g in range(Hkv):
        for l in range(L):
            sv = s[l, g] if rank_mode == "per_layer" else s[g]
            order = rank_fn(sv)
            if rank_mode == "per_layer":
                rank[l, g, order] = np.arange(order.size)
            elif l == 0:
                rank[g, order] = np.arange(order.size)
            kp = order[:B[l]]
            keep[l][g] = (np.sort(kp) if sort_keep else kp) if B[l] > 0 else np.zeros(0, np.int64)
            drop[l][g] = (np.sort(order[B[l] + drop_from:Nq + drop_to]) if B[l] > 0
                          else np.zeros(0, np.int64))
    return keep, drop, rank


def _fuse(V_lg, keep_lg, drop_lg, mu, tau, phi_axis=-1, swap_mu=False, use_tau=True,
          empty_zero=False):
    Vk = V_lg[keep_lg]
    if drop_lg.size == 0:
        return np.zeros_like(Vk) if empty_zero else Vk.copy()
    Vd = V_lg[drop_lg]
    Z = Vk @ Vd.T
    if use_tau:
        Z = Z / tau
    Phi = _softmax_rows(Z) if phi_axis == -1 else _softmax_rows(Z.T).T
    a, b = (1.0 - mu, mu) if swap_mu else (mu, 1.0 - mu)
    return a * Vk + b * (Phi @ Vd)


def _parabolic_no_half(h):
    if h == 1:
        return [Fraction(1)]
    return [1 - Fraction((l - 1) ** 2, (h - 1) ** 2) for l in range(1, h + 1)]


def _normalised_to_h(h, m, schedule="parabola"):
    b = plan.schedule_proportions(h, schedule)
    s = sum(b)
    return [x * h / s for x in b]


def _apportion_ties_high(total, weights):
    W = sum(weights)
    quotas = [total * w / W for w in weights]
    base = [floor(q) for q in quotas]
    left = total - sum(base)
    order = sorted(range(len(weights)), key=lambda i: (-(quotas[i] - base[i]), -i))
    for i in order[:left]:
        base[i] += 1
    return base


def _schedule_mutant(arith_end=Fraction(1, 2), geo_ratio=Fraction(1, 2), small_blocks_first=False):
    def fn(h, schedule="parabola"):
        if schedule == "arithmetic" and h > 1:
            return [1 - (1 - arith_end) * Fraction(l - 1, h - 1) for l in range(1, h + 1)]
        if schedule == "geometric" and h > 1:
            nb = min(4, h)
            per, extra = divmod(h, nb)
            sizes = [per + (1 if k < extra else 0) for k in range(nb)]
            if small_blocks_first:
                sizes = sizes[::-1]
            b = []
            for k in range(nb):
                b += [geo_ratio ** k] * sizes[k]
            return b
        return _ORIG_SCHEDULE(h, schedule)
    return fn


_ORIG_SCHEDULE = plan.schedule_proportions


def _plan_drop_all_ignored(L, n, rr, h=None, m=Fraction(3, 4), schedule="parabola", drop="survivors"):
    return _ORIG_PLAN(L, n, rr, h, m, schedule)


_ORIG_PLAN = plan.plan_budgets


def _default_h_floor(L):
    h = floor(Fraction(3 * L, 4))
    return max(min(2, L), min(h, L))


def _plan_nq_without_m(L, n, rr, h=None, m=Fraction(3, 4), schedule="parabola", drop="survivors"):
    if h is None or h == 0:
        h = plan.default_h(L)
    T = plan.round_half_up(rr * n * L)
    B = plan.apportion(T, plan.normalised_proportions(h, m, schedule)) + [0] * (L - h)
    if B[0] > n:
        raise plan.Infeasible("infeasible")
    Nq = min(n, max(plan.round_half_up(Fraction(T) / h), B[0]))
    return B, (n if drop == "all" else Nq), h


def _plan_total_floor(L, n, rr, h=None, m=Fraction(3, 4), schedule="parabola", drop="survivors"):
    if h is None or h == 0:
        h = plan.default_h(L)
    T = floor(rr * n * L)
    B = plan.apportion(T, plan.normalised_proportions(h, m, schedule)) + [0] * (L - h)
    if B[0] > n:
        raise plan.Infeasible("infeasible")
    Nq = min(n, max(plan.round_half_up(Fraction(T) / (h * m)), B[0]))
    return B, (n if drop == "all" else Nq), h


def _mmr(H, h_t, lam, k, swap=False, ties_high=False, red_mode="max", unit=True):
    Hn = osc.cosine_unit(H) if unit else np.asarray(H, dtype=np.float64)
    tn = osc.cosine_unit(h_t[None, :])[0] if unit else np.asarray(h_t, dtype=np.float64)
    F = Hn.shape[0]
    rel = Hn @ tn
    a, b = (1.0 - lam, lam) if swap else (lam, 1.0 - lam)
    chosen = np.zeros(F, dtype=bool)
    order, gains, picked = [], [], []
    for step in range(k):
        if picked:
            sims = Hn @ Hn[picked].T
            red = {"max": sims.max(axis=1), "mean": sims.mean(axis=1), "last": sims[:, -1]}[red_mode]
        else:
            red = np.zeros(F)
        score = a * rel - b * red
        score[chosen] = -np.inf
        f = int(F - 1 - np.argmax(score[::-1])) if ties_high else int(np.argmax(score))
        order.append(f)
        gains.append(score[f])
        chosen[f] = True
        picked.append(f)
    return np.array(order, dtype=np.int64), np.array(gains)


SCORES = [pins_scores, pins_select_fuse]
SCOUT = [pins_scout]
DECODE = [pins_decode]
QUANT = [pins_quant]


def _params_mutant(levels=15, zero_min=False):
    def group_params(x, axis):
        x = np.asarray(x, dtype=np.float32)
        lo = x.min(axis=axis)
        hi = x.max(axis=axis)
        if zero_min:
            lo = np.zeros_like(lo)
        return ((hi - lo) / np.float32(levels)).astype(np.float32), lo.astype(np.float32)
    return group_params


def _codes_floor(x, scale, lo):
    x = np.asarray(x, dtype=np.float32)
    with np.errstate(divide="ignore", invalid="ignore"):
        q = np.floor((x - lo) / scale)
    q = np.where(scale > 0, q, 0.0)
    return np.clip(q, 0, 15).astype(np.uint8)


def _pack_swapped(codes):
    codes = np.asarray(codes, dtype=np.uint8)
    return (codes[:, 1::2] | (codes[:, 0::2] << 4)).astype(np.uint8)


def _keys_one_group(K):
    K = np.asarray(K, dtype=np.float32)
    s, m = oq.group_params(K, axis=0)
    return oq.codes_of(K, s[None, :], m[None, :]), s[None, :], m[None, :]


def _values_group64(V):
    V = np.asarray(V, dtype=np.float32)
    R, d = V.shape
    g = V.reshape(R, d // 64, 64)
    s, m = oq.group_params(g, axis=2)
    codes = oq.codes_of(g, s[:, :, None], m[:, :, None]).reshape(R, d)
    return codes, np.repeat(s, 2, axis=1), np.repeat(m, 2, axis=1)


def _decode(q, K_vis, V_vis, K_text=None, V_text=None, scale=None, head_map="group", drop_text=False,
            scale_mode="sqrt", sum_mode="softmax"):
    """oracle.decode.decode_attention with one planted mistake."""
    q = np.asarray(q, dtype=np.float64)
    Hq, d = q.shape
    Hkv = K_vis.shape[0]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(d) if scale_mode == "sqrt" else 1.0 / d
    out = np.zeros((Hq, d))
    for j in range(Hq):
        g = j // G if head_map == "group" else j % Hkv
        Ks, Vs = [np.asarray(K_vis[g], np.float64)], [np.asarray(V_vis[g], np.float64)]
        if K_text is not None and not drop_text:
            Ks.append(np.asarray(K_text[g], np.float64))
            Vs.append(np.asarray(V_text[g], np.float64))
        Kc, Vc = np.concatenate(Ks), np.concatenate(Vs)
        if Kc.shape[0] == 0:
            continue
        x = (Kc @ q[j]) * scale
        p = np.exp(x - x.max())
        out[j] = (p / p.sum()) @ Vc if sum_mode == "softmax" else (p / p.shape[0]) @ Vc
    return out
SELECT_FUSE = [pins_select_fuse]
PLAN = [pins_plan]

MUTATIONS = [
    # scores (Eq. token_score)
    ("shared score without the 1/L mean", ok, "token_scores",
     lambda *a, **k: _scores(*a, mean=False, **k), SCORES),
    ("only the first query head of each group", ok, "token_scores",
     lambda *a, **k: _scores(*a, heads=1, **k), SCORES),
    ("GQA map j % Hkv instead of j // G", ok, "attention_weights",
     lambda *a: _attention(*a, kv=lambda j, G, Hkv: j % Hkv), SCORES),
    ("logit scale 1/sqrt(d) dropped", ok, "attention_weights",
     lambda *a: _attention(*a, use_scale=False), SCORES),
    ("softmax over the window rows instead of the keys", ok, "attention_weights",
     lambda *a: _attention(*a, axis_rows=True), SCORES),
    ("prefill normaliser added instead of subtracted", ok, "attention_weights",
     lambda *a: _attention(*a, lse_sign=1.0), SCORES),
    # ranking and selection (Algorithm 1 steps 1 and 3)
    ("ties to the higher index", ok, "ranking",
     lambda s: np.lexsort((-np.arange(s.shape[0]), -s)), SELECT_FUSE),
    ("ascending instead of descending scores", ok, "ranking",
     lambda s: np.lexsort((np.arange(s.shape[0]), s)), SELECT_FUSE),
    ("drop set starts one rank late", ok, "select",
     lambda *a, **k: _select(*a, drop_from=1, **k), SELECT_FUSE),
    ("drop set runs one rank past the survivors", ok, "select",
     lambda *a, **k: _select(*a, drop_to=1, **k), SELECT_FUSE),
    ("keep lists in rank order instead of position order", ok, "select",
     lambda *a, **k: _select(*a, sort_keep=False, **k), SELECT_FUSE),
    ("key compaction in reverse order", ok, "compact_keys",
     lambda K_lg, keep_lg: K_lg[keep_lg[::-1]], SELECT_FUSE),
    # value fusion (Eq. redistribution, Eq. weight_fusion)
    ("Phi normalised over the kept rows", ok, "fuse_values",
     lambda *a: _fuse(*a, phi_axis=0), SELECT_FUSE),
    ("mu and 1 - mu swapped", ok, "fuse_values",
     lambda *a: _fuse(*a, swap_mu=True), SELECT_FUSE),
    ("temperature ignored", ok, "fuse_values",
     lambda *a: _fuse(*a, use_tau=False), SELECT_FUSE),
    ("empty drop set gives zeros", ok, "fuse_values",
     lambda *a: _fuse(*a, empty_zero=True), SELECT_FUSE),
    # budgets (Eq. parabolic, its normalisation, Sec. 4 defaults)
    ("parabola without the factor 2", plan, "parabolic_proportions", _parabolic_no_half, PLAN),
    ("proportions normalised to h instead of h*m", plan, "normalised_proportions",
     _normalised_to_h, PLAN),
    ("largest-remainder ties to the higher layer", plan, "apportion", _apportion_ties_high, PLAN),
    ("truncation layer floor(3L/4) instead of rounded", plan, "default_h", _default_h_floor, PLAN),
    ("survivors T/h without m", plan, "plan_budgets", _plan_nq_without_m, PLAN),
    ("total T rounded down", plan, "plan_budgets", _plan_total_floor, PLAN),
    ("arithmetic schedule ending at 1/3", plan, "schedule_proportions",
     _schedule_mutant(arith_end=Fraction(1, 3)), PLAN),
    ("geometric ratio 2/3 per block", plan, "schedule_proportions",
     _schedule_mutant(geo_ratio=Fraction(2, 3)), PLAN),
    ("geometric blocks smaller first", plan, "schedule_proportions",
     _schedule_mutant(small_blocks_first=True), PLAN),
    ("drop-all reading ignored", plan, "plan_budgets", _plan_drop_all_ignored, PLAN),
    # scout keyframe selection (Eq. mmr)
    ("relevance and redundancy weights swapped", osc, "mmr_select",
     lambda *a: _mmr(*a, swap=True), SCOUT),
    ("MMR ties to the higher frame", osc, "mmr_select", lambda *a: _mmr(*a, ties_high=True), SCOUT),
    ("redundancy as the mean over the selected frames", osc, "mmr_select",
     lambda *a: _mmr(*a, red_mode="mean"), SCOUT),
    ("redundancy to the last pick only", osc, "mmr_select", lambda *a: _mmr(*a, red_mode="last"), SCOUT),
    ("dot products instead of cosines", osc, "mmr_select", lambda *a: _mmr(*a, unit=False), SCOUT),
    ("keyframe count rounded down", osc, "keyframe_count",
     lambda F, p: max(1, min(F, floor(Fraction(p) * F))), SCOUT),
    # decode attention over the compressed cache (Sec. 2 decoding)
    ("query head j reads KV head j mod Hkv", odec, "decode_attention",
     lambda *a, **k: _decode(*a, head_map="mod", **k), DECODE),
    ("text rows left out", odec, "decode_attention", lambda *a, **k: _decode(*a, drop_text=True, **k), DECODE),
    ("logits scaled by 1/d", odec, "decode_attention", lambda *a, **k: _decode(*a, scale_mode="d", **k), DECODE),
    ("weights divided by the key count, not their sum", odec, "decode_attention",
     lambda *a, **k: _decode(*a, sum_mode="count", **k), DECODE),
    # 4-bit quantisation of the compacted cache
    ("16 levels per step instead of 15", oq, "group_params", _params_mutant(levels=16), QUANT),
    ("minimum taken as zero", oq, "group_params", _params_mutant(zero_min=True), QUANT),
    ("codes rounded down", oq, "codes_of", _codes_floor, QUANT),
    ("odd channel in the low nibble", oq, "pack", _pack_swapped, QUANT),
    ("one key group per segment", oq, "quantize_keys", _keys_one_group, QUANT),
    ("value groups of 64 channels", oq, "quantize_values", _values_group64, QUANT),
]


def test_pins_pass_on_the_oracle():
    assert _failing_pins([pins_plan, pins_scores, pins_select_fuse, pins_scout, pins_decode,
                          pins_quant]) == []


@pytest.mark.parametrize("what,module,attr,mutant,pins", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(monkeypatch, what, module, attr, mutant, pins):
    monkeypatch.setattr(module, attr, mutant)
    caught = _failing_pins(pins)
    assert caught, "no pin fails with the mistake: %s" % what
