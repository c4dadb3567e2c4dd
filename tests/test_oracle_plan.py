"""Pins for the oracle planner (Eq. parabolic, its normalisation, the RR product of Sec. 4)."""
import itertools
import json
import os
from fractions import Fraction
from math import floor

import pytest

from oracle import plan

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_parabolic_endpoints_from_paper():
    # Sec. 3.2, right after Eq. (parabolic): b_1 = 1 and b_h = 0.5.
    for h in range(2, 130):
        b = plan.parabolic_proportions(h)
        assert b[0] == 1 and b[-1] == Fraction(1, 2)
        # "decaying slowly in early layers and more steeply in deeper layers": concave decrease
        steps = [b[i] - b[i + 1] for i in range(h - 1)]
        assert all(s > 0 for s in steps)
        assert all(steps[i] < steps[i + 1] for i in range(h - 2))


def test_parabolic_matches_formula_pointwise():
    # b_l = 1 - (l-1)^2 / (2 (h-1)^2), evaluated independently in floating point.
    for h in (2, 3, 7, 21, 60):
        b = plan.parabolic_proportions(h)
        for l in range(1, h + 1):
            assert abs(float(b[l - 1]) - (1 - (l - 1) ** 2 / (2.0 * (h - 1) ** 2))) < 1e-15


def test_normalisation_sums_to_h_m():
    # Sec. 3.2: {b_l} normalised so that sum_{l<=h} b_l = h * m.
    for h, m in itertools.product((1, 2, 5, 21, 60), (Fraction(3, 4), Fraction(1, 2), Fraction(1))):
        assert sum(plan.normalised_proportions(h, m)) == h * m


def test_default_truncation_from_paper():
    # Appendix "How To Determine the Truncation Layer": 48 of 64 layers = 3/4 depth.
    assert plan.default_h(64) == 48
    assert plan.default_h(28) == 21 and plan.default_h(80) == 60
    assert plan.default_h(1) == 1 and plan.default_h(2) == 2


def test_truncation_rounds_half_up():
    # The paper gives h = 3L/4 only where it is whole; the reading for other
    # depths rounds half up (4.5 -> 5, 7.5 -> 8, 22.5 -> 23, 5.25 -> 5).
    assert [plan.default_h(L) for L in (6, 10, 30, 7)] == [5, 8, 23, 5]


def test_rr_product_example_from_paper():
    # Sec. 4: p=0.75, q=0.67, h=3L/4, m=0.75 give RR ~ 28%.
    p, q, m = Fraction(3, 4), Fraction(67, 100), Fraction(3, 4)
    L = 64
    h = plan.default_h(L)
    rr = p * q * Fraction(h, L) * m
    assert abs(float(rr) - 0.28) < 0.005
    # With p = 1 the planner inverts the product: Nq = q*n survivors.
    n = 10000
    B, Nq, hh = plan.plan_budgets(L, n, q * Fraction(h, L) * m, h=h, m=m)
    assert hh == h and Nq == round(q * n)


@pytest.mark.parametrize("L,n,rr", [
    (1, 1024, Fraction(25, 100)), (28, 3136, Fraction(28, 100)), (28, 12544, Fraction(19, 100)),
    (80, 32768, Fraction(22, 100)), (28, 2048, Fraction(23, 100)), (5, 7, Fraction(1, 3)),
    (3, 1, Fraction(1, 10)), (64, 1000, Fraction(56, 100)),
])
def test_budget_closed_forms(L, n, rr):
    B, Nq, h = plan.plan_budgets(L, n, rr)
    T = floor(rr * n * L + Fraction(1, 2))
    assert sum(B) == T                                   # sum_l B_l = round(RR n L)
    assert all(b == 0 for b in B[h:])                    # layers l > h evicted
    assert all(B[i] >= B[i + 1] for i in range(L - 1))   # non-increasing
    assert B[0] <= Nq <= n
    if h >= 2 and B[h - 1] > 10:
        assert abs(B[0] - 2 * B[h - 1]) <= 2            # b_1 : b_h = 2 : 1
    # each budget within one unit of its exact quota
    w = plan.parabolic_proportions(h)
    for l in range(h):
        assert abs(B[l] - T * w[l] / sum(w)) < 1


def test_largest_remainder_bruteforce():
    # Exhaustive over all integer splits with the right total: the chosen one
    # minimises the sum of |B_l - quota_l| and, among minimisers, favours lower l.
    for T, ws in [(7, [3, 2, 2]), (10, [1, 1, 1]), (5, [4, 3, 2, 1]), (13, [5, 5, 3])]:
        wf = [Fraction(x) for x in ws]
        got = plan.apportion(T, wf)
        quotas = [T * x / sum(wf) for x in wf]
        best = None
        for cand in itertools.product(*(range(floor(q), floor(q) + 2) for q in quotas)):
            if sum(cand) != T:
                continue
            cost = sum(abs(c - q) for c, q in zip(cand, quotas))
            key = (cost, [-c for c in cand])
            if best is None or key < best[0]:
                best = (key, list(cand))
        assert got == best[1], (T, ws, got, best)


def test_infeasible():
    with pytest.raises(plan.Infeasible):
        plan.plan_budgets(4, 10, Fraction(1), h=2, m=Fraction(1, 2))


def test_golden_budgets_match_oracle():
    with open(os.path.join(GOLDEN, "budgets.json")) as f:
        gold = json.load(f)
    for case in gold["cases"]:
        B, Nq, h = plan.plan_budgets(case["L"], case["n"], Fraction(case["rr_num"], case["rr_den"]))
        assert (B, Nq, h) == (case["B"], case["Nq"], case["h"])


# ---------------------------------------------------------------------------
# budget schedules of the ablation table (readings in oracle/plan.py)

SCHED_CASES = [(28, 12544, Fraction(19, 100)), (28, 3136, Fraction(28, 100)),
               (80, 32768, Fraction(22, 100)), (5, 97, Fraction(1, 3)), (6, 1000, Fraction(1, 4)),
               (3, 50, Fraction(2, 5))]


@pytest.mark.parametrize("schedule", plan.SCHEDULES)
@pytest.mark.parametrize("L,n,rr", SCHED_CASES)
def test_schedule_closed_forms(schedule, L, n, rr):
    B, Nq, h = plan.plan_budgets(L, n, rr, schedule=schedule)
    T = floor(rr * n * L + Fraction(1, 2))
    assert sum(B) == T                                   # same total for every schedule
    assert all(b == 0 for b in B[h:])                    # layers l > h evicted
    assert all(B[i] >= B[i + 1] for i in range(L - 1))   # non-increasing
    assert min(n, max(B[0], floor(Fraction(T) / (h * Fraction(3, 4)) + Fraction(1, 2)))) == Nq


def test_fixed_schedule_is_uniform():
    # equal quotas: T // h each, the remainder to the lowest layers
    for L, n, rr in SCHED_CASES:
        B, _, h = plan.plan_budgets(L, n, rr, schedule="fixed")
        T = sum(B)
        assert B[:h] == [T // h + (1 if l < T % h else 0) for l in range(h)]


def test_arithmetic_schedule_is_linear_from_one_to_half():
    for h in (2, 3, 7, 21, 60):
        b = plan.schedule_proportions(h, "arithmetic")
        assert b[0] == 1 and b[-1] == Fraction(1, 2)
        steps = {b[i] - b[i + 1] for i in range(h - 1)}
        assert steps == {Fraction(1, 2 * (h - 1))}
    B, _, h = plan.plan_budgets(28, 12544, Fraction(19, 100), schedule="arithmetic")
    diffs = [B[i] - B[i + 1] for i in range(h - 1)]
    assert max(diffs) - min(diffs) <= 2                  # integer budgets still linear


def test_geometric_schedule_blocks():
    for h in (1, 2, 3, 4, 5, 21, 60):
        b = plan.schedule_proportions(h, "geometric")
        assert len(b) == h
        runs = [len(list(g)) for _, g in itertools.groupby(b)]
        assert len(runs) == min(4, h)                                  # four blocks (fewer if h < 4)
        assert max(runs) - min(runs) <= 1 and runs == sorted(runs, reverse=True)
        levels = [k for k, _ in itertools.groupby(b)]
        assert levels[0] == 1 and all(levels[i + 1] * 2 == levels[i] for i in range(len(levels) - 1))


def test_schedules_coincide_for_one_layer():
    for schedule in plan.SCHEDULES:
        assert plan.plan_budgets(1, 1024, Fraction(1, 4), schedule=schedule) == ([256], 341, 1)


def test_drop_all_keeps_budgets_and_takes_every_token():
    for L, n, rr in SCHED_CASES:
        for schedule in plan.SCHEDULES:
            B, Nq, h = plan.plan_budgets(L, n, rr, schedule=schedule)
            B2, Nq2, h2 = plan.plan_budgets(L, n, rr, schedule=schedule, drop="all")
            assert (B2, h2) == (B, h) and Nq2 == n
