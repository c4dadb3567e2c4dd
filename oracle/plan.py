"""Oracle planner: parabolic layer budgets in exact rational arithmetic.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Paper passages (VisCache, Sec. 3.2 "Token Scoring and Parabolic Budget
Allocation"; Sec. 4 "Implementation Details"; Algorithm 1 step 2):

* layers l > h are fully evicted; for l in [1, h] the budget proportion is
  b_l = 1 - (l-1)^2 / (2 (h-1)^2), so b_1 = 1 and b_h = 1/2   (Eq. parabolic);
* {b_l} is normalised so that sum_{l<=h} b_l = h*m                      (after Eq. parabolic);
* RR = p * q * (h/L) * m with p = 1 here (no frame filtering), defaults
  h = 3L/4, m = 0.75                                                     (Sec. 4).

Readings where the paper is silent:

* total kept (token, layer) pairs per KV head  T = round(RR * n * L), so that
  sum_l B_l equals the stated retention times tokens times layers;
* the normalised proportions scale the survivors Nq = q*n of the top-q step:
  B_l = b_l * h*m / (sum b) * Nq, hence sum_l B_l = h*m*q*n = T and
  Nq = T / (h*m) (rounded, at least B_1, at most n);
* integer budgets by largest remainder on exact rationals, ties to the lower l;
* h = round(3L/4) clamped to [min(2, L), L]; for h = 1 the single layer keeps
  proportion 1 (the formula is 0/0 there);
* round() is round-half-up on exact rationals.

Budget schedules of the ablation table (Sec. 4.3, Table "ablation": "uniform
budget per layer", "arithmetic progression", "geometric progression across
four layer blocks"); the table names them only, so each replaces b_l and
keeps everything else (layers l > h evicted, the normalisation to h*m, T,
largest remainder, Nq):

* fixed: b_l = 1;
* arithmetic: b_l = 1 - (l-1)/(2(h-1)), the parabola's end points 1 and 1/2;
* geometric: layers 1..h in min(4, h) contiguous blocks, sizes differing by
  at most one (larger blocks first), block k with b = (1/2)^k;
* all of them b = [1] when h = 1.

Drop set: "survivors" (default) drops the survivors minus the keep set;
"all" drops every token not kept (the other reading of V_d's n - b_l rows in
Sec. 3.2), i.e. Nq = n.
"""
from __future__ import annotations

from fractions import Fraction
from math import floor
from typing import List, Optional, Tuple


def round_half_up(x: Fraction) -> int:
    return floor(x + Fraction(1, 2))


def default_h(L: int) -> int:
    """Truncation layer h = 3L/4 (Sec. 4), rounded, within [min(2, L), L]."""
    h = round_half_up(Fraction(3 * L, 4))
    return max(min(2, L), min(h, L))


def parabolic_proportions(h: int) -> List[Fraction]:
    """b_l for l = 1..h (Eq. parabolic); [1] when h == 1."""
    if h == 1:
        return [Fraction(1)]
    return [1 - Fraction((l - 1) ** 2, 2 * (h - 1) ** 2) for l in range(1, h + 1)]


SCHEDULES = ("parabola", "fixed", "arithmetic", "geometric")


def schedule_proportions(h: int, schedule: str = "parabola") -> List[Fraction]:
    """b_l for l = 1..h under one of the budget schedules (see the module notes)."""
    if schedule not in SCHEDULES:
        raise ValueError("unknown schedule %r" % schedule)
    if schedule == "parabola":
        return parabolic_proportions(h)
    if h == 1:
        return [Fraction(1)]
    if schedule == "fixed":
        return [Fraction(1)] * h
    if schedule == "arithmetic":
        return [1 - Fraction(l - 1, 2 * (h - 1)) for l in range(1, h + 1)]
    nb = min(4, h)
    per, extra = divmod(h, nb)
    b = []
    for k in range(nb):
        b += [Fraction(1, 2 ** k)] * (per + (1 if k < extra else 0))
    return b


def normalised_proportions(h: int, m: Fraction, schedule: str = "parabola") -> List[Fraction]:
    """b_l rescaled so that their sum is h*m (normalisation after Eq. parabolic)."""
    b = schedule_proportions(h, schedule)
    s = sum(b)
    return [x * h * m / s for x in b]


def apportion(total: int, weights: List[Fraction]) -> List[int]:
    """Largest-remainder split of ``total`` in proportion to ``weights`` (ties -> lower index)."""
    W = sum(weights)
    quotas = [total * w / W for w in weights]
    base = [floor(q) for q in quotas]
    left = total - sum(base)
    order = sorted(range(len(weights)), key=lambda i: (-(quotas[i] - base[i]), i))
    for i in order[:left]:
        base[i] += 1
    return base


class Infeasible(ValueError):
    pass


def plan_budgets(L: int, n: int, rr: Fraction, h: Optional[int] = None,
                 m: Fraction = Fraction(3, 4), schedule: str = "parabola",
                 drop: str = "survivors") -> Tuple[List[int], int, int]:
    """Integer budgets B[0..L-1], survivors Nq and truncation layer h.

    Raises ``Infeasible`` when the largest layer budget would exceed n.
    """
    if drop not in ("survivors", "all"):
        raise ValueError("unknown drop set %r" % drop)
    if L < 1 or n < 1:
        raise ValueError("L and n must be >= 1")
    if not (0 < rr <= 1) or not (0 < m <= 1):
        raise ValueError("rr and m must be in (0, 1]")
    if h is None or h == 0:
        h = default_h(L)
    if not 1 <= h <= L:
        raise ValueError("h must be in [1, L]")
    T = round_half_up(rr * n * L)
    B = apportion(T, normalised_proportions(h, m, schedule)) + [0] * (L - h)
    if B[0] > n:
        raise Infeasible("retention %s cannot be met with h=%d, m=%s" % (rr, h, m))
    Nq = round_half_up(Fraction(T) / (h * m))
    Nq = min(n, max(Nq, B[0]))
    if drop == "all":
        Nq = n
    return B, Nq, h
