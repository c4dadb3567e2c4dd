"""Oracle planner: parabolic layer budgets in exact rational arithmetic.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Paper passages (VisCache, Sec. 3.2 "Token Scoring and Parabolic Budget
Allocation"; Sec. 4 "Implementation Details"; Algorithm 1 step 2):

* layers l > h are fully evicted; for l in [1, h] the budget proportion is
  b_l = 1 - (l-1)^2 / (2 (h-1)^2), so b_1 = 1 and b_h = 1/2   (Eq. parabolic);
* {b_l} is normalised so that sum_{l<=h} b_l = h*m                      (after Eq. parabolic);
* RR = p * q * (h/L) * m with p = 1 here (no frame filtering), defaults
  h = 3L/4, m = 0.75                                                     (Sec. 4).

Readings where the paper is silent (each listed in the design doc):

* total kept (token, layer) pairs per KV head  T = round(RR * n * L), so that
  sum_l B_l equals the stated retention times tokens times layers;
* the normalised proportions scale the survivors Nq = q*n of the top-q step:
  B_l = b_l * h*m / (sum b) * Nq, hence sum_l B_l = h*m*q*n = T and
  Nq = T / (h*m) (rounded, at least B_1, at most n);
* integer budgets by largest remainder on exact rationals, ties to the lower l;
* h = round(3L/4) clamped to [min(2, L), L]; for h = 1 the single layer keeps
  proportion 1 (the formula is 0/0 there);
* round() is round-half-up on exact rationals.
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


def normalised_proportions(h: int, m: Fraction) -> List[Fraction]:
    """b_l rescaled so that their sum is h*m (normalisation after Eq. parabolic)."""
    b = parabolic_proportions(h)
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
                 m: Fraction = Fraction(3, 4)) -> Tuple[List[int], int, int]:
    """Integer budgets B[0..L-1], survivors Nq and truncation layer h.

    Raises ``Infeasible`` when the largest layer budget would exceed n.
    """
    if L < 1 or n < 1:
        raise ValueError("L and n must be >= 1")
    if not (0 < rr <= 1) or not (0 < m <= 1):
        raise ValueError("rr and m must be in (0, 1]")
    if h is None or h == 0:
        h = default_h(L)
    if not 1 <= h <= L:
        raise ValueError("h must be in [1, L]")
    T = round_half_up(rr * n * L)
    B = apportion(T, normalised_proportions(h, m)) + [0] * (L - h)
    if B[0] > n:
        raise Infeasible("retention %s cannot be met with h=%d, m=%s" % (rr, h, m))
    Nq = round_half_up(Fraction(T) / (h * m))
    Nq = min(n, max(Nq, B[0]))
    return B, Nq, h
