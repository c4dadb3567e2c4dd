"""Writes tests/golden/budgets.json from the oracle planner only.

Run from the repository root:  python tests/golden/make_golden.py
The cases are the five workloads' (L, n, RR) plus edge shapes; the values
come from oracle.plan.plan_budgets (exact rationals), never from the CUDA path.
"""
import json
import os
import sys
from fractions import Fraction

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
from oracle import plan  # noqa: E402

CASES = [
    # (L, n, rr_num, rr_den)
    (1, 1024, 25, 100), (28, 3136, 28, 100), (28, 12544, 19, 100), (80, 32768, 22, 100),
    (28, 2048, 19, 100), (28, 16384, 28, 100), (28, 9999, 23, 100), (2, 5, 1, 2),
    (3, 1, 1, 10), (64, 4096, 28, 100), (128, 65536, 19, 100), (7, 129, 37, 100),
]


def main():
    out = []
    for L, n, a, b in CASES:
        B, Nq, h = plan.plan_budgets(L, n, Fraction(a, b))
        out.append(dict(L=L, n=n, rr_num=a, rr_den=b, B=B, Nq=Nq, h=h))
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "budgets.json")
    with open(path, "w") as f:
        json.dump({"source": "oracle.plan.plan_budgets", "cases": out}, f, indent=0)
        f.write("\n")


if __name__ == "__main__":
    main()
