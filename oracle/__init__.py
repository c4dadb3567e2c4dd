"""fp64 CPU oracle for the PruneKV visual-KV compression pass (VisCache, Sec. 3.2, Algorithm 1).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (the C-ABI library and its Python binding) never
calls it and shares no code with it; the only thing the two have in common is
the seeded input generator ``paper_2608_24063_gb300.synth``.

Every function here is a plain, slow restatement of the paper:

* ``plan.plan_budgets``    -- parabolic layer budgets, Eq. (parabolic) and the
  normalisation sum_l b_l = h*m that follows it; the retention product RR of
  Sec. 4 (Implementation Details).  Exact rationals (``fractions``).
* ``prunekv.token_scores`` -- Eq. (token_score): softmax attention weights
  summed over query rows and layers, 1/L mean; shared and layer-specific
  variants of Sec. 4.4 (shared vs. layer-specific ranking).
* ``prunekv.select``       -- top-q survivors and per-layer keep/drop sets,
  Algorithm 1 steps 1 and 3.
* ``prunekv.compact_keys`` -- "prune keys": kept key rows, Algorithm 1 step 3.
* ``prunekv.fuse_values``  -- Eq. (redistribution) and Eq. (weight_fusion).
* ``prunekv.prunekv``      -- Algorithm 1 end to end, dense varlen output.

All of it is pinned by ``tests/test_oracle_*.py`` against closed forms,
brute-force enumeration, invariants and library routines.  No function here is
"parity unpinned".
"""
from . import plan, prunekv  # noqa: F401
