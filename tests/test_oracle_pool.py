"""The layer-by-layer oracle of the full-size parity tests (``tests/oracle_pool.py``)
gives exactly what the whole-request oracle gives, and its output check catches a
wrong key bit and a wrong value row.  CPU only (two spawn-started workers)."""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import plan as oplan
from oracle import prunekv as ok
from paper_2608_24063_gb300 import synth
from tests import oracle_pool
from tests.parity import TOL

WL = synth.scaled(synth.WORKLOADS[3], "pool check: 7B structure, 3 layers, 2 heads, 300 tokens",
                  L=3, Hq=4, Hkv=2, d=32, requests=[synth.Request(300, 8, 28, 100, 50)])


@pytest.fixture(scope="module")
def opool():
    p = oracle_pool.pool(2)
    yield p
    p.close()
    p.join()


def _whole():
    q = synth.make_q(WL, 0)
    k, v = synth.make_kv(WL, 0, q)
    return q.double().numpy(), k, v


def test_layer_scores_equal_whole_request_oracle(opool):
    Qn, k, _ = _whole()
    Kn = k.double().numpy()
    res = opool.map(oracle_pool.layer_scores, [(WL, 0, l) for l in range(WL.L)])
    per_layer = np.stack([x[2] for x in res])
    assert np.array_equal(per_layer, ok.token_scores(Qn, Kn, rank_mode="per_layer"))
    assert np.array_equal(per_layer.sum(axis=0) / WL.L, ok.token_scores(Qn, Kn))


def test_layer_outputs_accepts_oracle_and_catches_planted_errors(opool):
    Qn, k, v = _whole()
    req = WL.requests[0]
    B, Nq, h = oplan.plan_budgets(WL.L, req.n, Fraction(req.rr_num, req.rr_den))
    out = ok.prunekv(Qn, k.double().numpy(), v.double().numpy(), B, Nq)
    Hkv, d = WL.Hkv, WL.d
    tasks, P = [], 0
    for l in range(WL.L):
        b = B[l]
        if b == 0:
            continue
        keep = np.stack([out["keep"][l][g] for g in range(Hkv)])
        drop = np.stack([out["drop"][l][g] for g in range(Hkv)])
        rows = slice(Hkv * P, Hkv * (P + b))
        kbits = k[l][torch.arange(Hkv)[:, None], torch.from_numpy(keep)].reshape(Hkv * b, d)
        kbits = kbits.contiguous().view(torch.int16).numpy()
        vout = torch.from_numpy(out["V_out"][rows]).to(torch.float32).to(torch.bfloat16).double().numpy()
        tasks.append([WL, 0, l, keep, drop, kbits, vout, 0.7, 1.0, TOL[torch.bfloat16]])
        P += b
    for t in tasks:
        assert oracle_pool.layer_outputs(tuple(t))[2] == []
    # one flipped key bit and one value row off by 10%: both reported
    bad_k = list(tasks[0])
    bad_k[5] = bad_k[5].copy()
    bad_k[5][3, 7] ^= 1
    bad_v = list(tasks[-1])
    bad_v[6] = bad_v[6].copy()
    bad_v[6][2] *= 1.1
    fails = opool.map(oracle_pool.layer_outputs, [tuple(bad_k), tuple(bad_v)])
    assert any("K_out" in f for f in fails[0][2])
    assert any("V_out" in f for f in fails[1][2])
