"""Pins for oracle selection (Algorithm 1 steps 1 and 3) and value fusion (Eq. redistribution,
Eq. weight_fusion)."""
import itertools
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import plan
from oracle import prunekv as ok


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def _bruteforce_keep(s, B):
    """Among all size-B subsets: maximal score sum, then lowest positions."""
    best = None
    for c in itertools.combinations(range(len(s)), B):
        key = (-sum(s[i] for i in c), c)
        if best is None or key < best:
            best = key
    return list(best[1])


@pytest.mark.parametrize("seed", range(6))
def test_topk_bruteforce_with_ties(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(3, 11))
    s = rng.integers(0, 4, size=n).astype(float)      # integer scores -> many exact ties
    for B in range(0, n + 1):
        order = ok.ranking(s)
        assert sorted(order[:B]) == _bruteforce_keep(list(s), B)


def test_select_invariants_shared():
    L, Hkv, n = 6, 3, 40
    s = np.abs(_rand((Hkv, n), 20))
    B, Nq, h = plan.plan_budgets(L, n, Fraction(1, 4))
    keep, drop, rank = ok.select(s, B, Nq)
    for g in range(Hkv):
        assert sorted(rank[g]) == list(range(n))
        for l in range(L):
            k, dr = keep[l][g], drop[l][g]
            assert len(k) == B[l] and list(k) == sorted(set(k))
            assert list(dr) == sorted(set(dr)) and not set(k) & set(dr)
            if B[l] > 0:
                assert len(dr) == Nq - B[l]
                assert set(k) | set(dr) == set(np.argsort(rank[g])[:Nq])
                assert all(rank[g][v] < B[l] for v in k)
            if l + 1 < L:
                assert set(keep[l + 1][g]) <= set(k)            # nested: one shared ranking


def test_select_per_layer_uses_own_ranking():
    L, Hkv, n = 3, 2, 16
    s = np.abs(_rand((L, Hkv, n), 21))
    B = [8, 6, 4]
    keep, drop, rank = ok.select(s, B, 10, rank_mode="per_layer")
    for l in range(L):
        for g in range(Hkv):
            assert list(keep[l][g]) == sorted(np.argsort(-s[l, g], kind="stable")[:B[l]])


def test_fuse_mu_one_is_plain_pruning():
    V = _rand((30, 8), 22).astype(np.float32).astype(np.float64)
    keep, drop = np.array([1, 4, 9]), np.array([0, 2, 3, 5])
    out = ok.fuse_values(V, keep, drop, mu=1.0, tau=1.0)
    assert np.array_equal(out, V[keep])                  # Sec. 3.2: mu = 1 recovers pruning


def test_fuse_mu_zero_replaces_values():
    V = _rand((12, 4), 23)
    keep, drop = np.array([0, 1]), np.array([5])
    out = ok.fuse_values(V, keep, drop, mu=0.0, tau=1.0)
    np.testing.assert_allclose(out, np.repeat(V[[5]], 2, axis=0), rtol=0, atol=0)


def test_fuse_empty_drop_set():
    V = _rand((10, 4), 24)
    keep = np.array([2, 3])
    assert np.array_equal(ok.fuse_values(V, keep, np.zeros(0, np.int64), 0.7, 1.0), V[keep])


def test_fuse_single_dropped_token():
    V = _rand((10, 6), 25)
    keep, drop = np.array([1, 2, 8]), np.array([4])
    out = ok.fuse_values(V, keep, drop, 0.7, 1.0)
    np.testing.assert_allclose(out, 0.7 * V[keep] + 0.3 * V[4], rtol=1e-15, atol=1e-15)


def test_fuse_constant_drop_rows():
    V = _rand((10, 6), 26)
    u = _rand((6,), 27)
    V[[0, 3, 5]] = u
    out = ok.fuse_values(V, np.array([1, 2]), np.array([0, 3, 5]), 0.6, 0.5)
    np.testing.assert_allclose(out, 0.6 * V[[1, 2]] + 0.4 * u, rtol=1e-14, atol=1e-14)


def test_fuse_temperature_limits():
    V = _rand((20, 5), 28)
    keep, drop = np.array([0, 1, 2]), np.arange(3, 20)
    hot = ok.fuse_values(V, keep, drop, 0.0, 1e12)                     # tau -> inf: mean of V_d
    np.testing.assert_allclose(hot, np.repeat(V[drop].mean(0, keepdims=True), 3, 0), atol=1e-9)
    cold = ok.fuse_values(V, keep, drop, 0.0, 1e-6)                    # tau -> 0: best match
    best = drop[np.argmax(V[keep] @ V[drop].T, axis=1)]
    np.testing.assert_allclose(cold, V[best], atol=1e-12)


def test_fuse_against_torch_sdpa():
    # Phi V_d is attention with queries V_k, keys = values = V_d, scale 1/tau.
    V = _rand((50, 16), 29)
    keep, drop = np.array([3, 7, 11, 20]), np.array([0, 1, 2, 30, 40, 49])
    tau, mu = 2.5, 0.7
    vk, vd = torch.from_numpy(V[keep]), torch.from_numpy(V[drop])
    o = torch.nn.functional.scaled_dot_product_attention(vk[None], vd[None], vd[None], scale=1 / tau)[0]
    np.testing.assert_allclose(ok.fuse_values(V, keep, drop, mu, tau),
                               (mu * vk + (1 - mu) * o).numpy(), rtol=1e-12, atol=1e-12)


def test_prunekv_layout_and_key_copy():
    L, Hq, Hkv, W, d, n = 4, 4, 2, 3, 8, 25
    Q, K, V = _rand((L, Hq, W, d), 30), _rand((L, Hkv, n, d), 31), _rand((L, Hkv, n, d), 32)
    B, Nq, h = plan.plan_budgets(L, n, Fraction(3, 10))
    out = ok.prunekv(Q, K, V, B, Nq)
    P = 0
    for l in range(L):
        for g in range(Hkv):
            r0 = Hkv * P + g * B[l]
            idx = out["idx_out"][r0:r0 + B[l]]
            assert np.array_equal(idx, out["keep"][l][g])
            assert np.array_equal(out["K_out"][r0:r0 + B[l]], K[l, g][idx])
        P += B[l]
    assert out["K_out"].shape[0] == Hkv * sum(B)
