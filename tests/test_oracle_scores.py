"""Pins for oracle.prunekv.token_scores (Eq. token_score; Sec. 4.4 ranking variants)."""
import numpy as np
import pytest
import torch

from oracle import prunekv as ok


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_single_row_is_textbook_softmax():
    # W = G = L = Hkv = 1: the score vector is one softmax row of q.k/sqrt(d).
    d, n = 16, 37
    q, K = _rand((1, 1, 1, d), 1), _rand((1, 1, n, d), 2)
    s = ok.token_scores(q, K)
    x = (K[0, 0] @ q[0, 0, 0]) / np.sqrt(d)
    ref = torch.softmax(torch.from_numpy(x), dim=0).numpy()
    np.testing.assert_allclose(s[0], ref, rtol=1e-13, atol=0)


def test_mass_invariant():
    # every softmax row sums to 1 -> sum_v s[g][v] = G*W (shared, 1/L mean) and per layer.
    L, Hq, Hkv, W, d, n = 3, 6, 2, 5, 8, 29
    Q, K = _rand((L, Hq, W, d), 3), _rand((L, Hkv, n, d), 4)
    s = ok.token_scores(Q, K)
    np.testing.assert_allclose(s.sum(axis=1), (Hq // Hkv) * W, rtol=1e-13)
    sl = ok.token_scores(Q, K, rank_mode="per_layer")
    np.testing.assert_allclose(sl.sum(axis=2), (Hq // Hkv) * W, rtol=1e-13)
    np.testing.assert_allclose(sl.mean(axis=0), s, rtol=1e-13)


def test_zero_queries_give_uniform_scores_and_identity_order():
    L, Hq, Hkv, W, d, n = 2, 4, 2, 3, 8, 17
    Q, K = np.zeros((L, Hq, W, d)), _rand((L, Hkv, n, d), 5)
    s = ok.token_scores(Q, K)
    np.testing.assert_allclose(s, 2 * W / n, rtol=1e-14)
    assert list(ok.ranking(s[0])) == list(range(n))


def test_against_torch_attention_with_identity_values():
    # softmax(QK^T/sqrt(d)) @ I = A: torch's SDPA (default scale 1/sqrt(d)) gives A
    # directly; its row sums over the group's queries are the scores.
    L, Hq, Hkv, W, d, n = 2, 6, 3, 4, 16, 24
    Q, K = _rand((L, Hq, W, d), 6), _rand((L, Hkv, n, d), 7)
    s = ok.token_scores(Q, K, rank_mode="per_layer")
    G = Hq // Hkv
    for l in range(L):
        q = torch.from_numpy(Q[l])                                   # [Hq][W][d]
        k = torch.from_numpy(K[l]).repeat_interleave(G, dim=0)       # head j -> KV head j // G
        eye = torch.eye(n, dtype=torch.float64).expand(Hq, n, n)
        A = torch.nn.functional.scaled_dot_product_attention(q, k, eye)
        ref = A.reshape(Hkv, G * W, n).sum(dim=1).numpy()
        np.testing.assert_allclose(s[l], ref, rtol=1e-12, atol=1e-15)


def test_gqa_mapping_contiguous_groups():
    # Queries of heads 0..G-1 are zero -> KV head 0 gets exactly uniform scores; a
    # strided mapping (j % Hkv) would mix in the random heads.
    L, Hq, Hkv, W, d, n = 1, 6, 3, 2, 8, 11
    Q = _rand((L, Hq, W, d), 8)
    Q[:, :2] = 0
    s = ok.token_scores(Q, _rand((L, Hkv, n, d), 9))
    np.testing.assert_allclose(s[0], 2 * W / n, rtol=1e-14)
    assert np.ptp(s[1]) > 1e-3 and np.ptp(s[2]) > 1e-3


def test_scale_and_layer_mean():
    # scale multiplies the logits; the shared score is the 1/L mean of per-layer scores.
    L, Hq, Hkv, W, d, n = 2, 2, 1, 3, 4, 9
    Q, K = _rand((L, Hq, W, d), 10), _rand((L, Hkv, n, d), 11)
    a = ok.token_scores(2 * Q, K, scale=0.25)
    b = ok.token_scores(Q, K, scale=0.5)
    np.testing.assert_allclose(a, b, rtol=1e-13)


def test_row_lse_mode():
    # Supplying the true log-sum-exp reproduces the softmax; lse + c scales by e^-c.
    L, Hq, Hkv, W, d, n = 2, 4, 2, 3, 8, 13
    Q, K = _rand((L, Hq, W, d), 12), _rand((L, Hkv, n, d), 13)
    sc = 1 / np.sqrt(d)
    lse = np.empty((L, Hq, W))
    G = Hq // Hkv
    for l in range(L):
        for j in range(Hq):
            x = (Q[l, j] @ K[l, j // G].T) * sc
            lse[l, j] = np.log(np.exp(x).sum(axis=1))
    np.testing.assert_allclose(ok.token_scores(Q, K, row_lse=lse), ok.token_scores(Q, K), rtol=1e-12)
    np.testing.assert_allclose(ok.token_scores(Q, K, row_lse=lse + 0.5),
                               ok.token_scores(Q, K) * np.exp(-0.5), rtol=1e-12)


def test_boosted_key_ranks_first():
    # A key aligned with every query receives the most attention in every row.
    L, Hq, Hkv, W, d, n = 1, 2, 1, 4, 8, 20
    Q = _rand((L, Hq, W, d), 14)
    K = 0.1 * _rand((L, Hkv, n, d), 15)
    K[0, 0, 7] = 5 * Q[0].reshape(-1, d).mean(axis=0) / np.linalg.norm(Q[0].reshape(-1, d).mean(axis=0))
    Q[0] = Q[0] + 2 * K[0, 0, 7] / np.linalg.norm(K[0, 0, 7])
    s = ok.token_scores(Q, K)
    assert ok.ranking(s[0])[0] == 7
