"""Pins for oracle.decode (decode attention over the compressed cache, Sec. 2 / 3.2)."""
import numpy as np
import pytest
import torch

from oracle import decode


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_against_torch_sdpa():
    # scaled dot-product attention with GQA, one query row per head
    Hq, Hkv, d, B, T = 8, 2, 16, 37, 5
    q, Kv, Vv, Kt, Vt = _rand((Hq, d), 1), _rand((Hkv, B, d), 2), _rand((Hkv, B, d), 3), \
        _rand((Hkv, T, d), 4), _rand((Hkv, T, d), 5)
    got = decode.decode_attention(q, Kv, Vv, Kt, Vt)
    K = torch.from_numpy(np.concatenate([Kv, Kt], axis=1)).repeat_interleave(Hq // Hkv, dim=0)
    V = torch.from_numpy(np.concatenate([Vv, Vt], axis=1)).repeat_interleave(Hq // Hkv, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q)[:, None, :], K, V)[:, 0]
    np.testing.assert_allclose(got, ref.numpy(), rtol=0, atol=1e-13)


def test_single_key_returns_its_value():
    q, K, V = _rand((4, 8), 6), _rand((2, 1, 8), 7), _rand((2, 1, 8), 8)
    got = decode.decode_attention(q, K, V)
    np.testing.assert_array_equal(got, np.repeat(V[:, 0], 2, axis=0))


def test_equal_logits_average_the_values():
    # identical keys give every key the same weight: the output is the mean value
    q = _rand((2, 8), 9)
    K = np.repeat(_rand((1, 1, 8), 10), 6, axis=1)
    V = _rand((1, 6, 8), 11)
    got = decode.decode_attention(q, K, V)
    np.testing.assert_allclose(got, np.repeat(V[0].mean(axis=0)[None], 2, axis=0), rtol=1e-13, atol=1e-14)


def test_evicted_layer_uses_text_only_or_gives_zeros():
    q = _rand((4, 8), 12)
    empty = np.zeros((2, 0, 8))
    Kt, Vt = _rand((2, 3, 8), 13), _rand((2, 3, 8), 14)
    np.testing.assert_allclose(decode.decode_attention(q, empty, empty, Kt, Vt),
                               decode.decode_attention(q, Kt, Vt), rtol=0, atol=0)
    assert not decode.decode_attention(q, empty, empty).any()


def test_key_order_does_not_matter():
    # attention is a set function of the (key, value) pairs
    q, K, V = _rand((4, 8), 15), _rand((2, 20, 8), 16), _rand((2, 20, 8), 17)
    perm = np.random.default_rng(18).permutation(20)
    np.testing.assert_allclose(decode.decode_attention(q, K[:, perm], V[:, perm]),
                               decode.decode_attention(q, K, V), rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("G", [1, 4, 7])
def test_gqa_map_contiguous_groups(G):
    # query head j reads KV head j // G: moving a KV head's data moves exactly its group
    Hkv, d = 3, 8
    q, K, V = _rand((G * Hkv, d), 19), _rand((Hkv, 9, d), 20), _rand((Hkv, 9, d), 21)
    base = decode.decode_attention(q, K, V)
    got = decode.decode_attention(q, K[::-1].copy(), V[::-1].copy())
    for j in range(G * Hkv):
        g = j // G
        alone = decode.decode_attention(q[j:j + 1], K[g:g + 1], V[g:g + 1])[0]
        np.testing.assert_allclose(base[j], alone, rtol=1e-13, atol=1e-14)
    assert not np.allclose(base, got) or Hkv == 1


def test_two_keys_closed_form():
    # keys k1, k2 with scaled logits differing by delta: the output is the
    # logistic mix sigma(delta) v1 + (1 - sigma(delta)) v2, whatever d is
    d = 16
    q = np.zeros((1, d))
    q[0, 0] = 2.0
    K = np.zeros((1, 2, d))
    K[0, 0, 0] = 3.0                      # logit 6 / sqrt(16) = 1.5
    K[0, 1, 0] = -1.0                     # logit -2 / 4 = -0.5
    V = np.zeros((1, 2, d))
    V[0, 0, :] = 1.0
    V[0, 1, :] = -3.0
    w = 1.0 / (1.0 + np.exp(-2.0))        # delta = 2
    got = decode.decode_attention(q, K, V)
    np.testing.assert_allclose(got[0], w * 1.0 + (1 - w) * -3.0, rtol=0, atol=1e-15)
