"""Pins for oracle.quant (4-bit quantisation of the compacted cache, Appendix
"Quantization"; asymmetric per-group scale and minimum, keys per channel,
values per row)."""
import numpy as np
import pytest

from oracle import quant


def _rand(shape, seed, scale=1.0):
    return (np.random.default_rng(seed).standard_normal(shape) * scale).astype(np.float32)


def test_ladder_is_exact():
    # a group holding min + k * step for k = 0..15 (dyadic) quantises to k and back exactly
    m, s = np.float32(-1.5), np.float32(0.25)
    col = m + s * np.arange(16, dtype=np.float32)
    K = np.tile(np.concatenate([col, col[::-1]])[:, None], (1, 4))     # 32 rows, 4 channels
    codes, scale, lo = quant.quantize_keys(K)
    assert scale.tolist() == [[0.25] * 4] and lo.tolist() == [[-1.5] * 4]
    np.testing.assert_array_equal(codes[:16, 0], np.arange(16))
    np.testing.assert_array_equal(quant.dequantize_keys(codes, scale, lo), K)


def test_half_steps_round_to_even():
    # step 1: 0.5 -> 0, 1.5 -> 2, 2.5 -> 2, 3.5 -> 4 (round half to even)
    V = np.zeros((1, 32), np.float32)
    V[0, :6] = [0.0, 15.0, 0.5, 1.5, 2.5, 3.5]
    codes, scale, lo = quant.quantize_values(V)
    assert scale[0, 0] == 1.0 and lo[0, 0] == 0.0
    assert codes[0, :6].tolist() == [0, 15, 0, 2, 2, 4]


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_extremes_map_to_0_and_15(seed):
    V = _rand((5, 64), seed)
    codes, _, _ = quant.quantize_values(V)
    g = V.reshape(5, 2, 32)
    c = codes.reshape(5, 2, 32)
    for r in range(5):
        for k in range(2):
            assert c[r, k, np.argmin(g[r, k])] == 0 and c[r, k, np.argmax(g[r, k])] == 15


@pytest.mark.parametrize("seed", [4, 5])
def test_reconstruction_within_half_a_step(seed):
    K = _rand((77, 64), seed, 3.0)
    codes, scale, lo = quant.quantize_keys(K)
    err = np.abs(quant.dequantize_keys(codes, scale, lo).astype(np.float64) - K)
    step = scale[np.arange(77) // 32].astype(np.float64)
    assert (err <= 0.5 * step * (1 + 1e-5) + 1e-6).all()
    V = _rand((9, 128), seed + 10, 3.0)
    codes, scale, lo = quant.quantize_values(V)
    err = np.abs(quant.dequantize_values(codes, scale, lo).astype(np.float64) - V)
    assert (err <= 0.5 * np.repeat(scale, 32, axis=1) * (1 + 1e-5) + 1e-6).all()


def test_constant_group_is_exact():
    K = np.full((20, 8), 0.3, np.float32)
    codes, scale, lo = quant.quantize_keys(K)
    assert not codes.any() and not scale.any()
    np.testing.assert_array_equal(quant.dequantize_keys(codes, scale, lo), K)


def test_key_groups_are_per_channel():
    # scaling one channel (an outlier channel) changes only that channel's codes and params
    K = _rand((32, 16), 6)
    base = quant.quantize_keys(K)
    K2 = K.copy()
    K2[:, 5] *= 100
    got = quant.quantize_keys(K2)
    keep = [c for c in range(16) if c != 5]
    for a, b in zip(base, got):
        np.testing.assert_array_equal(a[:, keep], b[:, keep])


def test_value_groups_are_rows_of_32_channels():
    V = _rand((3, 128), 7)
    base = quant.quantize_values(V)
    V2 = V.copy()
    V2[1, 70] = 50.0                     # row 1, channel group 2 (channels 64..95)
    got = quant.quantize_values(V2)
    changed = np.argwhere(base[1] != got[1]).tolist()
    assert changed == [[1, 2]]
    diff = np.argwhere(base[0] != got[0])
    assert set(map(tuple, diff[:, :1].tolist())) == {(1,)} and diff[:, 1].min() >= 64 and diff[:, 1].max() < 96


def test_ragged_last_key_group():
    # 40 rows: groups of 32 and 8 rows; a constant tail group has scale 0
    K = _rand((40, 4), 8)
    K[32:] = 2.0
    codes, scale, lo = quant.quantize_keys(K)
    assert scale.shape == (2, 4) and not scale[1].any() and (lo[1] == 2.0).all()
    assert not codes[32:].any()


def test_pack_layout():
    codes = np.array([[1, 2, 3, 4], [15, 0, 0, 15]], np.uint8)
    packed = quant.pack(codes)
    assert packed.tolist() == [[0x21, 0x43], [0x0F, 0xF0]]
    np.testing.assert_array_equal(quant.unpack(packed), codes)


def test_affine_change_keeps_the_codes():
    # x -> 4x - 1 (exact in float32 for these dyadic values) scales the step, not the codes
    V = (np.random.default_rng(9).integers(-64, 64, (4, 64)) / 8).astype(np.float32)
    a = quant.quantize_values(V)[0]
    b = quant.quantize_values(4 * V - 1)[0]
    np.testing.assert_array_equal(a, b)


def test_segment_order():
    # rows are request-major, then layer, then KV head; empty layers hold no rows
    segs = quant.segments([[3, 0], [2, 1]], Hkv=2)
    assert segs == [(0, 3), (3, 3), (6, 0), (6, 0), (6, 2), (8, 2), (10, 1), (11, 1)]


def test_cache_params_stack_over_segments():
    rng = np.random.default_rng(10)
    B = [[40, 3], [33, 0]]
    rows = sum(2 * sum(b) for b in B)
    K = rng.standard_normal((rows, 64)).astype(np.float32)
    V = rng.standard_normal((rows, 64)).astype(np.float32)
    kc, vc, kp, vp = quant.quantize_cache(K, V, B, Hkv=2)
    # groups: 2 x (2 + 1) for request 0, 2 x 2 for request 1
    assert kp.shape == (10, 64, 2) and vp.shape == (rows, 2, 2)
    assert kc.shape == (rows, 32) and vc.shape == (rows, 32)
    # the third segment (request 0, layer 1, head 0) starts at row 80 and is
    # group 4 in the stacking order: make it constant and find it there alone
    K2 = K.copy()
    K2[80:83] = 7.0
    kp2 = quant.quantize_cache(K2, V, B, Hkv=2)[2]
    assert (kp2[4, :, 0] == 0).all() and (kp2[4, :, 1] == 7).all()
    assert [g for g in range(10) if (kp2[g, :, 1] == 7).all()] == [4]
