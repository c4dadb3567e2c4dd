"""Oracle for 4-bit quantisation of the compacted cache (Appendix
"Quantization": the compressed visual KV combined with 4-bit KV cache
quantisation, KIVI-style).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

The paper combines its compressed cache with 4-bit quantisers without
defining one; the reading taken here is the asymmetric round-to-nearest
form with a per-group scale and minimum:

    scale = (max - min) / 15,   code = clamp(rint((x - min) / scale), 0, 15),
    x_hat = code * scale + min,

with keys grouped per channel over 32 consecutive kept rows of one
(request, layer, KV head) segment (the last group of a segment may be
shorter) and values grouped per row over 32 consecutive channels.  A group
whose values are all equal has scale 0 and codes 0.

The code is an integer decided by floating point, so it is decided here in
the kernel's precision: float32 operations in the order written above
(min and max are exact; the subtraction, the division and rint round to
nearest even).  Reconstruction is computed in float64 (code * scale is exact
there) and rounded once to float32, which is what a fused multiply-add does.
Codes are packed two per byte, the even channel in the low nibble.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np

GROUP = 32
LEVELS = 15


def group_params(x: np.ndarray, axis: int) -> Tuple[np.ndarray, np.ndarray]:
    """(scale, min) in float32 of the values of x along `axis`."""
    x = np.asarray(x, dtype=np.float32)
    lo = x.min(axis=axis)
    hi = x.max(axis=axis)
    scale = (hi - lo) / np.float32(LEVELS)
    return scale.astype(np.float32), lo.astype(np.float32)


def codes_of(x: np.ndarray, scale: np.ndarray, lo: np.ndarray) -> np.ndarray:
    """4-bit codes of x (float32 arithmetic) given broadcastable scale and min."""
    x = np.asarray(x, dtype=np.float32)
    with np.errstate(divide="ignore", invalid="ignore"):
        q = np.rint((x - lo) / scale)
    q = np.where(scale > 0, q, 0.0)
    return np.clip(q, 0, LEVELS).astype(np.uint8)


def reconstruct(codes: np.ndarray, scale: np.ndarray, lo: np.ndarray) -> np.ndarray:
    """code * scale + min, exact in float64, rounded once to float32."""
    return (codes.astype(np.float64) * scale.astype(np.float64) + lo.astype(np.float64)).astype(np.float32)


def pack(codes: np.ndarray) -> np.ndarray:
    """[rows][d] codes -> [rows][d/2] bytes, the even channel in the low nibble."""
    codes = np.asarray(codes, dtype=np.uint8)
    return (codes[:, 0::2] | (codes[:, 1::2] << 4)).astype(np.uint8)


def unpack(packed: np.ndarray) -> np.ndarray:
    packed = np.asarray(packed, dtype=np.uint8)
    out = np.empty((packed.shape[0], packed.shape[1] * 2), dtype=np.uint8)
    out[:, 0::2] = packed & 0x0F
    out[:, 1::2] = packed >> 4
    return out


def quantize_keys(K: np.ndarray) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """One segment K [B][d]: per-channel groups of GROUP rows.

    Returns (codes [B][d], scale [ceil(B/GROUP)][d], min [ceil(B/GROUP)][d]).
    """
    K = np.asarray(K, dtype=np.float32)
    B, d = K.shape
    nb = (B + GROUP - 1) // GROUP
    scale = np.zeros((nb, d), np.float32)
    lo = np.zeros((nb, d), np.float32)
    codes = np.zeros((B, d), np.uint8)
    for b in range(nb):
        blk = K[b * GROUP:(b + 1) * GROUP]
        s, m = group_params(blk, axis=0)
        scale[b], lo[b] = s, m
        codes[b * GROUP:(b + 1) * GROUP] = codes_of(blk, s[None, :], m[None, :])
    return codes, scale, lo


def quantize_values(V: np.ndarray) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Rows V [R][d]: per-row groups of GROUP channels.

    Returns (codes [R][d], scale [R][d/GROUP], min [R][d/GROUP]).
    """
    V = np.asarray(V, dtype=np.float32)
    R, d = V.shape
    g = V.reshape(R, d // GROUP, GROUP)
    scale, lo = group_params(g, axis=2)
    codes = codes_of(g, scale[:, :, None], lo[:, :, None]).reshape(R, d)
    return codes, scale, lo


def dequantize_keys(codes, scale, lo) -> np.ndarray:
    rows = np.arange(codes.shape[0]) // GROUP
    return reconstruct(codes, scale[rows], lo[rows])


def dequantize_values(codes, scale, lo) -> np.ndarray:
    R, d = codes.shape
    s = np.repeat(scale, GROUP, axis=1)
    m = np.repeat(lo, GROUP, axis=1)
    return reconstruct(codes, s, m)


def segments(B_per_request: Sequence[Sequence[int]], Hkv: int) -> List[Tuple[int, int]]:
    """(first row, rows) of every (request, layer, KV head) segment of the
    compacted cache, in its row order (request, then layer, then KV head)."""
    out, row = [], 0
    for B in B_per_request:
        for b in B:
            for _ in range(Hkv):
                out.append((row, b))
                row += b
    return out


def quantize_cache(K_out: np.ndarray, V_out: np.ndarray, B_per_request, Hkv: int):
    """The whole compacted cache: packed codes and (scale, min) pairs.

    K params are stacked over the segments' groups in row order:
    [sum_segments ceil(B/GROUP)][d][2]; V params are [rows][d/GROUP][2].
    """
    kc = np.zeros(K_out.shape, np.uint8)
    kp = []
    for row0, b in segments(B_per_request, Hkv):
        if b == 0:
            continue
        c, s, m = quantize_keys(K_out[row0:row0 + b])
        kc[row0:row0 + b] = c
        kp.append(np.stack([s, m], axis=-1))
    vc, vs, vm = quantize_values(V_out)
    kparams = np.concatenate(kp) if kp else np.zeros((0, K_out.shape[1], 2), np.float32)
    return pack(kc), pack(vc), kparams, np.stack([vs, vm], axis=-1)
