"""Oracle for the scout's keyframe selection, Eq. (mmr), in float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Sec. 3.1 ("Prompt-Aware Scout for Temporal Redundancy Filtering"): with
frame embeddings h_f and a prompt embedding h_t in a shared space, the MMR
score of a candidate frame f given the selected set Omega is

    lambda * sim(h_f, h_t) - (1 - lambda) * max_{f' in Omega} sim(h_f, h_f'),

sim the cosine similarity; the highest-scoring frame joins Omega until the
frame retention ratio p is reached (lambda = 0.7 in Sec. 4).

Readings where the paper is silent:

* the redundancy term is 0 while Omega is empty, so the first frame is the
  most prompt-relevant one;
* "until p is reached" stops at k = ceil(p * F) frames (at least 1) of F;
* ties go to the lower frame index;
* the cosine similarity with a zero vector is 0;
* the keyframes are returned in selection order and, as the video's frame
  subset, in ascending frame order.
"""
from __future__ import annotations

from fractions import Fraction
from math import ceil
from typing import Tuple

import numpy as np


def keyframe_count(F: int, p: Fraction) -> int:
    """k = ceil(p * F), at least 1, at most F."""
    return max(1, min(F, ceil(Fraction(p) * F)))


def cosine_unit(x: np.ndarray) -> np.ndarray:
    """Rows scaled to unit length (zero rows stay zero, so their similarities are 0)."""
    norm = np.sqrt((x * x).sum(axis=-1, keepdims=True))
    return np.divide(x, norm, out=np.zeros_like(x), where=norm > 0)


def mmr_select(H: np.ndarray, h_t: np.ndarray, lam: float, k: int) -> Tuple[np.ndarray, np.ndarray]:
    """Greedy MMR over the frames H [F][d] for the prompt h_t [d].

    Returns (order, gains): the k selected frames in selection order and the
    MMR score each had when it was picked.
    """
    Hn = cosine_unit(np.asarray(H, dtype=np.float64))
    tn = cosine_unit(np.asarray(h_t, dtype=np.float64)[None, :])[0]
    F = Hn.shape[0]
    rel = Hn @ tn                          # sim(h_f, h_t)
    red = np.zeros(F)                      # max_{f' in Omega} sim(h_f, h_f'), 0 for empty Omega
    chosen = np.zeros(F, dtype=bool)
    order, gains = [], []
    for step in range(k):
        score = lam * rel - (1.0 - lam) * red
        score[chosen] = -np.inf
        f = int(np.argmax(score))          # first maximum: the lower index wins ties
        order.append(f)
        gains.append(score[f])
        chosen[f] = True
        sims = Hn @ Hn[f]
        red = sims if step == 0 else np.maximum(red, sims)
    return np.array(order, dtype=np.int64), np.array(gains)


def scout(H: np.ndarray, h_t: np.ndarray, lam: float, p: Fraction):
    """Keyframes of one video: (order, keyframes ascending, gains)."""
    k = keyframe_count(H.shape[0], p)
    order, gains = mmr_select(H, h_t, lam, k)
    return order, np.sort(order), gains
