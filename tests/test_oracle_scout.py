"""Pins for oracle.scout (Eq. mmr, Sec. 3.1; lambda = 0.7, p = 0.75 in Sec. 4)."""
from fractions import Fraction
import numpy as np
import pytest

from oracle import scout


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_keyframe_count():
    # "until a target retention ratio p is reached": ceil(p F), at least one frame
    assert scout.keyframe_count(64, Fraction(3, 4)) == 48          # the paper's p on 64 frames
    assert scout.keyframe_count(10, Fraction(1, 3)) == 4
    assert scout.keyframe_count(7, Fraction(1)) == 7
    assert scout.keyframe_count(100, Fraction(1, 1000)) == 1


def test_lambda_one_is_top_k_by_relevance():
    # only the prompt term is left: a sort by cosine relevance, lower index on ties
    H, t = _rand((40, 16), 1), _rand(16, 2)
    H[7] = H[3]                                                    # an exact tie
    order, _ = scout.mmr_select(H, t, 1.0, 12)
    rel = (H @ t) / (np.linalg.norm(H, axis=1) * np.linalg.norm(t))
    ref = np.lexsort((np.arange(40), -rel))[:12]
    assert order.tolist() == ref.tolist()


def test_lambda_zero_is_farthest_point_selection():
    # lambda = 0: every first score is 0, so frame 0 wins the tie; then each
    # pick minimises the largest cosine to the chosen frames (greedy
    # farthest-point selection).  Eight directions on the axes and diagonals:
    # 0 deg, then 180 deg (cosine -1), then 90 deg (cosine 0 to both; 270 deg
    # ties and has the higher index), then 270 deg (the only one left at 0).
    H = np.array([[1, 0], [1, 1], [0, 1], [-1, 1], [-1, 0], [-1, -1], [0, -1], [1, -1]], float)
    order, _ = scout.mmr_select(H, np.array([1.0, 0.0]), 0.0, 4)
    assert order.tolist() == [0, 4, 2, 6]


def test_duplicate_frame_is_penalised_by_its_twin():
    # frames a, a, b with the prompt along a: after a, its twin scores
    # lambda - (1 - lambda) = 0.4, b (orthogonal) scores 0 - 0 = 0 -> the twin;
    # with lambda = 0.4 the twin scores -0.2 and b wins.
    H = np.array([[1.0, 0.0], [1.0, 0.0], [0.0, 1.0]])
    t = np.array([1.0, 0.0])
    assert scout.mmr_select(H, t, 0.7, 2)[0].tolist() == [0, 1]
    assert scout.mmr_select(H, t, 0.4, 2)[0].tolist() == [0, 2]


def test_gains_closed_form():
    # the recorded gain of each pick is lambda*rel - (1-lambda)*max cosine to the earlier picks
    H, t = _rand((20, 8), 3), _rand(8, 4)
    lam = 0.7
    order, gains = scout.mmr_select(H, t, lam, 6)
    Hn = H / np.linalg.norm(H, axis=1, keepdims=True)
    rel = Hn @ (t / np.linalg.norm(t))
    for i, f in enumerate(order):
        red = max((Hn[f] @ Hn[g] for g in order[:i]), default=0.0)
        assert abs(gains[i] - (lam * rel[f] - (1 - lam) * red)) < 1e-12


def test_cosine_against_library():
    sk = pytest.importorskip("sklearn.metrics.pairwise")
    H = _rand((30, 12), 5)
    Hn = scout.cosine_unit(H)
    np.testing.assert_allclose(Hn @ Hn.T, sk.cosine_similarity(H), rtol=0, atol=1e-13)


def test_scale_invariance_and_permutation_equivariance():
    H, t = _rand((25, 10), 6), _rand(10, 7)
    base = scout.mmr_select(H, t, 0.7, 10)[0]
    scaled = H * np.linspace(0.1, 9.0, 25)[:, None]
    assert scout.mmr_select(scaled, 3.0 * t, 0.7, 10)[0].tolist() == base.tolist()
    perm = np.random.default_rng(8).permutation(25)
    got = scout.mmr_select(H[perm], t, 0.7, 10)[0]
    assert perm[got].tolist() == base.tolist()


def test_zero_frame_has_zero_similarity():
    H = np.array([[0.0, 0.0], [1.0, 0.0], [0.0, -1.0]])
    t = np.array([0.0, 1.0])
    # relevances 0, 0, -1: frame 0 (lower index) first; then frame 1 (red 0,
    # rel 0) over frame 2 (red 0, rel -1)
    order, gains = scout.mmr_select(H, t, 0.7, 3)
    assert order.tolist() == [0, 1, 2] and gains[0] == 0.0


def test_scout_output_layout():
    H, t = _rand((16, 6), 9), _rand(6, 10)
    order, keys, gains = scout.scout(H, t, 0.7, Fraction(3, 4))
    assert len(order) == 12 and keys.tolist() == sorted(order.tolist())
    assert len(set(order.tolist())) == 12
