"""GPU parity of the scout's keyframe selection (Eq. mmr) against the fp64 oracle."""
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import scout as osc
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
TIE = 1e-5        # fp32 cosines (width <= 1024) are within ~1e-6 of fp64


def check_video(H, t, lam, p, order, keys, gains):
    """Replay the GPU's picks in the oracle: each must be a best MMR frame
    given the GPU's earlier picks (exactly, or within TIE of the best);
    returns the number of near-tie picks."""
    H64, t64 = H.double().numpy(), t.double().numpy()
    k = osc.keyframe_count(H64.shape[0], Fraction(*p))
    order = order.cpu().numpy().astype(np.int64)
    assert len(order) == k and len(set(order.tolist())) == k
    assert keys.cpu().numpy().tolist() == sorted(order.tolist())
    Hn = osc.cosine_unit(H64)
    tn = osc.cosine_unit(t64[None])[0]
    rel = Hn @ tn
    red = np.zeros(len(rel))
    chosen = np.zeros(len(rel), bool)
    near = 0
    for i, f in enumerate(order):
        score = lam * rel - (1 - lam) * red
        score[chosen] = -np.inf
        best = int(np.argmax(score))
        if f != best:
            assert score[best] - score[f] <= TIE, "pick %d: %d (%.9f) vs %d (%.9f)" % (i, f, score[f], best, score[best])
            near += 1
        assert abs(float(gains[i]) - score[f]) <= TIE
        chosen[f] = True
        red = Hn @ Hn[f] if i == 0 else np.maximum(red, Hn @ Hn[f])
    return near


@pytest.mark.parametrize("F,D", [(1, 8), (2, 16), (64, 512), (97, 512), (1024, 512), (4096, 64)])
def test_single_video_matches_oracle(F, D):
    H, t = synth.scout_embeddings(F * 7 + D, F, D)
    order, keys, gains, ks = vc.viscache_scout_mmr(H.to(DEV), t[None].to(DEV), [F], 0.7, (3, 4))
    torch.cuda.synchronize()
    near = check_video(H, t, 0.7, (3, 4), order, keys, gains.cpu())
    assert near <= 1
    if F <= 97:     # no near ties expected at these sizes: the oracle's own order
        ref, _ = osc.mmr_select(H.double().numpy(), t.double().numpy(), 0.7, ks[0])
        assert order.cpu().numpy().tolist() == ref.tolist()


def test_batch_equals_videos_one_by_one():
    sizes = [64, 1, 300, 17, 2048, 64]
    vids = [synth.scout_embeddings(100 + i, F, 512) for i, F in enumerate(sizes)]
    H = torch.cat([h for h, _ in vids]).to(DEV)
    T = torch.stack([t for _, t in vids]).to(DEV)
    order, keys, gains, ks = vc.viscache_scout_mmr(H, T, sizes, 0.7, (3, 4))
    torch.cuda.synchronize()
    off = 0
    for (h, t), F, k in zip(vids, sizes, ks):
        o1, k1, g1, _ = vc.viscache_scout_mmr(h.to(DEV), t[None].to(DEV), [F], 0.7, (3, 4))
        torch.cuda.synchronize()
        assert torch.equal(order[off:off + k], o1) and torch.equal(keys[off:off + k], k1)
        assert torch.equal(gains[off:off + k], g1)
        off += k


@pytest.mark.parametrize("lam", [0.0, 0.3, 1.0])
def test_lambda_extremes(lam):
    F = 200
    H, t = synth.scout_embeddings(7, F, 512)
    order, keys, gains, ks = vc.viscache_scout_mmr(H.to(DEV), t[None].to(DEV), [F], lam, (1, 2))
    torch.cuda.synchronize()
    assert check_video(H, t, lam, (1, 2), order, keys, gains.cpu()) <= 2
    if lam == 1.0:      # a sort by relevance
        Hn = osc.cosine_unit(H.double().numpy())
        rel = Hn @ osc.cosine_unit(t.double().numpy()[None])[0]
        top = set(np.lexsort((np.arange(F), -rel))[:ks[0]].tolist())
        assert set(order.cpu().numpy().tolist()) == top


def test_duplicate_and_zero_frames():
    H = torch.zeros(6, 32)
    H[1, 0] = 1.0
    H[2, 0] = 2.0            # same direction as frame 1
    H[3, 1] = 1.0
    H[4, 2] = -1.0           # frame 0 and 5 stay zero
    t = torch.zeros(32)
    t[0] = 1.0
    order, keys, gains, ks = vc.viscache_scout_mmr(H.to(DEV), t[None].to(DEV), [6], 0.7, (1, 1))
    torch.cuda.synchronize()
    ref, _ = osc.mmr_select(H.double().numpy(), t.double().numpy(), 0.7, 6)
    assert order.cpu().numpy().tolist() == ref.tolist()


def test_bad_arguments_rejected():
    H = torch.zeros(4, 8, device=DEV)
    T = torch.zeros(1, 8, device=DEV)
    with pytest.raises(vc.VisCacheError):
        vc.viscache_scout_mmr(H, T, [4], 1.5)
    with pytest.raises(vc.VisCacheError):
        vc.viscache_scout_mmr(H, T, [4], 0.7, (0, 4))
    with pytest.raises(vc.VisCacheError):
        vc.viscache_scout_mmr(torch.zeros(5000, 8, device=DEV), T, [5000])
