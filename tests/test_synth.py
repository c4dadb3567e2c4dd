"""Pins for the seeded input generator (shared by the oracle and the CUDA path)."""
import math

import numpy as np
import torch

from paper_2608_24063_gb300 import synth


def test_splitmix64_known_answer():
    # SplitMix64 (Steele, Lea, Flood 2014) seeded with 0: the state advances by the
    # golden-ratio increment and the first output is 0xE220A8397B1DCDAF.
    assert synth.mix64(synth._GAMMA) == 0xE220A8397B1DCDAF
    z = synth.raw64(0, 0, 3, "cpu")
    ref = [synth.mix64((i + 1) * synth._GAMMA) for i in range(3)]
    assert [v & ((1 << 64) - 1) for v in z.tolist()] == ref


def test_counter_slices_are_consistent():
    a = synth.normal(1234, 0, 1000, "cpu")
    b = synth.normal(1234, 400, 100, "cpu")
    assert torch.equal(a[400:500], b)


def test_normal_moments():
    x = synth.normal(99, 0, 1 << 20, "cpu").numpy()
    assert abs(x.mean()) < 5e-3 and abs(x.var() - 1) < 5e-3
    assert np.abs(x).max() <= math.sqrt(12) + 1e-9


def test_bf16_rounding_is_rne():
    x = torch.tensor([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -8 + 2 ** -20], dtype=torch.float64)
    y = synth._round(x, torch.bfloat16).to(torch.float64)
    assert y.tolist() == [1.0, 1.0 + 2 ** -6, 1.0 + 2 ** -7]


def test_planted_boost_and_structure():
    wl = synth.scaled(synth.WORKLOADS[3], "tiny", L=2, Hq=4, Hkv=2,
                      requests=[synth.Request(600, 16, 19, 100, 60)])
    q = synth.make_q(wl, 0)
    K, V = synth.make_kv(wl, 0, q)
    assert K.shape == (2, 2, 600, wl.d) and K.dtype == torch.bfloat16
    planted = synth.planted_tokens(wl, 0)
    assert len(planted) == 8 * 60 and planted == list(range(planted[0], planted[0] + 480))
    # mean scaled logit of planted keys minus unplanted ones ~ boost * sigma
    qf, kf = q.double(), K.double()
    G = wl.G
    x = torch.einsum("jwd,jnd->jwn", qf[0], kf[0].repeat_interleave(G, 0)) / math.sqrt(wl.d)
    others = [v for v in range(1, 600) if v not in set(planted)]
    lift = x[:, :, planted].mean() - x[:, :, others].mean()
    assert abs(float(lift) - wl.boost_sigma * wl.logit_sigma()) < 0.5
    # sink token
    assert float(x[:, :, 0].mean()) > 6 * wl.logit_sigma()
    # adjacent frames correlated ~ rho for values
    v0 = V[0, 0].double()
    a, b = v0[60:540].flatten(), v0[0:480].flatten()
    rho = float(torch.corrcoef(torch.stack([a, b]))[0, 1])
    assert abs(rho - 0.9) < 0.05


def test_workload_shapes():
    w3 = synth.WORKLOADS[3]
    assert (w3.L, w3.Hq, w3.Hkv, w3.d, w3.requests[0].n, w3.requests[0].W) == (28, 28, 4, 128, 12544, 64)
    w5 = synth.WORKLOADS[5]
    assert len(w5.requests) == 8
    for r in w5.requests:
        assert 2048 <= r.n <= 16384 and 32 <= r.W <= 128 and r.rr_num in (19, 23, 28)
