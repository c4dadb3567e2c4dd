"""Seeded synthetic inputs shaped like the paper's long-video workloads.

This module holds none of the PruneKV arithmetic.  It only draws the three
tensors the compression pass consumes -- the observation-window queries
``Qw [L][Hq][W][d]`` and the visual key/value cache ``K, V [L][Hkv][n][d]`` --
with the structure the workloads call for (planted relevant tokens, an
attention-sink token, per-channel key outliers, frame-to-frame redundancy).
Both the fp64 oracle and the CUDA path read their inputs from here, so this is
the only code the two share.

Random numbers come from a counter-based generator: SplitMix64 (Steele, Lea
and Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014;
64-bit golden-ratio increment followed by the published two-multiply
finaliser).  Every element's draw depends only on (stream key, element index),
so any slice can be regenerated on its own, and the draws are written with
torch int64/float64 element-wise operations only: each operation is exact or
a single IEEE-rounded multiply/add, so the same bits come out on the CPU and
on a CUDA device.  Approximately normal variates are Irwin-Hall sums of four
16-bit uniforms, rescaled to mean 0 and variance 1 (tails end at +-sqrt(12)).
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import torch

_M64 = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15
_C1 = 0xBF58476D1CE4E5B9
_C2 = 0x94D049BB133111EB
# Irwin-Hall(4) of 16-bit uniforms: mean 4 * 65535 / 2, std 65536 / sqrt(3).
_IH_MEAN = 2 * 65535
_IH_SCALE = math.sqrt(3.0) / 65536.0

# Stream tags: one independent stream per tensor kind.
TAG_Q, TAG_K, TAG_V, TAG_CHOICE = 1, 2, 3, 4
TAG_SCOUT = 5


def _signed(u: int) -> int:
    u &= _M64
    return u - (1 << 64) if u >= (1 << 63) else u


def mix64(z: int) -> int:
    """SplitMix64 finaliser on a Python int (mod 2**64)."""
    z &= _M64
    z = ((z ^ (z >> 30)) * _C1) & _M64
    z = ((z ^ (z >> 27)) * _C2) & _M64
    return z ^ (z >> 31)


def stream_key(*parts: int) -> int:
    """Hash a tuple of non-negative ints into a 64-bit stream key."""
    k = 0x243F6A8885A308D3
    for p in parts:
        k = mix64((k + _GAMMA * (int(p) + 1)) & _M64)
    return k


def _srl(x: torch.Tensor, k: int) -> torch.Tensor:
    # logical right shift of int64 lanes
    return (x >> k) & ((1 << (64 - k)) - 1)


def _mix64_t(z: torch.Tensor) -> torch.Tensor:
    z = z ^ _srl(z, 30)
    z = z * _signed(_C1)
    z = z ^ _srl(z, 27)
    z = z * _signed(_C2)
    return z ^ _srl(z, 31)


def raw64(key: int, start: int, count: int, device) -> torch.Tensor:
    """SplitMix64 outputs ``start .. start+count-1`` of stream ``key`` (int64 bits)."""
    idx = torch.arange(start + 1, start + count + 1, dtype=torch.int64, device=device)
    z = idx * _signed(_GAMMA) + _signed(key)
    return _mix64_t(z)


def normal(key: int, start: int, count: int, device) -> torch.Tensor:
    """Approximately N(0,1) float64 draws ``start .. start+count-1`` of stream ``key``."""
    z = raw64(key, start, count, device)
    s = (z & 0xFFFF) + ((z >> 16) & 0xFFFF) + ((z >> 32) & 0xFFFF) + _srl(z, 48)
    return (s - _IH_MEAN).to(torch.float64) * _IH_SCALE


class _Choices:
    """Deterministic host-side integer choices (frame offsets, token picks)."""

    def __init__(self, key: int):
        self.key, self.i = key, 0

    def next(self) -> int:
        self.i += 1
        return mix64((self.key + _GAMMA * self.i) & _M64)

    def randint(self, lo: int, hi: int) -> int:
        """Uniform integer in [lo, hi] (inclusive)."""
        return lo + self.next() % (hi - lo + 1)

    def sample(self, population: int, k: int) -> List[int]:
        """k distinct ints from range(population), partial Fisher-Yates, sorted."""
        pool = list(range(population))
        for j in range(k):
            t = j + self.next() % (population - j)
            pool[j], pool[t] = pool[t], pool[j]
        return sorted(pool[:k])


@dataclasses.dataclass(frozen=True)
class Request:
    """One request's visual segment and its retention target."""
    n: int                      # visual tokens
    W: int                      # observation-window query rows
    rr_num: int                 # overall retention ratio RR = rr_num / rr_den
    rr_den: int
    frame_len: int              # tokens per frame (last frame may be partial)


@dataclasses.dataclass(frozen=True)
class Workload:
    """A synthetic workload: model shape, input distribution and requests."""
    name: str
    L: int
    Hq: int
    Hkv: int
    d: int
    dtype: str                  # "bf16" or "f32"
    requests: Tuple[Request, ...]
    seed: int
    planted_frac: float = 0.0   # fraction of tokens planted as relevant (no frame structure)
    relevant_frames: int = 0    # contiguous frames whose keys are boosted
    boost_sigma: float = 3.0    # boost of planted / relevant tokens, in logit sigmas
    sink_sigma: float = 0.0     # boost of token 0 (attention sink); 0 disables
    outlier_frac: float = 0.0   # fraction of key channels scaled (per layer, KV head)
    outlier_scale: float = 10.0
    ar_rho: float = 0.0         # AR(1) coefficient between adjacent frames (K and V)

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def n_outlier(self) -> int:
        return int(math.ceil(self.outlier_frac * self.d)) if self.outlier_frac > 0 else 0

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def logit_sigma(self) -> float:
        """Std of a scaled logit q.k/sqrt(d) for unit-variance q, k under the channel scales."""
        no = self.n_outlier
        return math.sqrt((self.d - no + no * self.outlier_scale ** 2) / self.d)


def _round(x64: torch.Tensor, dtype) -> torch.Tensor:
    """float64 -> float32 (RNE) -> dtype (RNE)."""
    x = x64.to(torch.float32)
    return x if dtype == torch.float32 else x.to(dtype)


def make_q(wl: Workload, r: int, device="cpu") -> torch.Tensor:
    """Observation-window queries of request r: [L][Hq][W][d], i.i.d. ~N(0,1)."""
    req = wl.requests[r]
    per_layer = wl.Hq * req.W * wl.d
    out = torch.empty((wl.L, wl.Hq, req.W, wl.d), dtype=wl.torch_dtype, device=device)
    for l in range(wl.L):
        x = normal(stream_key(wl.seed, TAG_Q, r, l), 0, per_layer, device)
        out[l] = _round(x, wl.torch_dtype).view(wl.Hq, req.W, wl.d)
    return out


def _choices(wl: Workload, r: int, *parts) -> _Choices:
    return _Choices(stream_key(wl.seed, TAG_CHOICE, r, *parts))


def planted_tokens(wl: Workload, r: int) -> List[int]:
    """Token positions whose keys are boosted toward the window queries."""
    req = wl.requests[r]
    if wl.planted_frac > 0:
        k = int(round(wl.planted_frac * req.n))
        return _choices(wl, r, 0).sample(req.n, k)
    if wl.relevant_frames > 0:
        n_frames = -(-req.n // req.frame_len)
        nf = min(wl.relevant_frames, n_frames)
        f0 = _choices(wl, r, 1).randint(0, n_frames - nf)
        return list(range(f0 * req.frame_len, min(req.n, (f0 + nf) * req.frame_len)))
    return []


def outlier_channels(wl: Workload, r: int, l: int, g: int) -> List[int]:
    if wl.n_outlier == 0:
        return []
    return _choices(wl, r, 2, l, g).sample(wl.d, wl.n_outlier)


def plant_vectors(wl: Workload, q: torch.Tensor, sigma: float) -> torch.Tensor:
    """Per (layer, KV head) float64 vector p with mean_i(q_i . p)/sqrt(d) = sigma * logit_sigma.

    p points along the mean of the group's window queries (q as rounded, on CPU).
    """
    qc = q.detach().to("cpu", torch.float64)
    L, Hq, W, d = qc.shape
    G = wl.G
    out = torch.zeros((L, wl.Hkv, d), dtype=torch.float64)
    for l in range(L):
        for g in range(wl.Hkv):
            mu = qc[l, g * G:(g + 1) * G].reshape(-1, d).mean(dim=0)
            nn = float((mu * mu).sum())
            out[l, g] = mu * (sigma * wl.logit_sigma() * math.sqrt(d) / nn)
    return out


def make_kv(wl: Workload, r: int, q: torch.Tensor, device="cpu",
            layers: Optional[Sequence[int]] = None):
    """Visual key/value cache of request r: two [L][Hkv][n][d] tensors.

    Structure (each step optional per workload): i.i.d. ~N(0,1) draws; AR(1)
    across frames at equal within-frame position; key outlier channels scaled;
    planted/relevant tokens and the sink token shifted along the group's mean
    window query.  ``q`` is the request's rounded Qw (any device).
    ``layers`` restricts generation to a subset (others left uninitialised).
    """
    req = wl.requests[r]
    n, d, H = req.n, wl.d, wl.Hkv
    dt = wl.torch_dtype
    K = torch.empty((wl.L, H, n, d), dtype=dt, device=device)
    V = torch.empty((wl.L, H, n, d), dtype=dt, device=device)
    planted = planted_tokens(wl, r)
    p_boost = plant_vectors(wl, q, wl.boost_sigma).to(device) if planted else None
    p_sink = plant_vectors(wl, q, wl.sink_sigma).to(device) if wl.sink_sigma > 0 else None
    planted_t = torch.tensor(planted, dtype=torch.int64, device=device) if planted else None
    c_eps = math.sqrt(1.0 - wl.ar_rho * wl.ar_rho)
    P = req.frame_len
    for l in (range(wl.L) if layers is None else layers):
        for tag, dst in ((TAG_K, K), (TAG_V, V)):
            x = normal(stream_key(wl.seed, tag, r, l), 0, H * n * d, device).view(H, n, d)
            if wl.ar_rho != 0.0:
                eps = x
                x = torch.empty_like(eps)
                x[:, :P] = eps[:, :P]
                for a in range(P, n, P):
                    b = min(a + P, n)
                    x[:, a:b] = (x[:, a - P:b - P] * wl.ar_rho) + (eps[:, a:b] * c_eps)
            if tag == TAG_K:
                for g in range(H):
                    ch = outlier_channels(wl, r, l, g)
                    if ch:
                        cht = torch.tensor(ch, dtype=torch.int64, device=device)
                        x[g][:, cht] = x[g][:, cht] * wl.outlier_scale
                if planted_t is not None:
                    x[:, planted_t, :] = x[:, planted_t, :] + p_boost[l][:, None, :]
                if p_sink is not None:
                    x[:, 0, :] = x[:, 0, :] + p_sink[l]
            dst[l] = _round(x, dt)
    return K, V


# ---------------------------------------------------------------------------
# The five workloads.  Shapes follow the model families the paper evaluates
# (Qwen2-7B-shaped 28 layers x 28/4 heads, 72B-shaped 80 layers x 64/8 heads,
# head_dim 128); the paper's video benchmarks are not available, so these
# seeded tensors stand in for their prefill caches.

SEED = 20261202


def _ragged_requests(count: int = 8) -> Tuple[Request, ...]:
    ch = _Choices(stream_key(SEED, 5, 0xB47C))
    rrs = (19, 23, 28)
    out = []
    for _ in range(count):
        n = ch.randint(2048, 16384)
        W = ch.randint(32, 128)
        rr = rrs[ch.randint(0, 2)]
        out.append(Request(n=n, W=W, rr_num=rr, rr_den=100, frame_len=196))
    return tuple(out)


WORKLOADS = {
    1: Workload("single-layer GQA2 d64 fp32, n=1024, W=32, RR=25%", L=1, Hq=8, Hkv=4, d=64,
                dtype="f32", requests=(Request(1024, 32, 25, 100, 1024),), seed=SEED + 1,
                planted_frac=0.05, boost_sigma=3.0),
    2: Workload("7B-shape bf16, 16x196=3136 tokens, W=64, RR=28%", L=28, Hq=28, Hkv=4, d=128,
                dtype="bf16", requests=(Request(3136, 64, 28, 100, 196),), seed=SEED + 2,
                sink_sigma=8.0, outlier_frac=0.02),
    3: Workload("7B-shape bf16, 64x196=12544 tokens, W=64, RR=19%", L=28, Hq=28, Hkv=4, d=128,
                dtype="bf16", requests=(Request(12544, 64, 19, 100, 196),), seed=SEED + 3,
                sink_sigma=8.0, outlier_frac=0.02, relevant_frames=8, boost_sigma=3.0,
                ar_rho=0.9),
    4: Workload("72B-shape bf16, 128x256=32768 tokens, W=128, RR=22%", L=80, Hq=64, Hkv=8,
                d=128, dtype="bf16", requests=(Request(32768, 128, 22, 100, 256),),
                seed=SEED + 4, sink_sigma=8.0, outlier_frac=0.02, relevant_frames=8,
                boost_sigma=3.0, ar_rho=0.9),
    5: Workload("ragged batch of 8 on the 7B shape, bf16", L=28, Hq=28, Hkv=4, d=128,
                dtype="bf16", requests=_ragged_requests(), seed=SEED + 5, sink_sigma=8.0,
                outlier_frac=0.02, relevant_frames=8, boost_sigma=3.0, ar_rho=0.9),
}


def scaled(wl: Workload, name: str, *, L=None, Hq=None, Hkv=None, d=None, dtype=None,
           requests=None, seed=None) -> Workload:
    """A smaller workload with the same input structure (for fast tests)."""
    return dataclasses.replace(
        wl, name=name, L=wl.L if L is None else L, Hq=wl.Hq if Hq is None else Hq,
        Hkv=wl.Hkv if Hkv is None else Hkv, d=wl.d if d is None else d,
        dtype=wl.dtype if dtype is None else dtype,
        requests=wl.requests if requests is None else tuple(requests),
        seed=wl.seed if seed is None else seed)


def replicated(wl: Workload, copies: int) -> Workload:
    """The workload's request list repeated `copies` times.  Request r draws from
    its own streams (the request index is part of every stream key), so the copies
    have the same shapes and structure and different values; copy 0 is `wl`'s own
    requests, bit for bit."""
    return dataclasses.replace(wl, requests=tuple(wl.requests) * copies)


def generate(wl: Workload, device="cpu", indices: Optional[Sequence[int]] = None):
    """Requests' (Qw, K, V) as lists of per-request tensors on ``device``: all of
    them, or those with the given indices (in that order)."""
    qs, ks, vs = [], [], []
    for r in (range(len(wl.requests)) if indices is None else indices):
        q = make_q(wl, r, "cpu")
        k, v = make_kv(wl, r, q, device)
        qs.append(q.to(device))
        ks.append(k)
        vs.append(v)
    return qs, ks, vs


# ---------------------------------------------------------------------------
# Scout inputs: frame and prompt embeddings (stand-ins for CLIP ViT-B/32
# outputs, width 512).  A video is a run of scenes; a frame is its scene's
# centre plus per-frame noise (consecutive frames of a scene are near
# duplicates), and the prompt sits near the centre of one scene.  No MMR
# arithmetic here.

def scout_embeddings(seed: int, F: int, D: int = 512, noise: float = 0.5,
                     scene_len: int = 8) -> Tuple[torch.Tensor, torch.Tensor]:
    """(H [F][D] fp32, prompt [D] fp32) on the CPU, the same bits every time."""
    n_scenes = (F + scene_len - 1) // scene_len
    centres = normal(stream_key(TAG_SCOUT, seed, 0), 0, n_scenes * D, "cpu").view(n_scenes, D)
    eps = normal(stream_key(TAG_SCOUT, seed, 1), 0, F * D, "cpu").view(F, D)
    scene = torch.arange(F) // scene_len
    H = centres[scene] + noise * eps
    target = _Choices(stream_key(TAG_SCOUT, seed, 2)).randint(0, n_scenes - 1)
    prompt = centres[target] + noise * normal(stream_key(TAG_SCOUT, seed, 3), 0, D, "cpu")
    return H.to(torch.float32), prompt.to(torch.float32)
