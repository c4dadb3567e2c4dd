#!/usr/bin/env python
"""Throughput of the PruneKV visual-KV compression pass on GB300.

One step = one prunekv_compress call (plan, score, select, fuse, compact) over
one request of the selected workload (default: 7B shape, 28 layers, 28/4
heads, d=128, 64 frames x 196 = 12,544 visual tokens, 64 window rows, 19%
retention, bf16).  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 3] [--impl ours|reference]

--impl reference times the fp64 CPU oracle (the slow, obviously correct
program the CUDA path is checked against) on bounded samples of the same
workload, on the host cores.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "PruneKV visual-KV tokens×layers compressed/s at 1 GB300; % of roofline"
UNIT = "tokens*layers/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="time direct launches instead of a CUDA graph")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sustain-seconds", type=float, default=1.5,
                    help="repeat the K-step window for this long under the clock sampler (0: only the headline window)")
    ap.add_argument("--schedule", choices=list(SCHEDULES), default="parabola",
                    help="layer-budget schedule (the paper's ablation axes); parabola is the method")
    ap.add_argument("--stage", choices=["prunekv", "scout", "decode", "quant"], default="prunekv",
                    help="prunekv: the compression pass (the headline); scout: MMR keyframe selection")
    ap.add_argument("--requests", type=int, default=16, help="--stage decode: concurrent requests")
    ap.add_argument("--decode-cache", choices=["both", "compressed", "full", "kv4"], default="both",
                    help="--stage decode: which caches to time")
    ap.add_argument("--rank", choices=["shared", "per_layer"], default="shared",
                    help="ranking: one order per KV head from the layer mean (method default) or per layer")
    ap.add_argument("--drop", choices=["survivors", "all"], default="survivors",
                    help="drop set: survivors of the top-q step (method) or every non-kept token")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=p["hbm_gbs"], tc=p["bf16_tflops"], tc_sus=p.get("bf16_tflops_sustained"),
                    source="measured")
    return dict(hbm=6800.0, tc=1900.0, tc_sus=1700.0, source="fallback")


# ---------------------------------------------------------------------------
# Algorithmic work of one pass (what the method must do, each logit once).

SCHEDULES = {"parabola": 0, "fixed": 1, "arithmetic": 2, "geometric": 3}
DROPS = {"survivors": 0, "all": 1}


def plans_for(wl, vc, schedule="parabola", drop="survivors"):
    out = []
    for r in wl.requests:
        B, Nq, h = vc.viscache_plan_budgets_ex(wl.L, r.n, r.rr_num, r.rr_den, 0, 3, 4,
                                               SCHEDULES[schedule], DROPS[drop])
        out.append((B, Nq, h))
    return out


def algorithmic(wl, plans):
    eb = 2 if wl.dtype == "bf16" else 4
    tot = dict(bytes=0, flops_score=0, flops_fuse=0, k_bytes=0, gather_bytes=0, gather_v_bytes=0,
               gather_kv_bytes=0, fuse_bytes=0, surv_v_bytes=0, tokens_layers=0)
    for r, (B, Nq, h) in zip(wl.requests, plans):
        T = sum(B)
        row = wl.d * eb
        k_all = wl.L * wl.Hkv * r.n * row
        q = wl.L * wl.Hq * r.W * row
        kept_k = wl.Hkv * T * row
        surv_v = sum(1 for b in B if b > 0) * wl.Hkv * Nq * row
        out = 2 * wl.Hkv * T * row
        tot["bytes"] += k_all + q + kept_k + surv_v + out
        tot["k_bytes"] += k_all + q
        tot["gather_bytes"] += 2 * kept_k              # kept keys read and written
        tot["gather_v_bytes"] += 2 * surv_v            # survivor values read, slab written
        tot["gather_kv_bytes"] += 2 * (kept_k + surv_v)
        tot["fuse_bytes"] += surv_v + wl.Hkv * T * row
        tot["surv_v_bytes"] += surv_v
        tot["flops_score"] += 2 * wl.Hq * r.W * r.n * wl.d * wl.L
        tot["flops_fuse"] += 4 * wl.Hkv * wl.d * sum(b * (Nq - b) for b in B if b > 0)
        tot["tokens_layers"] += r.n * wl.L
    return tot


# per kernel: (kind, work key) -> achieved = work / time
KERNEL_WORK = {
    "score_lse_simt": ("tensor", "flops_score"),
    "score_colsum_simt": ("tensor", "flops_score"),
    "score_lse_tc": ("tensor", "flops_score"),
    "score_colsum_tc": ("tensor", "flops_score"),
    "fuse_v_simt": ("tensor", "flops_fuse"),
    "fuse_v_tc": ("tensor", "flops_fuse"),
    "gather_kv": ("hbm", "gather_kv_bytes"),
    "gather_v": ("hbm", "gather_v_bytes"),
    "gather_k": ("hbm", "gather_bytes"),
}


def traffic_for(kernel, workload):
    """dram bytes per launch from the committed ncu summary: only for the workload
    it was captured on, and only while the kernel's source is unchanged."""
    path = os.path.join(ROOT, "profiles", "traffic.md")
    if workload is None or not os.path.exists(path):
        return None
    for line in open(path):
        cells = [c.strip() for c in line.strip().strip("|").split("|")]
        if len(cells) != 5 or cells[0] != kernel or cells[1] != workload:
            continue
        src = os.path.join(ROOT, cells[2])
        if not os.path.exists(src):
            return None
        with open(src, "rb") as f:
            digest = hashlib.sha256(f.read()).hexdigest()[:16]
        return int(cells[4]) if digest == cells[3] else None
    return None


# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "200", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------
def oracle_sample(wl, layers, seed_layer0=0, schedule="parabola", drop="survivors", rank="shared"):
    """Run the fp64 oracle on the first `layers` layers of request 0; returns (seconds, tokens*layers)."""
    import numpy as np
    import torch
    from fractions import Fraction

    from oracle import plan as oplan
    from oracle import prunekv as ok
    from paper_2608_24063_gb300 import synth

    sub = synth.scaled(wl, "sample", L=layers, requests=[wl.requests[0]])
    q = synth.make_q(sub, 0)
    k, v = synth.make_kv(sub, 0, q)
    Qn, Kn, Vn = (t.to(torch.float64).numpy() for t in (q, k, v))
    r = sub.requests[0]
    B, Nq, h = oplan.plan_budgets(layers, r.n, Fraction(r.rr_num, r.rr_den), schedule=schedule, drop=drop)
    t0 = time.perf_counter()
    ok.prunekv(Qn, Kn, Vn, B, Nq, mu=0.7, tau=1.0, rank_mode=rank)
    dt = time.perf_counter() - t0
    return dt, r.n * layers


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def run_reference(args, wl):
    """--impl reference: the oracle timed on the host cores, one bounded sample per step."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    layers = 1
    for _ in range(args.warmup):
        oracle_sample(wl, layers, schedule=args.schedule, drop=args.drop, rank=args.rank)
    times = []
    tl = 0
    for _ in range(args.steps):
        dt, tl = oracle_sample(wl, layers, schedule=args.schedule, drop=args.drop, rank=args.rank)
        times.append(dt)
    sec = sum(times) / len(times)
    val = tl / sec
    cfg = workload_config(wl, args)
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded, structure of the paper's long-video workloads)",
            "config": cfg,
            "cpu_baseline": {"value": val, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                             "sample": "Algorithm 1 on layer 1 of %d (all %d tokens, %d window rows) per step" %
                                       (wl.L, wl.requests[0].n, wl.requests[0].W)},
            "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def rank_requests(wl, world, rank):
    """Weak scaling: the job is `world` copies of the workload's requests (each copy
    its own seeded values), split over the ranks by the work-balanced request
    partition; no data-path collective.  Returns (job workload, this rank's request
    indices, this rank's workload view).  At world = 1 the job is the workload."""
    from paper_2608_24063_gb300 import shard, synth
    job = synth.replicated(wl, world)
    costs = [shard.request_cost(r.n, r.W, wl.L, wl.Hq) for r in job.requests]
    mine = shard.partition_requests(costs, world)[rank]
    view = synth.scaled(job, job.name, requests=[job.requests[i] for i in mine])
    return job, mine, view


def max_over_ranks(x, world, dist, device):
    """Max of a host float over all ranks (the timed region is the slowest rank's)."""
    if world <= 1:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(units_all_ranks, ms_per_step):
    """Whole-job throughput: the units of all ranks / the slowest rank's step time."""
    return units_all_ranks / (ms_per_step * 1e-3)


def workload_config(wl, args=None):
    r = wl.requests[0]
    in_bytes = sum(wl.L * (wl.Hq * q.W + 2 * wl.Hkv * q.n) * wl.d * (2 if wl.dtype == "bf16" else 4)
                   for q in wl.requests)
    return {"workload": wl.name, "requests": len(wl.requests), "L": wl.L, "Hq": wl.Hq,
            "Hkv": wl.Hkv, "d": wl.d, "n_vis": [q.n for q in wl.requests],
            "W": [q.W for q in wl.requests],
            "retention": ["%d/%d" % (q.rr_num, q.rr_den) for q in wl.requests],
            "h": "3L/4", "m": 0.75, "mu": 0.7, "tau": 1.0, "rank": getattr(args, "rank", "shared"),
            "schedule": getattr(args, "schedule", "parabola"), "drop": getattr(args, "drop", "survivors"),
            "l2": "inputs larger than L2 (%.2f GB of Qw+K+V > 129 MB)" % (in_bytes / 1e9)}


def run_scout(args):
    """--stage scout: Eq. (mmr) keyframe selection on a batch of synthetic videos."""
    import torch
    from fractions import Fraction

    from oracle import scout as osc
    from paper_2608_24063_gb300 import synth
    from paper_2608_24063_gb300 import viscache as vc

    n_vid, F, D, lam, p = 64, 64, 512, 0.7, (3, 4)
    vids = [synth.scout_embeddings(1000 + i, F, D) for i in range(n_vid)]
    cfg = {"workload": "scout: %d videos x %d frames, D=%d (CLIP ViT-B/32 width), lambda=%.1f, p=%d/%d"
           % (n_vid, F, D, lam, p[0], p[1]), "videos": n_vid, "frames": F, "D": D}
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return
        for _ in range(args.warmup):
            osc.scout(vids[0][0].double().numpy(), vids[0][1].double().numpy(), lam, Fraction(*p))
        t0 = time.perf_counter()
        for i in range(args.steps):
            h, t = vids[i % n_vid]
            osc.scout(h.double().numpy(), t.double().numpy(), lam, Fraction(*p))
        dt = (time.perf_counter() - t0) / args.steps
        val = 1.0 / dt
        print(json.dumps({"metric": "scout keyframe selection videos/s", "value": val, "unit": "videos/s",
                          "impl": "reference", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                          "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
                          "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": cfg,
                          "cpu_baseline": {"value": val, "unit": "videos/s", "cores": cpu_cores(),
                                           "kind": "oracle", "sample": "one video per step"},
                          "e2e": {"value": val, "unit": "videos/s", "h2d_bytes_per_step": 0,
                                  "d2h_bytes_per_step": 0}}))
        return
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    H = torch.cat([h for h, _ in vids]).to(dev)
    T = torch.stack([t for _, t in vids]).to(dev)
    sizes = [F] * n_vid
    o0, k0, g0, _ = vc.viscache_scout_mmr(H, T, sizes, lam, p)
    nf = (__import__("ctypes").c_int32 * n_vid)(*sizes)
    wsb = torch.empty(max(vc.lib().viscache_scout_workspace_size(n_vid, nf, D), 256), dtype=torch.uint8,
                      device=dev)

    def step():
        return vc.viscache_scout_mmr(H, T, sizes, lam, p, out=(o0, k0, g0), ws=wsb)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        step()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    vc.viscache_profile_enable(True)
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize()
    kern = {k: v[0] / v[1] for k, v in vc.viscache_profile_read().items()}
    vc.viscache_profile_enable(False)
    # end to end: embeddings from pinned host memory, keyframes back to the host
    hH, hT = H.cpu().pin_memory(), T.cpu().pin_memory()
    a.record()
    for _ in range(args.steps):
        order, keys, gains, ks = vc.viscache_scout_mmr(hH.to(dev, non_blocking=True),
                                                       hT.to(dev, non_blocking=True), sizes, lam, p,
                                                       out=(o0, k0, g0), ws=wsb)
        keys.cpu()
    b.record()
    torch.cuda.synchronize()
    ems = a.elapsed_time(b) / args.steps
    # the oracle on the host cores, a bounded sample
    t0 = time.perf_counter()
    nv = 0
    while time.perf_counter() - t0 < min(args.cpu_seconds, 5.0) or nv == 0:
        h, t = vids[nv % n_vid]
        osc.scout(h.double().numpy(), t.double().numpy(), lam, Fraction(*p))
        nv += 1
    cpu = nv / (time.perf_counter() - t0)
    k = ks[0]
    print(json.dumps({
        "metric": "scout keyframe selection videos/s", "value": n_vid / (ms * 1e-3), "unit": "videos/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded scene-structured embeddings)", "config": cfg,
        "kernels_ms_per_step": kern, "gpu_launches": len(kern) * args.steps,
        "picks_per_video": k, "kernel_us_per_batch": sum(kern.values()) * 1e3,
        "cpu_baseline": {"value": cpu, "unit": "videos/s", "cores": cpu_cores(), "kind": "oracle",
                         "sample": "%d videos, one at a time (fp64 numpy)" % nv},
        "e2e": {"value": n_vid / (ems * 1e-3), "unit": "videos/s",
                "h2d_bytes_per_step": int(hH.numel() * 4 + hT.numel() * 4),
                "d2h_bytes_per_step": int(keys.numel() * 4)}}))


def run_decode(args):
    """--stage decode: one decode step's attention in every layer over the
    compressed cache (the pass's output layout) and, for comparison, over the
    full cache (every B_l = n, the same kernels)."""
    import torch

    from oracle import decode as odec
    from paper_2608_24063_gb300 import viscache as vc

    n_req, L, Hq, Hkv, d, n, T, rr = args.requests, 28, 28, 4, 128, 12544, 512, (19, 100)
    cfg = {"workload": "decode step, %d requests on the 7B shape (L=%d, Hq=%d, Hkv=%d, d=%d, bf16), "
                       "n=%d visual + T=%d text tokens, RR=%d%%" % (n_req, L, Hq, Hkv, d, n, T, rr[0]),
           "requests": n_req, "L": L, "Hq": Hq, "Hkv": Hkv, "d": d, "n_vis": n, "text": T,
           "retention": "%d/%d" % rr, "schedule": "parabola"}
    metric = "decode-step attention tokens/s over the compressed visual cache (all layers)"
    batch_c = vc.Batch([n] * n_req, [64] * n_req, [rr] * n_req)
    prm_c = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    B, _, _ = vc.viscache_plan_budgets(L, n, *rr)
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return
        import numpy as np
        rng = np.random.default_rng(5)
        Kc = [rng.standard_normal((Hkv, b, d)) for b in B]
        Vc = [rng.standard_normal((Hkv, b, d)) for b in B]
        Kt, Vt = rng.standard_normal((Hkv, T, d)), rng.standard_normal((Hkv, T, d))
        q = rng.standard_normal((Hq, d))

        def one_request():
            for l in range(L):
                odec.decode_attention(q, Kc[l], Vc[l], Kt, Vt)

        for _ in range(args.warmup):
            one_request()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            one_request()
        dt = (time.perf_counter() - t0) / args.steps
        val = 1.0 / dt
        print(json.dumps({"metric": metric, "value": val, "unit": "tokens/s", "impl": "reference",
                          "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
                          "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
                          "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": cfg,
                          "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": cpu_cores(),
                                           "kind": "oracle", "sample": "one request's step (all layers) per step"},
                          "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                                  "d2h_bytes_per_step": 0}}))
        return
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(12544)

    def normal(*shape):
        return torch.empty(shape, dtype=torch.bfloat16, device=dev).normal_(generator=gen)

    batch_f = vc.Batch([n] * n_req, [64] * n_req, [(1, 1)] * n_req)
    prm_f = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16, h=L, m=(1, 1), schedule=vc.VC_SCHED_FIXED)
    rows_c = vc.compressed_rows(batch_c, prm_c)
    texts = [T] * n_req
    names = ("full", "compressed", "kv4") if args.decode_cache == "both" else (args.decode_cache,)
    caches = {}
    if "compressed" in names or "kv4" in names:
        caches["compressed"] = (batch_c, prm_c, normal(rows_c, d), normal(rows_c, d))
    if "kv4" in names:
        # the compressed cache's visual rows in 4-bit form
        kv4 = vc.viscache_kv4_quantize(batch_c, prm_c, caches["compressed"][2], caches["compressed"][3])
        caches["kv4"] = (batch_c, prm_c, kv4, None)
    if "full" in names:
        caches["full"] = (batch_f, prm_f, normal(n_req * L * Hkv * n, d), normal(n_req * L * Hkv * n, d))
    Kt, Vt = normal(L, n_req * Hkv * T, d), normal(L, n_req * Hkv * T, d)
    q = normal(L, n_req, Hq, d)
    out = torch.empty_like(q)
    ws = torch.empty(max(vc.viscache_decode_workspace_size(b, p, texts) for b, p, _, _ in caches.values()),
                     dtype=torch.uint8, device=dev)
    if args.decode_cache == "kv4":
        del caches["compressed"]

    def step(name, qq=q):
        b, p, K, V = caches[name]
        for l in range(L):
            if name == "kv4":
                vc.viscache_decode_attention_kv4(b, p, l, qq[l], K, Kt[l], Vt[l], texts, out=out[l], ws=ws)
            else:
                vc.viscache_decode_attention(b, p, l, qq[l], K, V, Kt[l], Vt[l], texts, out=out[l], ws=ws)

    res = {}
    clk = None
    for name in names:
        for _ in range(max(3, args.warmup)):
            step(name)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            step(name)
            with torch.cuda.graph(g):
                step(name)
        torch.cuda.current_stream().wait_stream(s)
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if name == "compressed":
            clocks = ClockSampler(local)
            clocks.start()
        a.record()
        for _ in range(args.steps):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        if name == "compressed":
            clk = clocks.stop()
        ms = a.elapsed_time(b) / args.steps
        vc.viscache_profile_enable(True)
        for _ in range(args.steps):
            step(name)
        torch.cuda.synchronize()
        prof = vc.viscache_profile_read()
        kern = {k: v[0] / args.steps for k, v in prof.items()}
        launches = {k: v[1] // args.steps for k, v in prof.items()}
        vc.viscache_profile_enable(False)
        del g
        res[name] = (ms, kern, launches)
    if len(names) == 1:
        # one cache alone (a profiling run): its time and kernel split only
        ms, kern, launches = res[names[0]]
        print(json.dumps({"stage": "decode", "cache": names[0], "requests": n_req, "ms_per_step": ms,
                          "kernels_ms_per_step": kern, "launches_per_step": launches, "clocks": clk}))
        return
    ms, kern, launches = res["compressed"]
    ms_full, kern_full, _ = res["full"]
    ms_q4, kern_q4, _ = res["kv4"]
    # algorithmic bytes of a step: every cached K and V row of every layer once
    # plus the query rows (the main kernel, L launches a step); achieved =
    # those bytes over the launches' summed event time
    kv_rows = sum(n_req * Hkv * (b + T) for b in B)
    kv_rows_full = L * n_req * Hkv * (n + T)
    q_bytes = L * n_req * Hq * d * 2
    pk = peaks()
    main_kernel = max(kern, key=kern.get)
    t_part = kern.get(main_kernel, float("nan")) * 1e-3
    achieved = (kv_rows * d * 2 * 2 + q_bytes) / t_part / 1e9
    t_part_f = kern_full.get(main_kernel, float("nan")) * 1e-3
    achieved_f = (kv_rows_full * d * 2 * 2 + q_bytes) / t_part_f / 1e9
    # end to end through the public call: this step's query rows from pinned
    # host memory, the attention outputs back to the host
    hq = q.cpu().pin_memory()
    hout = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
    qd = torch.empty_like(q)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for _ in range(2):
        qd.copy_(hq, non_blocking=True)
        step("compressed", qd)
        hout.copy_(out, non_blocking=True)
    torch.cuda.synchronize()
    a.record()
    for _ in range(args.steps):
        qd.copy_(hq, non_blocking=True)
        step("compressed", qd)
        hout.copy_(out, non_blocking=True)
    b.record()
    torch.cuda.synchronize()
    ems = a.elapsed_time(b) / args.steps
    # the oracle on the host cores: one request's step over every layer
    import numpy as np
    Kc, Vc = caches["compressed"][2], caches["compressed"][3]
    Kn = [Kc[Hkv * sum(B[:l]):Hkv * sum(B[:l + 1])].double().cpu().numpy().reshape(Hkv, B[l], d) for l in range(L)]
    Vn = [Vc[Hkv * sum(B[:l]):Hkv * sum(B[:l + 1])].double().cpu().numpy().reshape(Hkv, B[l], d) for l in range(L)]
    Ktn = [Kt[l, :Hkv * T].double().cpu().numpy().reshape(Hkv, T, d) for l in range(L)]
    Vtn = [Vt[l, :Hkv * T].double().cpu().numpy().reshape(Hkv, T, d) for l in range(L)]
    qn = q[:, 0].double().cpu().numpy()
    t0 = time.perf_counter()
    nr = 0
    while time.perf_counter() - t0 < min(args.cpu_seconds, 10.0) or nr == 0:
        for l in range(L):
            odec.decode_attention(qn[l], Kn[l], Vn[l], Ktn[l], Vtn[l])
        nr += 1
    cpu = nr / (time.perf_counter() - t0)
    print(json.dumps({
        "metric": metric, "value": n_req / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded normal cache)",
        "config": dict(cfg, launch="cuda graph of the %d per-layer calls" % L,
                       l2="a step reads %.2f GB of cache > 129 MB L2" % (kv_rows * d * 4 / 1e9)),
        "full_cache": {"ms_per_step": ms_full, "value": n_req / (ms_full * 1e-3),
                       "speedup_of_compressed": ms_full / ms,
                       "kernels_ms_per_step": kern_full,
                       "main_kernel_gbs": achieved_f},
        "kv4_cache": {"ms_per_step": ms_q4, "value": n_req / (ms_q4 * 1e-3),
                      "speedup_vs_compressed": ms / ms_q4, "kernels_ms_per_step": kern_q4,
                      "cache_bytes_per_step": int(sum(n_req * Hkv * b for b in B) * (d + d // 32 * 8)
                                                  + sum(n_req * Hkv * -(-b // 32) * d * 8 for b in B)
                                                  + L * n_req * Hkv * T * d * 2 * 2)},
        "kernels_ms_per_step": kern,
        "roofline": {"kernel": main_kernel, "bound": "hbm", "achieved": achieved,
                     "peak": pk["hbm"], "unit": "GB/s", "frac": achieved / pk["hbm"],
                     "traffic": traffic_for(main_kernel, "decode, %d requests" % n_req),
                     "peak_source": pk["source"]},
        "cpu_baseline": {"value": cpu, "unit": "tokens/s", "cores": cpu_cores(), "kind": "oracle",
                         "sample": "%d single-request steps over all %d layers (fp64 numpy)" % (nr, L)},
        "e2e": {"value": n_req / (ems * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": int(q.numel() * 2), "d2h_bytes_per_step": int(out.numel() * 2)},
        "gpu_launches": sum(launches.values()) * args.steps, "clocks": clk}))


def run_quant(args):
    """--stage quant: 4-bit quantisation of the compacted cache of 16 requests
    on the 7B shape (the decode workload's cache), and its reconstruction."""
    import numpy as np
    import torch

    from oracle import quant as oq
    from paper_2608_24063_gb300 import viscache as vc

    n_req, L, Hq, Hkv, d, n, rr = args.requests, 28, 28, 4, 128, 12544, (19, 100)
    batch = vc.Batch([n] * n_req, [64] * n_req, [rr] * n_req)
    prm = vc.make_params(L, Hq, Hkv, d, vc.VC_BF16)
    rows, groups = vc.viscache_kv4_sizes(batch, prm)
    cfg = {"workload": "4-bit quantisation of the compacted cache: %d requests on the 7B shape "
                       "(L=%d, Hkv=%d, d=%d, bf16), n=%d, RR=%d%%: %d rows of K and of V"
                       % (n_req, L, Hkv, d, n, rr[0], rows),
           "requests": n_req, "rows": rows, "key_groups": groups, "group": oq.GROUP}
    metric = "compacted KV quantised to 4 bits, input GB/s"
    in_bytes = 2 * rows * d * 2
    out_bytes = 2 * rows * d // 2 + groups * d * 8 + rows * (d // 32) * 8
    rank = int(os.environ.get("RANK", "0"))
    sample_rows = 32768

    def oracle_rate(K, V, seconds):
        t0, done = time.perf_counter(), 0
        while time.perf_counter() - t0 < seconds or done == 0:
            oq.quantize_keys(K)
            oq.quantize_values(V)
            done += K.shape[0]
        return done * d * 2 * 2 / (time.perf_counter() - t0) / 1e9

    if args.impl == "reference":
        if rank != 0:
            return
        rng = np.random.default_rng(3)
        K = rng.standard_normal((sample_rows, d)).astype(np.float32)
        V = rng.standard_normal((sample_rows, d)).astype(np.float32)
        for _ in range(args.warmup):
            oq.quantize_keys(K[:1024])
        t0 = time.perf_counter()
        for _ in range(args.steps):
            oq.quantize_keys(K)
            oq.quantize_values(V)
        dt = (time.perf_counter() - t0) / args.steps
        val = sample_rows * d * 2 * 2 / dt / 1e9
        print(json.dumps({"metric": metric, "value": val, "unit": "GB/s", "impl": "reference", "n_gpus": 1,
                          "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3,
                          "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                          "data": "synthetic", "config": cfg,
                          "cpu_baseline": {"value": val, "unit": "GB/s", "cores": cpu_cores(), "kind": "oracle",
                                           "sample": "%d rows of K and V per step" % sample_rows},
                          "e2e": {"value": val, "unit": "GB/s", "h2d_bytes_per_step": 0,
                                  "d2h_bytes_per_step": 0}}))
        return
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    gen = torch.Generator(device=dev)
    gen.manual_seed(4)
    K = torch.empty((rows, d), dtype=torch.bfloat16, device=dev).normal_(generator=gen)
    V = torch.empty((rows, d), dtype=torch.bfloat16, device=dev).normal_(generator=gen)
    out = vc.viscache_kv4_quantize(batch, prm, K, V)
    hat = vc.viscache_kv4_dequantize(batch, prm, *out)

    def quantize():
        vc.viscache_kv4_quantize(batch, prm, K, V, out=out)

    def dequantize():
        vc.viscache_kv4_dequantize(batch, prm, *out, out=hat)

    res = {}
    clk = None
    for name, fn in (("quantize", quantize), ("dequantize", dequantize)):
        for _ in range(max(3, args.warmup)):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if name == "quantize":
            clocks = ClockSampler(local)
            clocks.start()
        a.record()
        for _ in range(args.steps):
            fn()
        b.record()
        torch.cuda.synchronize()
        if name == "quantize":
            clk = clocks.stop()
        vc.viscache_profile_enable(True)
        for _ in range(args.steps):
            fn()
        torch.cuda.synchronize()
        prof = vc.viscache_profile_read()
        vc.viscache_profile_enable(False)
        res[name] = (a.elapsed_time(b) / args.steps, {k: v[0] / args.steps for k, v in prof.items()},
                     sum(v[1] for v in prof.values()))
    ms, kern, launches = res["quantize"]
    ms_dq, kern_dq, _ = res["dequantize"]
    pk = peaks()
    t_k = kern.get("kv4_quantize", float("nan")) * 1e-3
    achieved = (in_bytes + out_bytes) / t_k / 1e9
    # end to end: the cache from pinned host memory, codes and parameters back
    hK, hV = K.cpu().pin_memory(), V.cpu().pin_memory()
    dK, dV = torch.empty_like(K), torch.empty_like(V)
    hout = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True) for x in out]
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        dK.copy_(hK, non_blocking=True)
        dV.copy_(hV, non_blocking=True)
        vc.viscache_kv4_quantize(batch, prm, dK, dV, out=out)
        for h, x in zip(hout, out):
            h.copy_(x, non_blocking=True)
    b.record()
    torch.cuda.synchronize()
    ems = a.elapsed_time(b) / args.steps
    Ks = K[:sample_rows].float().cpu().numpy()
    Vs = V[:sample_rows].float().cpu().numpy()
    cpu = oracle_rate(Ks, Vs, min(args.cpu_seconds, 5.0))
    print(json.dumps({
        "metric": metric, "value": in_bytes / (ms * 1e-3) / 1e9, "unit": "GB/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded normal cache)",
        "config": dict(cfg, l2="%.2f GB of K and V per step > 129 MB L2" % (in_bytes / 1e9)),
        "compression": in_bytes / out_bytes,
        "dequantize": {"ms_per_step": ms_dq, "kernels_ms_per_step": kern_dq},
        "kernels_ms_per_step": kern,
        "roofline": {"kernel": "kv4_quantize", "bound": "hbm", "achieved": achieved, "peak": pk["hbm"],
                     "unit": "GB/s", "frac": achieved / pk["hbm"], "traffic": None,
                     "peak_source": pk["source"]},
        "cpu_baseline": {"value": cpu, "unit": "GB/s", "cores": cpu_cores(), "kind": "oracle",
                         "sample": "%d rows of K and V, repeated for ~5 s (fp32 numpy)" % sample_rows},
        "e2e": {"value": in_bytes / (ems * 1e-3) / 1e9, "unit": "GB/s", "h2d_bytes_per_step": int(in_bytes),
                "d2h_bytes_per_step": int(sum(x.numel() * x.element_size() for x in out))},
        "gpu_launches": launches, "clocks": clk}))


def main():
    args = parse()
    if args.stage != "prunekv" and int(os.environ.get("RANK", "0")) != 0:
        # the scout, decode and quantisation stages are single-GPU measurements:
        # under torchrun the other ranks leave without work, rank 0 prints
        return
    if args.stage == "quant":
        run_quant(args)
        return
    if args.stage == "scout":
        run_scout(args)
        return
    if args.stage == "decode":
        run_decode(args)
        return
    from paper_2608_24063_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    if args.impl == "reference":
        run_reference(args, wl)
        return

    import torch
    import torch.distributed as dist

    from paper_2608_24063_gb300 import viscache as vc

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    st = torch.cuda.current_stream()

    # inputs: generated on the device, resident in HBM before timing
    job, mine, wl_rank = rank_requests(wl, world, rank)
    job_units = sum(r.n * wl.L for r in job.requests)
    qs, ks, vs = synth.generate(job, dev, mine)
    Q = torch.cat([q.flatten() for q in qs]) if len(qs) > 1 else qs[0]
    K = torch.cat([k.flatten() for k in ks]) if len(ks) > 1 else ks[0]
    V = torch.cat([v.flatten() for v in vs]) if len(vs) > 1 else vs[0]
    del qs, ks, vs
    batch = vc.Batch([r.n for r in wl_rank.requests], [r.W for r in wl_rank.requests],
                     [(r.rr_num, r.rr_den) for r in wl_rank.requests])
    prm = vc.make_params(wl.L, wl.Hq, wl.Hkv, wl.d, vc.VC_BF16 if wl.dtype == "bf16" else vc.VC_F32,
                         schedule=SCHEDULES[args.schedule], drop_mode=DROPS[args.drop],
                         rank_mode=vc.VC_RANK_PER_LAYER if args.rank == "per_layer" else vc.VC_RANK_SHARED)
    rows = vc.compressed_rows(batch, prm)
    K_out = torch.empty((rows, wl.d), dtype=K.dtype, device=dev)
    V_out = torch.empty((rows, wl.d), dtype=V.dtype, device=dev)
    idx = torch.empty(rows, dtype=torch.int32, device=dev)
    ws = torch.empty(vc.prunekv_workspace_size(batch, prm), dtype=torch.uint8, device=dev)

    def step():
        vc.prunekv_compress(batch, prm, Q, K, V, K_out, V_out, idx, ws)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    assert vc.prunekv_get_status(ws) == vc.VC_OK

    # the step as a CUDA graph of the same public call (one launch per step);
    # direct launches if capture is unavailable
    graph = None
    if not args.no_graph:
        try:
            cap = torch.cuda.Stream()
            cap.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(cap):
                step()
            torch.cuda.current_stream().wait_stream(cap)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                step()
            for _ in range(max(3, args.warmup)):
                g.replay()
            torch.cuda.synchronize()
            graph = g
        except Exception:
            graph = None
    run = graph.replay if graph is not None else step

    # timed region 1: the headline (no per-kernel events)
    clocks = ClockSampler(local)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(st)
    for _ in range(args.steps):
        run()
    t1.record(st)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms = max_over_ranks(t0.elapsed_time(t1), world, dist, dev)
    ms_step = ms / args.steps
    # the same K-step window repeated until ~1.5 s of load have run, with the
    # clock sampler still going, so the clock record covers a long load; the
    # headline stays the first window of exactly K steps
    windows = []
    if args.steps > 0:
        n_more = max(0, min(2000, int(math.ceil(args.sustain_seconds * 1e3 / max(ms, 1e-3))) - 1))
        ea = [torch.cuda.Event(enable_timing=True) for _ in range(n_more + 1)]
        for i in range(n_more):
            ea[i].record(st)
            for _ in range(args.steps):
                run()
        ea[n_more].record(st)
        torch.cuda.synchronize()
        windows = [ea[i].elapsed_time(ea[i + 1]) / args.steps for i in range(n_more)]
    clk = clocks.stop()
    if clk is not None:
        clk["window_s"] = round((ms + sum(windows) * args.steps) / 1e3, 3)
    sustained = None
    if windows:
        sustained = {"windows": len(windows), "steps_per_window": args.steps,
                     "ms_per_step_median": statistics.median(windows),
                     "ms_per_step_min": min(windows), "ms_per_step_max": max(windows)}
    assert vc.prunekv_get_status(ws) == vc.VC_OK

    # the same steps as direct calls (no graph, no per-kernel events)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    d0.record(st)
    for _ in range(args.steps):
        step()
    d1.record(st)
    torch.cuda.synchronize()
    ms_direct = max_over_ranks(d0.elapsed_time(d1), world, dist, dev) / max(args.steps, 1)

    # timed region 2: the same steps as direct calls with the library's event
    # pair around every kernel launch (per-kernel durations and launch count)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    vc.viscache_profile_enable(True)
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize()
    kern = vc.viscache_profile_read()
    vc.viscache_profile_enable(False)
    assert vc.prunekv_get_status(ws) == vc.VC_OK

    plans = plans_for(wl_rank, vc, args.schedule, args.drop)
    work = algorithmic(wl_rank, plans)
    value = job_value(job_units, ms_step)
    pk = peaks()

    # dominant kernel; its DRAM traffic was captured for the default options on one GPU
    default_opts = (world == 1 and args.schedule == "parabola" and args.drop == "survivors"
                    and args.rank == "shared")
    traffic_wl = "workload %d" % args.workload if default_opts else None
    dom = max(kern.items(), key=lambda kv: kv[1][0]) if kern else None
    roof = None
    if dom:
        name, (tot_ms, launches) = dom
        kind, key = KERNEL_WORK.get(name, ("hbm", "bytes"))
        per = tot_ms / max(launches, 1) * 1e-3
        if kind == "tensor":
            ach = work[key] / per / 1e12
            roof = {"kernel": name, "bound": "tensor", "achieved": ach, "peak": pk["tc"],
                    "unit": "TFLOP/s", "frac": ach / pk["tc"], "traffic": traffic_for(name, traffic_wl),
                    "peak_source": pk["source"] + " bf16 dense burst"}
        else:
            ach = work[key] / per / 1e9
            roof = {"kernel": name, "bound": "hbm", "achieved": ach, "peak": pk["hbm"],
                    "unit": "GB/s", "frac": ach / pk["hbm"], "traffic": traffic_for(name, traffic_wl),
                    "peak_source": pk["source"] + " copy bandwidth"}
    t_hbm = work["bytes"] / (pk["hbm"] * 1e9)
    t_tc = work["flops_score"] / (pk["tc"] * 1e12)
    t_fuse = work["flops_fuse"] / (pk["tc"] * 1e12)
    pass_roof = {"t_roofline_us": max(t_hbm, t_tc) * 1e6, "frac": max(t_hbm, t_tc) / (ms_step * 1e-3),
                 "t_roofline_incl_fusion_us": max(t_hbm, t_tc + t_fuse) * 1e6,
                 "frac_incl_fusion": max(t_hbm, t_tc + t_fuse) / (ms_step * 1e-3),
                 "bytes": work["bytes"], "flops_score": work["flops_score"],
                 "flops_fuse": work["flops_fuse"]}

    # end to end through the public API with host buffers: every step copies its
    # inputs from pinned host memory, compresses, and copies the compressed cache
    # back; steps are pipelined over two buffer sets and three streams (copy in,
    # compute, copy out), as a server streaming requests through one GPU would
    e2e = None
    if not args.no_e2e:
        hQ = [torch.empty(Q.shape, dtype=Q.dtype, pin_memory=True) for _ in range(2)]
        hK = [torch.empty(K.shape, dtype=K.dtype, pin_memory=True) for _ in range(2)]
        hV = [torch.empty(V.shape, dtype=V.dtype, pin_memory=True) for _ in range(2)]
        for i in range(2):
            hQ[i].copy_(Q); hK[i].copy_(K); hV[i].copy_(V)
        oK = [torch.empty(K_out.shape, dtype=K_out.dtype, pin_memory=True) for _ in range(2)]
        oV = [torch.empty(V_out.shape, dtype=V_out.dtype, pin_memory=True) for _ in range(2)]
        oI = [torch.empty(idx.shape, dtype=idx.dtype, pin_memory=True) for _ in range(2)]
        dQ = [Q, torch.empty_like(Q)]
        dK = [K, torch.empty_like(K)]
        dV = [V, torch.empty_like(V)]
        dKo = [K_out, torch.empty_like(K_out)]
        dVo = [V_out, torch.empty_like(V_out)]
        dI = [idx, torch.empty_like(idx)]
        # V can stay in pinned host memory when the device reads it directly:
        # only the survivors' rows then cross to the GPU (read by the gather)
        v_accessible = all(vc.viscache_device_accessible(t) for t in hV)
        s_in, s_cmp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
        ev = lambda: torch.cuda.Event()
        in_done, cmp_done, out_done = [ev(), ev()], [ev(), ev()], [ev(), ev()]

        def measure_e2e(v_host):
            def e2e_step(i):
                bsel = i % 2
                if i >= 2:
                    s_in.wait_event(cmp_done[bsel])        # step i-2 has finished reading these inputs
                with torch.cuda.stream(s_in):
                    dQ[bsel].copy_(hQ[bsel], non_blocking=True)
                    dK[bsel].copy_(hK[bsel], non_blocking=True)
                    if not v_host:
                        dV[bsel].copy_(hV[bsel], non_blocking=True)
                    in_done[bsel].record(s_in)
                s_cmp.wait_event(in_done[bsel])
                if i >= 2:
                    s_cmp.wait_event(out_done[bsel])       # step i-2's outputs are back on the host
                vc.prunekv_compress(batch, prm, dQ[bsel], dK[bsel], hV[bsel] if v_host else dV[bsel],
                                    dKo[bsel], dVo[bsel], dI[bsel], ws, stream=s_cmp)
                cmp_done[bsel].record(s_cmp)
                s_out.wait_event(cmp_done[bsel])
                with torch.cuda.stream(s_out):
                    oK[bsel].copy_(dKo[bsel], non_blocking=True)
                    oV[bsel].copy_(dVo[bsel], non_blocking=True)
                    oI[bsel].copy_(dI[bsel], non_blocking=True)
                    out_done[bsel].record(s_out)

            for i in range(4):
                e2e_step(i)
            torch.cuda.synchronize()
            e_steps = max(4, min(args.steps, 12))
            if world > 1:
                dist.barrier()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s_in)
            for i in range(e_steps):
                e2e_step(i)
            s_out.wait_stream(s_in)
            s_out.wait_stream(s_cmp)
            b.record(s_out)
            torch.cuda.synchronize()
            assert vc.prunekv_get_status(ws) == vc.VC_OK
            assert torch.equal(oI[(e_steps - 1) % 2], dI[(e_steps - 1) % 2].cpu())
            ems = max_over_ranks(a.elapsed_time(b) / e_steps, world, dist, dev)
            v_bytes = work["surv_v_bytes"] if v_host else V.numel() * V.element_size()
            return {"value": job_value(job_units, ems), "unit": UNIT,
                    "ms_per_step": ems, "pipelined": "copy-in / compress / copy-out on three streams",
                    "v_source": "pinned host memory read by the gather kernel (survivor rows only)"
                                if v_host else "copied to the device every step",
                    "h2d_bytes_per_step": int(Q.numel() * Q.element_size() + K.numel() * K.element_size()
                                              + v_bytes),
                    "d2h_bytes_per_step": int(K_out.numel() * K_out.element_size()
                                              + V_out.numel() * V_out.element_size()
                                              + idx.numel() * idx.element_size())}

        e2e = measure_e2e(v_accessible)
        if v_accessible:
            # beside it, every input copied to the device every step
            e2e["full_copy"] = measure_e2e(False)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        dt1, tl1 = oracle_sample(wl, 1, schedule=args.schedule, drop=args.drop, rank=args.rank)
        layers = max(1, min(wl.L, int(args.cpu_seconds / max(dt1, 1e-3))))
        dt, tl = oracle_sample(wl, layers, schedule=args.schedule, drop=args.drop, rank=args.rank) if layers > 1 else (dt1, tl1)
        cpu = {"value": tl / dt, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": "Algorithm 1 (fp64 numpy) on the first %d of %d layers of the workload's "
                         "request (all %d tokens, %d window rows): %.1f s" %
                         (layers, wl.L, wl.requests[0].n, wl.requests[0].W, dt)}

    launches = sum(c for _, c in kern.values())
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16"
                if wl.dtype == "bf16" else "f32",
                "data": "synthetic (seeded, structure of the paper's long-video workloads)",
                "config": dict(workload_config(wl, args), launch="cuda graph of the prunekv_compress call"
                               if graph is not None else "direct prunekv_compress calls"),
                "ms_per_step_direct": ms_direct, "sustained": sustained,
                "roofline": roof, "pass_roofline": pass_roof,
                "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches,
                "kernels_ms_per_step": {k: v[0] / args.steps for k, v in kern.items()},
                "clocks": clk}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
