#!/usr/bin/env python
"""Benchmark of schedule-driven cached denoising on one GB300 (one JSON line).

Default workload: the scale-up policy (12 layers, n_emb 512, 8 heads, horizon
32 x action dim 14, 4 observation tokens of dim 512, 100 DDPM steps), batch
1024, bf16, with Bernoulli refresh lattices at fractions 0.125 / 0.25 / 0.5 /
1.0.  One step is one evo_denoise call (1024 action chunks, each a full
100-step denoising query).  `value` is chunks/s at the headline fraction
0.125; the line also carries the p50 call latency and chunks/s of every
fraction, the FLOP ratio they imply, the roofline of the loop's launch
sequence, an end-to-end figure through the C ABI with host buffers, the CPU
oracle timed on this machine's host cores, and sub-records (chunks/s, p50,
roofline fraction) for the other workloads: Push-T-shaped batch 1,
manipulation batch 64, scale-up batch 256 and the 64 x 16 population call.

--impl reference times the CPU oracle itself on the same workload.
Multi-GPU (torchrun): every rank runs an independent replica (the path has no
exchange between chunks); value = chunks of all ranks / max rank time.
"""
from __future__ import annotations

import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2607_20293_gb300 import synth  # noqa: E402

WORKLOADS = {
    # name: (config, fractions, headline fraction, schedule kind)
    "pusht": ("pusht", [1.0, 0.5, 0.125], 0.125, "bernoulli"),
    "tiny": ("tiny", [1.0, 0.5], 0.5, "bernoulli_t0"),
    "manip": ("manip", [1.0, 0.5, 0.125], 0.125, "bernoulli"),
    "scale256": ("scale256", [1.0, 0.5, 0.25, 0.125], 0.125, "bernoulli"),
    "scale1024": ("scale1024", [1.0, 0.5, 0.25, 0.125], 0.125, "bernoulli"),
    # redundancy-aware initialisation (Eq. 6 map + Eq. 7 sampling) on Push-T-shaped activations
    "redundancy": ("pusht", [1.0], 1.0, "bernoulli"),
    # published and baseline schedules on the Push-T-shaped policy, batch 1
    "schedules": ("pusht", [1.0], 1.0, "bernoulli"),
    # schedule search with GPU population fitness (the paper's GA configuration)
    "search": ("pusht", [1.0], 1.0, "bernoulli"),
    # 64 candidate lattices (Eq. 7 from a synthetic map, density 5-60 %) x 16 observations, one call
    "population": ("population", [1.0], 1.0, "guided"),
}
DEFAULT_WORKLOAD = "scale1024"
# sub-records of the default line: (workload, timed steps at the headline fraction)
SUBRECORDS = [("pusht", 100), ("manip", 20), ("scale256", 10), ("population", 5)]
OTHER_FRACTION_STEPS = 5         # timed steps at the sweep's other fractions
SUSTAINED_STEP_MS = 50.0         # a timed step this long runs at the sustained (power-capped) clock
REDUNDANCY_SAMPLES = 16          # all-refresh queries whose activations build the map
FP32_LANES_PER_SM = 128          # GB300 SM: 4 x 32 FP32 lanes, one FMA (2 FLOPs) per lane per clock
L2_FLUSH_BYTES = 256 << 20


def describe(cfg: dict, n: int) -> str:
    return (f"L{cfg['n_layer']} E{cfg['n_emb']} h{cfg['n_head']} H{cfg['horizon']} A{cfg['action_dim']} "
            f"obs {cfg['n_obs']}x{cfg['obs_dim']} T{cfg['n_steps']} {cfg['sampler'].upper()} batch {n} {cfg['dtype']}")


def schedule(cfg: dict, frac: float, kind: str) -> np.ndarray:
    U, T = 3 * cfg["n_layer"], cfg["n_steps"]
    return synth.bernoulli_schedule(U, T, frac, seed=3, force_t0=(kind == "bernoulli_t0"))


def algorithmic_bytes(cfg: dict, S: np.ndarray, n: int) -> int:
    """Bytes the cached loop must move per launch: the weights of every refreshed
    unit (SA: W_qkv, W_o; CA: W_q, W_o -- memory keys/values are per query;
    FFN: W_1, W_2), the per-step input/output projections, and one cache
    tile per lattice cell and sample (written on refresh, read on skip)."""
    E, H, A = cfg["n_emb"], cfg["horizon"], cfg["action_dim"]
    es = 2 if cfg["dtype"] == "bf16" else 4
    unit_w = [4 * E * E * es, 2 * E * E * es, 8 * E * E * es]
    U, T = S.shape
    w = sum(int(S[b].sum()) * unit_w[b % 3] for b in range(U))
    fixed = T * ((A * E + H * E + E * A) * 4)
    cache = U * T * n * H * E * es
    return w + fixed + cache


# ---------------------------------------------------------------------------- helpers

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(values, device: str):
    """Element-wise maximum of per-rank timings (seconds) over the process group."""
    import torch
    import torch.distributed as tdist
    t = torch.tensor([float(v) for v in values], device=device, dtype=torch.float64)
    tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


class Clocks:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.proc = None
        self.index = index
        self.path = os.path.join(tempfile.gettempdir(), f"evo_bench_clocks_{os.getpid()}_{index}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
            # the sampler's start-up (driver queries) stays out of the timed region:
            # return once its first sample is written (at most 3 s)
            t0 = time.perf_counter()
            while time.perf_counter() - t0 < 3.0 and self.proc.poll() is None:
                self.f.flush()
                if os.path.getsize(self.path) > 0:
                    break
                time.sleep(0.02)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def measured_peaks() -> dict:
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return {}


def _code_only(src: str) -> str:
    """C/C++/CUDA source without its comments and blank lines."""
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    return "\n".join(line.rstrip() for line in src.splitlines() if line.strip())


def kernel_source_hash() -> str:
    """Hash of the code (comments left out) of every CUDA/C++ source of the
    library: a recorded ncu figure is used only while the kernels it was taken
    on are unchanged."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_20293_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        if f.endswith((".cu", ".cuh", ".h", ".cpp")):
            h.update(f.encode())
            h.update(_code_only(open(os.path.join(csrc, f)).read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str):
    """DRAM bytes per loop launch (cluster path: the loop kernel; batch-wide path:
    the whole launch sequence of one call) from the committed ncu summary, if it
    was taken on the current kernel sources."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        rec = json.load(open(path))
    except Exception:
        return None
    ent = rec.get(workload)
    if not ent or ent.get("kernel_sha") != kernel_source_hash():
        return None
    return ent.get("bytes_per_launch")


def roofline(workload: str, cfg: dict, n: int, rec: dict) -> dict:
    """Roofline of the loop for one sweep point.  Batch >= 64: tensor-bound,
    algorithmic FLOPs = evo_flops x samples over the loop's own event span,
    against the measured bf16 peak -- the sustained (power-capped) figure when a
    timed step lasts SUSTAINED_STEP_MS or more, else the burst figure.  Smaller
    batches: HBM, algorithmic bytes (weights of refreshed units, per-step
    projections, one cache tile per lattice cell) over the loop kernel's time."""
    peaks = measured_peaks()
    kern_ms = rec["kernel_ms_mean"]
    if n >= 64:
        sustained = statistics.median(rec["ms"]) >= SUSTAINED_STEP_MS
        key = "bf16_tflops_sustained" if sustained else "bf16_tflops"
        alg = rec["flops_per_chunk"] * n
        achieved = alg / (kern_ms / 1000.0) / 1e12
        peak = peaks.get(key) or (1700.0 if sustained else 1900.0)
        src = (("measured bf16 sustained (timed step >= %g ms)" % SUSTAINED_STEP_MS) if sustained
               else "measured bf16 burst") if key in peaks else "fallback"
        roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": recorded_traffic(workload), "peak_source": src}
    else:
        alg = rec["alg_bytes"]
        achieved = alg / (kern_ms / 1000.0) / 1e9
        peak = peaks.get("hbm_gbs", 6800.0)
        roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": recorded_traffic(workload),
                "peak_source": "measured HBM copy" if "hbm_gbs" in peaks else "fallback"}
    roof["kernel"] = ("batch-wide launch sequence of one call (tcgen05 GEMMs, attention, row kernels)"
                      if rec["path"] == "wide" else "evo::job_kernel (persistent cluster loop)")
    roof["algorithmic_per_launch"] = alg
    roof["kernel_ms"] = kern_ms
    return roof


# ---------------------------------------------------------------------------- CPU oracle

def _oracle_chunk(args):
    name, frac, kind, seed = args
    from oracle import evo_oracle as O
    cfg = synth.config(name)
    W = synth.make_weights(cfg, 0)
    obs = synth.make_obs(cfg, 1, 1000 + seed)
    noise = synth.make_noise(cfg, 1, 2000 + seed)
    S = schedule(cfg, frac, kind)
    O.denoise(W, cfg, obs, noise, S)
    return 1


def oracle_round(pool, name, frac, kind, n_chunks, base_seed=0) -> float:
    t0 = time.perf_counter()
    pool.map(_oracle_chunk, [(name, frac, kind, base_seed + i) for i in range(n_chunks)])
    return time.perf_counter() - t0


def make_pool():
    import multiprocessing as mp
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[v] = "1"
    workers = max(1, min(16, os.cpu_count() or 1))
    return mp.get_context("spawn").Pool(workers), workers


def cpu_baseline(name, frac, kind, pool, workers) -> dict:
    oracle_round(pool, name, frac, kind, workers)           # warm the workers (imports, weights)
    n = workers * 2
    dt = oracle_round(pool, name, frac, kind, n, base_seed=100)
    batch = synth.config(name)["batch"]
    subset = f"a subset of {n} of the workload's {batch} samples, " if n < batch else ""
    return {"value": n / dt, "unit": "chunks/s", "cores": workers, "kind": "oracle",
            "sample": f"{subset}{n} single-sample chunks of the same workload at refresh fraction {frac}, "
                      f"one float64 numpy oracle process per core"}


# ---------------------------------------------------------------------------- GPU arm

def measure(workload, fracs, head_frac, kind, steps, warmup, world=1, rank=0, local=0, e2e_steps=None):
    """Time evo_denoise on one workload over a sweep of refresh fractions.
    Returns the per-fraction records, the handle's launch info and the byte
    counts of the end-to-end copies."""
    import torch
    from paper_2607_20293_gb300 import binding

    name = WORKLOADS[workload][0]
    cfg = synth.config(name)
    n = cfg["batch"]
    W = synth.make_weights(cfg, 0)
    obs = synth.make_obs(cfg, n, 1 + 17 * rank)
    noise = synth.make_noise(cfg, n, 2 + 17 * rank)
    ev = binding.Evo(cfg, W, n)
    d_obs, d_noise = torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda()
    out = torch.empty((n, cfg["horizon"], cfg["action_dim"]), device="cuda")
    h_obs, h_noise = torch.from_numpy(obs).pin_memory(), torch.from_numpy(noise).pin_memory()
    h_out = torch.empty((n, cfg["horizon"], cfg["action_dim"])).pin_memory()
    flush = torch.empty(L2_FLUSH_BYTES // 4, device="cuda")
    stream = torch.cuda.current_stream()
    k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    k0.record(stream)                # torch creates the CUDA events on first record
    k1.record(stream)
    ev.set_profile_events(k0, k1)
    dist = world > 1
    if dist:
        import torch.distributed as tdist

    def one(S, e2e=False):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        if e2e:
            d_obs.copy_(h_obs, non_blocking=True)
            d_noise.copy_(h_noise, non_blocking=True)
        ev.denoise(d_obs, d_noise, S, out=out)
        if e2e:
            h_out.copy_(out, non_blocking=True)
        b.record(stream)
        b.synchronize()
        return a.elapsed_time(b), k0.elapsed_time(k1)

    sweep = {}
    for frac in sorted(fracs, key=lambda f: f != head_frac):
        head = frac == head_frac
        S = schedule(cfg, frac, kind)
        n_steps = steps if head else min(steps, OTHER_FRACTION_STEPS)
        for _ in range(max(3, warmup)):
            one(S)
        if dist:
            tdist.barrier()
        torch.cuda.synchronize()
        clocks = Clocks(local) if head else None
        if clocks:
            clocks.start()
        ms, kern, launches = [], [], 0
        for _ in range(n_steps):
            a, k = one(S)
            ms.append(a)
            kern.append(k)
            launches += ev.last_call()["kernels"]
        torch.cuda.synchronize()
        if dist:
            tdist.barrier()
        clk = clocks.stop() if clocks else None
        e2e = [one(S, e2e=True)[0] for _ in range(e2e_steps or n_steps)] if head else []
        fl = ev.flops(S)
        sweep[frac] = {"chunks_per_s": n * 1000.0 / statistics.mean(ms), "p50_ms": statistics.median(ms),
                       "kernel_ms_mean": statistics.mean(kern), "flops_per_chunk": fl, "ms": ms, "kernel_ms": kern,
                       "e2e_ms": e2e, "clocks": clk, "alg_bytes": algorithmic_bytes(cfg, S, n), "S": S,
                       "launches": launches, "launches_per_call": launches / n_steps,
                       "path": ev.last_call()["path"], "steps": n_steps}
    if ev.status() != binding.OK:
        raise RuntimeError("device status reported an error")
    info = dict(ev.launch_info(), path=sweep[head_frac]["path"])
    ev.close()
    return cfg, n, sweep, info, int(obs.nbytes + noise.nbytes), int(h_out.numel() * 4)


def sweep_summary(workload, cfg, n, sweep):
    full = sweep.get(1.0)
    return {str(f): {"chunks_per_s": r["chunks_per_s"], "p50_ms": r["p50_ms"], "steps": r["steps"],
                     "kernel_ms": r["kernel_ms_mean"], "gflop_per_chunk": r["flops_per_chunk"] / 1e9,
                     "flop_ratio_vs_full": (full["flops_per_chunk"] / r["flops_per_chunk"]) if full else None,
                     "speedup_vs_full": (r["chunks_per_s"] / full["chunks_per_s"]) if full else None,
                     "roofline_frac": roofline(workload, cfg, n, r)["frac"],
                     "path": r["path"], "launches_per_call": r["launches_per_call"]}
            for f, r in sorted(sweep.items(), key=lambda kv: -kv[0])}


def subrecord(workload, steps, warmup):
    """Chunks/s, p50 and roofline fraction of one other workload (no e2e, no clocks)."""
    if workload == "population":
        line = run_population(argparse.Namespace(steps=steps, warmup=warmup), None, None)
        return {k: line[k] for k in ("metric", "value", "unit", "p50_ms", "ms_per_step", "roofline",
                                     "gpu_launches", "launch")} | {"workload": line["config"]["workload"],
                                                                   "launches_per_call": line["gpu_launches"] / steps}
    _, fracs, head_frac, kind = WORKLOADS[workload]
    cfg, n, sweep, info, _, _ = measure(workload, fracs, head_frac, kind, steps, warmup, e2e_steps=0)
    head = sweep[head_frac]
    return {"workload": f"{workload}-shaped: {describe(cfg, n)}", "value": head["chunks_per_s"],
            "unit": "chunks/s", "p50_ms": head["p50_ms"], "refresh_fraction": head_frac,
            "roofline": roofline(workload, cfg, n, head), "launches_per_call": head["launches_per_call"],
            "launch": info, "sweep": sweep_summary(workload, cfg, n, sweep)}


def run_ours(args, world, rank, local):
    import torch
    from paper_2607_20293_gb300 import binding, build

    torch.cuda.set_device(local)
    build.build()
    binding.load()
    name, fracs, head_frac, kind = WORKLOADS[args.workload]
    if args.fractions:
        fracs, head_frac = args.fractions, args.fractions[0]
    cfg, n, sweep, info, bytes_in, bytes_out = measure(args.workload, fracs, head_frac, kind, args.steps,
                                                       args.warmup, world, rank, local)
    headline = sweep[head_frac]
    total_s = sum(headline["ms"]) / 1000.0
    total_e2e = sum(headline["e2e_ms"]) / 1000.0
    if world > 1:
        total_s, total_e2e = max_over_ranks([total_s, total_e2e], "cuda")
    subs = {}
    if args.workload == DEFAULT_WORKLOAD and not args.no_subrecords and world == 1:
        for wl, st in SUBRECORDS:
            subs[wl] = subrecord(wl, st, args.warmup)
    if rank != 0:
        return None
    chunks = n * args.steps * world
    line = {
        "metric": "action chunks/s (p50 chunk latency and refresh-fraction sweep alongside)",
        "value": chunks / total_s,
        "unit": "chunks/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": 1000.0 * total_s / args.steps,
        "p50_ms": headline["p50_ms"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": cfg["dtype"],
        "data": "synthetic (seeded N(0,0.02) weights, N(0,1) observation features and noise)",
        "config": {"workload": f"{args.workload}-shaped: {describe(cfg, n)}", "batch": n,
                   "refresh_fraction": head_frac, "schedule": f"{kind} lattice, seed 3",
                   "l2": "flushed between timed steps (256 MiB write)",
                   "parallelism": f"replicas x{world}"},
        "sweep": sweep_summary(args.workload, cfg, n, sweep),
        "roofline": roofline(args.workload, cfg, n, headline),
        "e2e": {"value": chunks / total_e2e, "unit": "chunks/s", "h2d_bytes_per_step": bytes_in,
                "d2h_bytes_per_step": bytes_out,
                "lattice": "host lattice passed every call; the handle re-uploads it only when it changes"},
        "gpu_launches": headline["launches"],
        "clocks": headline["clocks"],
        "launch": info,
    }
    if subs:
        line["subrecords"] = subs
    return line, cfg


def run_redundancy(args, rank):
    """Dissimilarity maps (Eq. 6 and variants) from the all-refresh trace of
    REDUNDANCY_SAMPLES Push-T-shaped queries, and 64 guided schedules (Eq. 7)."""
    import torch
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    cfg = synth.config("pusht")
    N, U, T, H, E = REDUNDANCY_SAMPLES, 3 * cfg["n_layer"], cfg["n_steps"], cfg["horizon"], cfg["n_emb"]
    W = synth.make_weights(cfg, 0)
    ev = binding.Evo(cfg, W, N)
    obs = torch.from_numpy(synth.make_obs(cfg, N, 1)).cuda()
    noise = torch.from_numpy(synth.make_noise(cfg, N, 2)).cuda()
    trace = torch.zeros((T, U, N, H, E), device="cuda")
    ones = np.ones((U, T), np.uint8)
    flush = torch.empty(L2_FLUSH_BYTES // 4, device="cuda")

    def timed(fn, reps):
        out = []
        for i in range(max(3, args.warmup) + reps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            if i >= max(3, args.warmup):
                out.append(a.elapsed_time(b))
        return statistics.median(out)

    clocks = Clocks(int(os.environ.get("LOCAL_RANK", "0")))
    clocks.start()
    trace_ms = timed(lambda: ev.denoise(obs, noise, ones, trace=trace), args.steps)
    maps = {}
    for m in binding.METRICS:
        maps[m] = timed(lambda: binding.redundancy_map(trace, m), args.steps)
    d = binding.redundancy_map(trace, "cosine")
    P, K = 64, 240
    rnd = torch.from_numpy(synth.guided_randoms(P, K, 7).view(np.int64)).cuda()
    guided_ms = timed(lambda: binding.guided_schedules(d, K, rnd), args.steps)
    clk = clocks.stop()
    n = H * E
    pair_flops = 2.0 * U * N * n * T * (T + 1) / 2          # cosine: one multiply-add per entry and pair
    sm = torch.cuda.get_device_properties(0).multi_processor_count
    mhz = (clk or {}).get("sm_max_mhz") or 2070.0
    peak = sm * FP32_LANES_PER_SM * 2 * mhz * 1e6 / 1e12
    achieved = pair_flops / (maps["cosine"] * 1e-3) / 1e12
    return {
        "metric": "redundancy map latency (Eq. 6 cosine from 16 all-refresh Push-T queries) and guided schedules/s (Eq. 7)",
        "value": maps["cosine"], "unit": "ms", "higher_is_better": False, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "dtype": "f32", "data": "synthetic",
        "config": {"workload": f"redundancy map: {describe(cfg, N)}, U {U} x T {T} lattice, n {n} entries per activation",
                   "l2": "flushed between timed calls (256 MiB write)"},
        "map_ms": maps, "trace_collection_ms": trace_ms,
        "guided": {"schedules": P, "K": K, "ms": guided_ms, "schedules_per_s": P / (guided_ms * 1e-3)},
        "roofline": {"bound": "alu", "kernel": "pair_kernel (cosine)", "achieved": achieved, "peak": peak,
                     "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
                     "peak_source": f"{sm} SMs x {FP32_LANES_PER_SM} FP32 lanes x 2 FLOP x {mhz:.0f} MHz"},
        "clocks": clk,
    }


def published_lattices(task: str):
    """BAC and EVO lattices [24][100] of the paper's appendix tables (tests/golden)."""
    bac = np.zeros((24, 100), np.uint8)
    evo = np.zeros((24, 100), np.uint8)
    b = 0
    with open(os.path.join(ROOT, "tests", "golden", f"schedules_{task}.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            _, bl, el = [p.strip() for p in line.split(";")]
            bac[b, [int(v) for v in bl.split()]] = 1
            evo[b, [int(v) for v in el.split()]] = 1
            b += 1
    return bac, evo


POP_MAP_SEED, POP_BUDGET_SEED, POP_RANDOM_SEED = 5, 6, 7
POP_METRIC = "candidate action chunks/s (P x N per evo_denoise_population call, p50 call latency alongside)"


def _oracle_pop_chunk(args):
    """One (candidate, observation) chunk of the population workload on the oracle;
    the candidate lattice is drawn with the oracle's own Eq. 7 sampler."""
    p, seed = args
    from oracle import evo_oracle as O
    cfg = synth.config("population")
    W = synth.make_weights(cfg, 0)
    P, L, T = cfg["n_candidates"], cfg["n_layer"], cfg["n_steps"]
    d = synth.dissimilarity_map(L, T, POP_MAP_SEED)
    Ks = synth.population_budgets(P, L * T, POP_BUDGET_SEED)
    rnd = synth.guided_randoms(P, int(Ks.max()), POP_RANDOM_SEED)
    S = O.guided_sample(O.guided_weights(d, 0.05, 2), int(Ks[p % P]), rnd[p % P]).reshape(L, T)
    O.denoise(W, cfg, synth.make_obs(cfg, 1, 1000 + seed), synth.make_noise(cfg, 1, 2000 + seed), S)
    return 1


def run_population(args, pool, workers):
    """Population evaluation: P candidate lattices [P][L][T] drawn by the library's
    Eq. 7 sampler from a synthetic dissimilarity map (densities 5-60 %), each on
    N observations, plus the all-refresh reference, in one evo_denoise_population
    call; dev_l2 per candidate.  value = candidate chunks (P x N) per second."""
    import torch
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    cfg = synth.config("population")
    W = synth.make_weights(cfg, 0)
    P, N, L, T = cfg["n_candidates"], cfg["batch"], cfg["n_layer"], cfg["n_steps"]
    obs, noise = synth.make_obs(cfg, N, 1), synth.make_noise(cfg, N, 2)
    d = torch.from_numpy(synth.dissimilarity_map(L, T, POP_MAP_SEED).astype(np.float32)).cuda()
    Ks = synth.population_budgets(P, L * T, POP_BUDGET_SEED)
    rnd = torch.from_numpy(synth.guided_randoms(P, int(Ks.max()), POP_RANDOM_SEED).view(np.int64)).cuda()
    pop = torch.cat([binding.guided_schedules(d, int(Ks[p]), rnd[p:p + 1, :int(Ks[p])]) for p in range(P)])
    ev = binding.Evo(cfg, W, (P + 1) * N)
    d_obs, d_noise = torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda()
    h_obs, h_noise = torch.from_numpy(obs).pin_memory(), torch.from_numpy(noise).pin_memory()
    out = torch.empty((P, N, cfg["horizon"], cfg["action_dim"]), device="cuda")
    dev = torch.empty((P,), device="cuda")
    h_dev = torch.empty((P,)).pin_memory()
    flush = torch.empty(L2_FLUSH_BYTES // 4, device="cuda")
    k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    k0.record()
    k1.record()
    ev.set_profile_events(k0, k1)

    def one(e2e=False):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        if e2e:
            d_obs.copy_(h_obs, non_blocking=True)
            d_noise.copy_(h_noise, non_blocking=True)
        ev.population(d_obs, d_noise, pop, out=out, dev=dev)
        if e2e:
            h_dev.copy_(dev, non_blocking=True)
        b.record()
        b.synchronize()
        return a.elapsed_time(b), k0.elapsed_time(k1)

    for _ in range(max(3, args.warmup)):
        one()
    clocks = Clocks(int(os.environ.get("LOCAL_RANK", "0")))
    clocks.start()
    steps, kern, launches = [], [], 0
    for _ in range(args.steps):
        ms, kms = one()
        steps.append(ms)
        kern.append(kms)
        launches += ev.last_call()["kernels"]
    clk = clocks.stop()
    e2e = [one(e2e=True)[0] for _ in range(args.steps)]
    if ev.status() != binding.OK:
        raise RuntimeError("device status reported an error")
    S_host = pop.cpu().numpy()
    flops = N * (sum(ev.flops(S_host[p]) for p in range(P)) + ev.flops(np.ones((L, T), np.uint8)))
    full = N * (P + 1) * ev.flops(np.ones((L, T), np.uint8))
    kern_ms = statistics.mean(kern)
    peaks = measured_peaks()
    sustained = statistics.median(steps) >= SUSTAINED_STEP_MS
    key = "bf16_tflops_sustained" if sustained else "bf16_tflops"
    peak = peaks.get(key) or (1700.0 if sustained else 1900.0)
    peak_src = (("measured bf16 sustained (timed step >= %g ms)" % SUSTAINED_STEP_MS) if sustained
                else "measured bf16 burst") if key in peaks else "fallback"
    achieved = flops / (kern_ms / 1000.0) / 1e12
    path = ev.last_call()["path"]
    info = dict(ev.launch_info(), path=path)
    ev.close()
    line = {
        "metric": POP_METRIC,
        "value": P * N * 1000.0 / statistics.mean(steps), "unit": "chunks/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": statistics.mean(steps), "p50_ms": statistics.median(steps),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": cfg["dtype"],
        "data": "synthetic (seeded weights, observations, noise; candidates by Eq. 7 from a synthetic map)",
        "config": {"workload": f"population evaluation: {P} candidates x {N} observations + the all-refresh "
                               f"reference, lattice {L} x {T}; {describe(cfg, N)}",
                   "candidates": P, "observations": N, "density": [float(Ks.min()) / (L * T), float(Ks.max()) / (L * T)],
                   "l2": "flushed between timed steps (256 MiB write)", "parallelism": "replicas x1"},
        "flop_ratio_vs_all_full": full / flops,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                     "traffic": recorded_traffic("population"), "peak_source": peak_src,
                     "kernel": ("batch-wide launch sequence of one call (tcgen05 GEMMs, attention, row kernels)"
                                if path == "wide" else "evo::job_kernel (persistent cluster loop)"),
                     "algorithmic_per_launch": flops, "kernel_ms": kern_ms},
        "e2e": {"value": P * N * 1000.0 / statistics.mean(e2e), "unit": "chunks/s",
                "h2d_bytes_per_step": int(obs.nbytes + noise.nbytes), "d2h_bytes_per_step": int(h_dev.numel() * 4)},
        "gpu_launches": launches, "clocks": clk, "launch": info,
    }
    if pool is not None:
        pool.map(_oracle_pop_chunk, [(p, p) for p in range(workers)])          # warm the workers
        n = workers * 2
        t0 = time.perf_counter()
        pool.map(_oracle_pop_chunk, [(3 * i, 100 + i) for i in range(n)])
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": n / dt, "unit": "chunks/s", "cores": workers, "kind": "oracle",
                                "sample": f"{n} single (candidate, observation) chunks of the same population "
                                          f"(candidates 0, 3, 6, ...), one float64 numpy oracle process per core"}
    return line


def run_schedules(args):
    """Push-T batch 1: chunks/s of the full lattice, EfficientVLA's fixed interval
    (M = 8, 10), the paper's BAC and EVO Push-T lattices and Bernoulli(0.125)."""
    import torch
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    cfg = synth.config("pusht")
    W = synth.make_weights(cfg, 0)
    ev = binding.Evo(cfg, W, 1)
    obs = torch.from_numpy(synth.make_obs(cfg, 1, 1)).cuda()
    noise = torch.from_numpy(synth.make_noise(cfg, 1, 2)).cuda()
    out = torch.empty((1, cfg["horizon"], cfg["action_dim"]), device="cuda")
    flush = torch.empty(L2_FLUSH_BYTES // 4, device="cuda")
    bac, evo = published_lattices("pusht")
    lattices = {"full": np.ones((24, 100), np.uint8),
                "EfficientVLA M=8": binding.schedule_fixed_interval(24, 100, 8),
                "EfficientVLA M=10": binding.schedule_fixed_interval(24, 100, 10),
                "BAC (paper, Push-T)": bac, "EVO (paper, Push-T, K=240)": evo,
                "Bernoulli 0.125": schedule(cfg, 0.125, "bernoulli")}
    clocks = Clocks(int(os.environ.get("LOCAL_RANK", "0")))
    clocks.start()
    rows = {}
    for name, S in lattices.items():
        ts = []
        for i in range(max(3, args.warmup) + args.steps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            ev.denoise(obs, noise, S, out=out)
            b.record()
            b.synchronize()
            if i >= max(3, args.warmup):
                ts.append(a.elapsed_time(b))
        rows[name] = {"cells": int(S.sum()), "gflop_per_chunk": ev.flops(S) / 1e9, "p50_ms": statistics.median(ts),
                      "chunks_per_s": 1000.0 / statistics.mean(ts)}
    clk = clocks.stop()
    full = rows["full"]
    for r in rows.values():
        r["flop_ratio_vs_full"] = full["gflop_per_chunk"] / r["gflop_per_chunk"]
        r["speedup_vs_full"] = r["chunks_per_s"] / full["chunks_per_s"]
    best = rows["EVO (paper, Push-T, K=240)"]
    return {"metric": "action chunks/s per schedule (Push-T-shaped, batch 1)", "value": best["chunks_per_s"],
            "unit": "chunks/s", "higher_is_better": True, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "dtype": cfg["dtype"], "data": "synthetic",
            "config": {"workload": f"published / baseline schedules: {describe(cfg, 1)}; value = the paper's EVO lattice",
                       "l2": "flushed between timed steps (256 MiB write)"},
            "schedules": rows, "clocks": clk}


def run_search(args):
    """Genetic search (population 30, elites 10, 30 generations, K = 240) on the
    Push-T-shaped policy; fitness = -dev_l2 of evo_denoise_population over 4
    observations (GPU), half of the initial individuals guided by the Eq. 6 map
    of 16 all-refresh queries."""
    import torch
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    cfg = synth.config("pusht")
    W = synth.make_weights(cfg, 0)
    U, T, H, E = 3 * cfg["n_layer"], cfg["n_steps"], cfg["horizon"], cfg["n_emb"]
    n_fit, n_map, pop_size = 4, REDUNDANCY_SAMPLES, 30
    ev = binding.Evo(cfg, W, max((pop_size + 1) * n_fit, n_map))
    obs = torch.from_numpy(synth.make_obs(cfg, n_fit, 5)).cuda()
    noise = torch.from_numpy(synth.make_noise(cfg, n_fit, 6)).cuda()
    mobs = torch.from_numpy(synth.make_obs(cfg, n_map, 7)).cuda()
    mnoise = torch.from_numpy(synth.make_noise(cfg, n_map, 8)).cuda()
    calls = []

    def fitness(S):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        _, dev = ev.population(obs, noise, S.astype(np.uint8), want_actions=False)
        b.record()
        out = [-float(v) for v in dev.cpu().numpy()]
        calls.append((len(S), a.elapsed_time(b), ev.last_call()["path"]))
        return out

    torch.cuda.synchronize()
    t0 = time.perf_counter()
    tr = torch.zeros((T, U, n_map, H, E), device="cuda")
    ev.denoise(mobs, mnoise, np.ones((U, T), np.uint8), trace=tr)
    d = binding.redundancy_map(tr, "cosine").cpu().numpy()
    t1 = time.perf_counter()
    S, best, st = binding.search(U, T, 240, fitness, d_map=d, population=pop_size, elites=10, generations=30,
                                 guided=15, seed=1)
    t2 = time.perf_counter()
    gpu_ms = sum(c[1] for c in calls)
    flops_ratio = ev.flops(np.ones((U, T), np.uint8)) / ev.flops(S)
    return {"metric": "schedule search wall time (GA: population 30, elites 10, 30 generations, K = 240; "
                      "fitness -dev_l2 of evo_denoise_population over 4 observations)",
            "value": t2 - t0, "unit": "s", "higher_is_better": False, "n_gpus": 1, "steps": 1, "warmup": 0,
            "dtype": cfg["dtype"], "data": "synthetic",
            "config": {"workload": f"schedule search: {describe(cfg, n_fit)}, lattice {U} x {T}"},
            "map_s": t1 - t0, "search_s": t2 - t1, "generations": st["generations"],
            "evaluations": st["evaluations"], "memo_hits": st["memo_hits"],
            "fitness_calls": len(calls), "fitness_gpu_ms": gpu_ms,
            "candidate_evaluations_per_s": st["evaluations"] / (t2 - t1),
            "population_path": calls[-1][2] if calls else None,
            "best_fitness": best, "best_flop_ratio_vs_full": flops_ratio, "best_cells": int(S.sum())}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-subrecords", action="store_true",
                    help="default workload only: skip the other workloads' sub-records")
    ap.add_argument("--fractions", type=float, nargs="*", default=None,
                    help="refresh fractions to sweep (default: the workload's; the headline is the first)")
    args = ap.parse_args()
    world, rank, local = dist_env()
    name, fracs, head_frac, kind = WORKLOADS[args.workload]
    if args.fractions:
        head_frac = args.fractions[0]
    if args.workload == "redundancy" and args.impl == "ours":
        if rank == 0:
            print(json.dumps(run_redundancy(args, rank)))
        return
    if args.workload == "search" and args.impl == "ours":
        if rank == 0:
            print(json.dumps(run_search(args)))
        return
    if args.workload == "schedules" and args.impl == "ours":
        if rank == 0:
            print(json.dumps(run_schedules(args)))
        return
    if args.workload == "population" and args.impl == "ours":
        if rank == 0:
            pool = workers = None
            if world == 1 and not args.no_cpu_baseline:
                pool, workers = make_pool()          # spawned before the first GPU call
            try:
                print(json.dumps(run_population(args, pool, workers)))
            finally:
                if pool is not None:
                    pool.close()
        return

    if args.impl == "reference":
        if rank != 0:
            return
        pool, workers = make_pool()

        def rnd(base):
            if args.workload != "population":
                return oracle_round(pool, name, head_frac, kind, workers, base_seed=base)
            t0 = time.perf_counter()
            pool.map(_oracle_pop_chunk, [(3 * (base + i), base + i) for i in range(workers)])
            return time.perf_counter() - t0

        try:
            for _ in range(max(1, min(args.warmup, 3))):
                rnd(0)
            times = [rnd(10 * i) for i in range(args.steps)]
        finally:
            pool.close()
        total = sum(times)
        v = workers * args.steps / total
        cfg = synth.config(name)
        print(json.dumps({
            "impl": "reference",
            "metric": POP_METRIC if args.workload == "population"
            else "action chunks/s (p50 chunk latency and refresh-fraction sweep alongside)",
            "value": v, "unit": "chunks/s", "n_gpus": 0, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * total / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{args.workload}-shaped: {describe(cfg, cfg['batch'])}", "batch": cfg["batch"],
                       "refresh_fraction": head_frac, "schedule": f"{kind} lattice, seed 3"},
            "cpu_baseline": {"value": v, "unit": "chunks/s", "cores": workers, "kind": "oracle",
                             "sample": f"each step: a subset of {workers} single-sample chunks of the workload's "
                                       f"{cfg['batch']} samples, one float64 numpy oracle process per core"},
            "e2e": {"value": v, "unit": "chunks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }))
        return

    pool = workers = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        pool, workers = make_pool()          # spawned before the first GPU call
    dist = world > 1
    if dist:
        import torch
        import torch.distributed as tdist
        torch.cuda.set_device(local)
        tdist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    res = run_ours(args, world, rank, local)
    if res is not None:
        line, cfg = res
        if pool is not None:
            line["cpu_baseline"] = cpu_baseline(name, head_frac, kind, pool, workers)
            pool.close()
        print(json.dumps(line))
    if dist:
        tdist.barrier()
        tdist.destroy_process_group()


if __name__ == "__main__":
    main()
