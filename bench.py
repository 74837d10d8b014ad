"""Benchmark of the MeanField joint-configuration scorer on GB300.

One step = one exhaustive surrogate search over the large workload: N = 6
models with 24 options each (24**6 = 191,102,976 joint configurations),
12->64->64->2 predictors, VRAM cap 180 GB, top-32 and the feasible count,
enumerated in launches of 2**24 candidates.  All inputs are seeded synthetic
draws (paper_2609_02109_gb300.workload).  The GA decision latency (N = 5,
population 1024, 100 generations, 8 scenarios), the fixed-context decision with
the paper's GA settings (Sec. IV: population 100, 30 generations), the stress
workload and the fixed-context scans are measured after the timed steps and
reported in the same JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--precision bf16|fp32]
    python bench.py --impl reference ...   # the CPU oracle as the reference arm

Multi-GPU (torchrun, one rank per GPU): the ranks split the same space into
contiguous index ranges, search their range on their GPU and exchange the k best
(score, index) pairs and the feasible counts in one NCCL all-gather
(paper_2609_02109_gb300.shard.search_sharded): the total work per step is fixed,
so the scaling is strong.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2609_02109_gb300 import workload as W  # noqa: E402

METRIC = "joint configs scored/s (N=6 exhaustive, % of roofline); p50 GA decision ms"
UNIT = "configs/s"
K_TOP = 32
CHUNK = 1 << 24
L2_FLUSH_BYTES = 256 << 20

# DRAM bytes (read + write) of one scoring launch from the ncu capture of the scoring
# kernel on this workload, valid only while the kernel's sources are the ones that were
# captured (sha256 prefix of k_tc.cu + mf_internal.cuh).  fp32: a first-pass launch of
# the exact variant (models 0-2), which writes the 16-byte partial record of each of its
# 2^24 candidates for the second pass (which reads them back).
NCU_TRAFFIC = {"bf16": ("0e1142bf651b8a11", 2091008), "fp32": ("0e1142bf651b8a11", 207531776)}


def _traffic(prec):
    import hashlib
    ent = NCU_TRAFFIC.get(prec)
    if ent is None:
        return None
    h = hashlib.sha256()
    for f in ("k_tc.cu", "mf_internal.cuh"):
        with open(os.path.join(ROOT, "paper_2609_02109_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return ent[1] if h.hexdigest()[:16] == ent[0] else None


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "sm_max_mhz": 2070.0}, "fallback"


def flops_per_candidate(prob) -> int:
    """Algorithmic FLOPs of one candidate: 2 x (multiply-adds of every layer) x N."""
    din = prob["d_local"] + 4
    h1, h2 = prob["hidden1"], prob["hidden2"]
    macs = din * h1 + (h1 * h2 + h2 * 2 if h2 else h1 * 2)
    return 2 * macs * int(prob["n_options"].size)


def workload_config(prec):
    return {
        "workload": "large exhaustive: N=6 models x 24 options (24^6 = 191,102,976 joint configs), "
                    "per-model MLP 12->64->64->2, VRAM cap 180 GB, SLA~U(0.5,2), w~U(0.5,1.5), "
                    "top-32 + feasible count, launches of 2^24 candidates",
        "precision": prec,
        "seed": 3,
        "l2": "flushed between timed steps (256 MiB device write); scoring inputs are on-chip "
              "tables and weights",
    }


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.out = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.out.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.out:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1].split()[0]))
                mx.append(float(parts[2].split()[0]))
            except ValueError:
                continue
            for name, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU baseline: the oracle on a bounded sample of the same workload
# ---------------------------------------------------------------------------
def cpu_baseline(prob, target_s=15.0):
    from oracle.oracle import Oracle
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    o = Oracle(prob, nthreads=cores)
    n = 200000
    while True:  # grow the sample until it takes about target_s (at least 10 s)
        t = time.perf_counter()
        o.exhaustive(K_TOP, lo=0, hi=n)
        dt = time.perf_counter() - t
        if dt >= 10.0 or n >= 24 ** 6:
            break
        n = int(min(n * max(2.0, target_s / max(dt, 1e-3)), 24 ** 6))
    # one core, on a sample of about a fifth of that time
    o1 = Oracle(prob, nthreads=1)
    n1 = max(20000, n // (5 * max(cores, 1)))
    t = time.perf_counter()
    o1.exhaustive(K_TOP, lo=0, hi=n1)
    dt1 = time.perf_counter() - t
    return {"value": n / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"fp64 C oracle exhaustive search (top-32 + count) over indices [0, {n}) "
                      f"of the same N=6 space, {dt:.1f} s",
            "single_thread": {"value": n1 / dt1, "unit": UNIT, "cores": 1,
                              "sample": f"indices [0, {n1}), {dt1:.1f} s"}}


def run_reference(args):
    """Reference arm: the CPU oracle, timed on the host cores, per step a bounded sample."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from oracle.oracle import Oracle, build
    build()
    prob = W.large(precision="fp32")
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    o = Oracle(prob, nthreads=cores)
    t = time.perf_counter()
    o.exhaustive(K_TOP, lo=0, hi=20000)
    rate = 20000 / max(time.perf_counter() - t, 1e-6)
    budget = 150.0 / max(args.steps + args.warmup, 1)
    n = int(min(max(rate * min(budget, 20.0), 5e4), 5e7))
    for _ in range(args.warmup):
        o.exhaustive(K_TOP, lo=0, hi=min(n, 20000))
    times = []
    for s in range(args.steps):
        lo = (s * n) % (prob_size := 24 ** 6)
        hi = min(lo + n, prob_size)
        t = time.perf_counter()
        o.exhaustive(K_TOP, lo=lo, hi=hi)
        times.append(time.perf_counter() - t)
    total = sum(times)
    value = n * args.steps / total
    sample = f"fp64 C oracle exhaustive search over {n} consecutive indices per step of the N=6 space"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config("f64"),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def fp32_peak(torch, device):
    """The fp32 FMA rate of a cuBLAS fp32 GEMM with TF32 off (8192^3, best of five
    after two warm-ups): the measured stand-in for the FP32 pipe's peak, as the bf16
    peak is cuBLAS's bf16 GEMM."""
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        n = 8192
        a = torch.randn(n, n, device=f"cuda:{device}", dtype=torch.float32)
        b = torch.randn(n, n, device=f"cuda:{device}", dtype=torch.float32)
        for _ in range(2):
            torch.matmul(a, b)
        best = float("inf")
        stream = torch.cuda.current_stream(device)
        for _ in range(5):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            torch.matmul(a, b)
            e1.record(stream)
            e1.synchronize()
            best = min(best, e0.elapsed_time(e1))
        del a, b
        return 2.0 * n ** 3 / (best / 1e3) / 1e12
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev


def tight_throughput(mf, torch, device):
    """The large workload's space with SLA ceilings ~ U(0.1, 0.9), where the latency
    mask binds: the SLA mask, the bf16 shortlist band around the ceilings and the fp32
    re-scoring of the shortlist are all on the timed path."""
    prob = W.large(precision="bf16")
    W.set_scenario(prob, 31, W.TIGHT_SLA)
    n = 24 ** 6
    stream = torch.cuda.current_stream(device)
    peaks, src = _peaks()
    with mf.Context(prob, device=device) as ctx:
        ctx.search(K_TOP, chunk=CHUNK)
        ms, score_ms = [], []
        for _ in range(3):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize(device)
            e0.record(stream)
            res = ctx.search(K_TOP, chunk=CHUNK)
            e1.record(stream)
            e1.synchronize()
            st = ctx.stats()
            ms.append(e0.elapsed_time(e1))
            score_ms.append(st["score_ms_last"] / st["score_launches_last"])
    launch_ms = float(np.median(score_ms))
    achieved = flops_per_candidate(prob) * (n / 12) / (launch_ms / 1e3) / 1e12
    peak = float(peaks["bf16_tflops"])
    return {"workload": "large space (N=6 x 24 options), scenario 31 with SLA ~ U(0.1, 0.9): latency mask binds",
            "value": n / (float(np.median(ms)) / 1e3), "unit": UNIT, "ms": float(np.median(ms)),
            "feasible_fraction": res["count"] / n, "count": res["count"], "best": res["best_idx"],
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                         "frac": achieved / peak, "launch_ms": launch_ms,
                         "peak_source": f"{src} bf16 burst"}}


# tf32 dense tensor rate relative to bf16 (NVIDIA's nominal 1.1 vs 2.25 PFLOP/s)
TF32_PER_BF16 = 1.1 / 2.25


def exact_roofline(achieved, sgemm_tflops):
    """Roofline of the exact fp32 tensor-core variant: every product costs three tf32
    products (hi.hi, hi.lo, lo.hi), so its ceiling is a third of the tf32 peak (the
    measured bf16 burst x the nominal tf32 / bf16 ratio)."""
    peaks, src = _peaks()
    tf32 = float(peaks["bf16_tflops"]) * TF32_PER_BF16
    return {"bound": "tensor", "achieved": achieved, "peak": tf32, "unit": "TFLOP/s", "frac": achieved / tf32,
            "frac_of_split_ceiling": 3 * achieved / tf32,
            "peak_source": f"{src} bf16 burst x {TF32_PER_BF16:.3f} (nominal tf32 / bf16); 3 tf32 products per product",
            "cuda_core_peak": sgemm_tflops}


def exact_throughput(mf, torch, device, sgemm_tflops):
    """The exact fp32 search of the large workload: the tensor-core variant (3-term
    tf32 split) and, for comparison, the CUDA-core scorer."""
    prob = W.large(precision="fp32")
    n = 24 ** 6
    stream = torch.cuda.current_stream(device)
    out = {}
    for prec in ("fp32", "fp32_simt"):
        with mf.Context(prob, device=device, precision=prec) as ctx:
            ctx.search(K_TOP, chunk=CHUNK)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize(device)
            e0.record(stream)
            res = ctx.search(K_TOP, chunk=CHUNK)
            e1.record(stream)
            e1.synchronize()
            st = ctx.stats()
        ms = e0.elapsed_time(e1)
        launch_ms = st["score_ms_last"] / st["score_launches_last"]
        achieved = flops_per_candidate(prob) * (n / st["score_launches_last"]) / (launch_ms / 1e3) / 1e12
        out[prec] = dict(value=n / (ms / 1e3), ms=ms, best=res["best_idx"], count=res["count"],
                         path=int(st["scoring_path"]), achieved=achieved, launch_ms=launch_ms,
                         launches=int(st["score_launches_last"]))
    tc, simt = out["fp32"], out["fp32_simt"]
    roof = exact_roofline(tc["achieved"], sgemm_tflops) if tc["path"] == 2 else \
        {"bound": "fp32", "achieved": tc["achieved"], "peak": sgemm_tflops, "unit": "TFLOP/s",
         "frac": tc["achieved"] / sgemm_tflops, "peak_source": "measured cuBLAS fp32 GEMM (TF32 off), this run"}
    roof["launch_ms"] = tc["launch_ms"]
    return {"workload": "large exhaustive, exact fp32 path (tensor cores, 3-term tf32 split; "
                        "two weight passes of three models)", "value": tc["value"], "unit": UNIT, "ms": tc["ms"],
            "best": tc["best"], "count": tc["count"], "roofline": roof,
            "cuda_cores": {"value": simt["value"], "unit": UNIT, "ms": simt["ms"], "best": simt["best"],
                           "count": simt["count"], "achieved": simt["achieved"], "unit_achieved": "TFLOP/s",
                           "frac": simt["achieved"] / sgemm_tflops,
                           "peak_source": "measured cuBLAS fp32 GEMM (TF32 off), this run"}}


def stress_throughput(mf, torch, device):
    """The stress workload (2^32 candidates, bf16, eight 20->128->128->2 predictors in
    three shared-memory passes), one warm-up and one timed search."""
    prob = W.stress(precision="bf16")
    n = 2 ** 32
    stream = torch.cuda.current_stream(device)
    with mf.Context(prob, device=device) as ctx:
        ctx.search(64, chunk=1 << 26)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(device)
        e0.record(stream)
        res = ctx.search(64, chunk=1 << 26)
        e1.record(stream)
        e1.synchronize()
        st = ctx.stats()
    ms = e0.elapsed_time(e1)
    peaks, src = _peaks()
    achieved = flops_per_candidate(prob) * n / (st["score_ms_last"] / 1e3) / 1e12
    return {"workload": "stress exhaustive: N=8 x 16 options (2^32 joint configs), 20->128->128->2 bf16, "
                        "soft latency penalty 0.1, VRAM cap 180 GB, top-64, chunks of 2^26",
            "value": n / (ms / 1e3), "unit": UNIT, "ms": ms, "count": res["count"],
            "roofline": {"achieved": achieved, "peak": float(peaks["bf16_tflops_sustained"]), "unit": "TFLOP/s",
                         "frac": achieved / float(peaks["bf16_tflops_sustained"]),
                         "flops_per_candidate": flops_per_candidate(prob), "peak_source": f"{src} bf16 sustained"}}


def fixed_context_throughput(mf, torch, device):
    """Fixed-context mode (observed state held fixed, Eq. 3 utility): table build and
    the table-lookup exhaustive scan over the large and stress spaces."""
    peaks, _ = _peaks()
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    issue = sms * 4 * 32 * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6  # lane-instructions/s
    out = {}
    stream = torch.cuda.current_stream(device)
    for name, prob, seed in (("large", W.large(precision="fp32"), 3), ("stress", W.stress(precision="fp32"), 5)):
        fc = W.fc_scenario(prob, seed)
        n = int(np.prod(prob["n_options"].astype(np.float64)))
        N = int(prob["n_options"].size)
        with mf.Context(prob, device=device) as ctx:
            t0 = time.perf_counter()
            ctx.fc_set(fc)
            set_ms = 1e3 * (time.perf_counter() - t0)
            ctx.fc_search(32, chunk=1 << 30)
            times, scans = [], []
            for _ in range(5):  # median of five searches
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize(device)
                e0.record(stream)
                res = ctx.fc_search(32, chunk=1 << 30)
                e1.record(stream)
                e1.synchronize()
                times.append(e0.elapsed_time(e1))
                scans.append(ctx.stats()["score_ms_last"])
        ms = float(np.median(times))
        ops = 3 * N * n / (float(np.median(scans)) / 1e3)  # N table loads and 2N adds per candidate
        out[name] = {"candidates": n, "value": n / (ms / 1e3), "unit": UNIT, "ms": ms, "fc_set_ms": set_ms,
                     "count": res["count"],
                     "roofline": {"bound": "alu", "achieved": ops, "peak": issue, "unit": "lane-ops/s",
                                  "frac": ops / issue,
                                  "peak_source": f"{sms} SMs x 4 schedulers x 32 lanes x max SM clock",
                                  "ops_per_candidate": 3 * N}}
    return out


def ga_latency(mf, torch, device, decisions_per_scenario):
    """p50/p99 of complete GA decisions (host call -> result on host) over 8 scenarios."""
    g = W.GA_PARAMS
    wall, dev = [], []
    gaps = []
    for sc in W.GA_SCENARIO_SEEDS:
        prob = W.ga_scenario(sc)
        with mf.Context(prob, device=device) as ctx:
            best = ctx.search(1)["best_score"]
            ctx.ga_run(g, 999)  # first call: kernel attributes, buffers (or the graph capture)
            stream = torch.cuda.current_stream(device)
            for j in range(decisions_per_scenario):
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize(device)
                t0 = time.perf_counter()
                e0.record(stream)
                J, genome = ctx.ga_run(g, W.GA_RUN_SEEDS[j % len(W.GA_RUN_SEEDS)])
                e1.record(stream)
                t1 = time.perf_counter()
                e1.synchronize()
                wall.append(1e3 * (t1 - t0))
                dev.append(e0.elapsed_time(e1))
                gaps.append(100.0 * (best - J) / abs(best) if best != 0 else 0.0)
    q = lambda a, p: float(np.percentile(np.asarray(a), p))  # noqa: E731
    return {"p50_ms": q(wall, 50), "p99_ms": q(wall, 99), "device_p50_ms": q(dev, 50),
            "decisions": len(wall), "scenarios": len(W.GA_SCENARIO_SEEDS),
            "gap_pct_avg": float(np.mean(gaps)), "gap_pct_worst": float(np.max(gaps)),
            "config": "N=5 paper-scale problem (78,732 configs), pop 1024, 100 generations, "
                      "tournament 4, uniform crossover, mutation 0.05, elitism 1, fp32 fitness",
            "gap_vs": "exhaustive optimum of the same scenario (fp32)"}


def paper_ga_latency(mf, torch, device, decisions_per_scenario):
    """p50/p99 of complete fixed-context decisions with the paper's GA (Sec. III-B,
    Sec. IV): mf_fc_set (predictions for every option under the observed state and the
    utility table) followed by mf_fc_ga_run, host call -> decision on host, over the
    8 scenarios of the N=5 problem."""
    g = W.PAPER_GA_PARAMS
    wall, set_ms, ga_ms, gaps, exh = [], [], [], [], []
    infeasible = 0
    for sc in W.GA_SCENARIO_SEEDS:
        prob = W.ga_scenario(sc)
        fc = W.fc_scenario(prob, sc)
        with mf.Context(prob, device=device) as ctx:
            ctx.fc_set(fc)
            best = ctx.fc_search(1)["best_score"]
            infeasible += 0 if np.isfinite(best) else 1
            ctx.fc_ga_run(g, 999)  # first call: kernel attributes and buffers
            for j in range(decisions_per_scenario):
                torch.cuda.synchronize(device)
                t0 = time.perf_counter()
                ctx.fc_set(fc)
                t1 = time.perf_counter()
                J, genome = ctx.fc_ga_run(g, W.GA_RUN_SEEDS[j % len(W.GA_RUN_SEEDS)])
                t2 = time.perf_counter()
                wall.append(1e3 * (t2 - t0))
                set_ms.append(1e3 * (t1 - t0))
                ga_ms.append(1e3 * (t2 - t1))
                if np.isfinite(best):  # (a landscape whose floors no configuration meets has no gap)
                    gaps.append(100.0 * (best - J) / abs(best) if best != 0 else 0.0)
                # the exhaustive decision over the same landscape, for the paper's GA-vs-exhaustive ratio
                torch.cuda.synchronize(device)
                t0 = time.perf_counter()
                ctx.fc_set(fc)
                ctx.fc_search(1)
                exh.append(1e3 * (time.perf_counter() - t0))
    q = lambda a, p: float(np.percentile(np.asarray(a), p))  # noqa: E731
    return {"p50_ms": q(wall, 50), "p99_ms": q(wall, 99), "exhaustive_p50_ms": q(exh, 50), "fc_set_p50_ms": q(set_ms, 50),
            "fc_ga_run_p50_ms": q(ga_ms, 50), "decisions": len(wall), "scenarios": len(W.GA_SCENARIO_SEEDS),
            "gap_pct_avg": float(np.mean(gaps)) if gaps else None,
            "gap_pct_worst": float(np.max(gaps)) if gaps else None,
            "scenarios_without_feasible_config": infeasible,
            "config": "N=5 paper-scale problem (78,732 configs), fixed observed state, Eq. 3 utility, "
                      "pop 100, 30 generations, tournament 3, crossover p 0.7, mutation 0.1, elitism 1, "
                      "repair by rejection sampling",
            "gap_vs": "exhaustive optimum of the same fixed-context landscape",
            "paper_context_ms": "26 (8.5 local predictions + 17 GA; exhaustive 131), the paper's own measurement "
                                "on its hardware: context only"}


def run_gpu(args):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    import __graft_entry__
    if rank == 0 or world == 1:
        __graft_entry__.build()
    if dist:
        dist.barrier()
    from paper_2609_02109_gb300 import mf

    from paper_2609_02109_gb300 import shard

    prec = args.precision
    prob = W.large(precision=prec)  # every rank: the same space, its own index range
    n_cand = 24 ** 6
    device = local
    stream = torch.cuda.current_stream(device)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=f"cuda:{device}")
    def step(ctx):
        if dist:  # this rank's range, then the all-gather of the k best pairs and the counts
            return shard.search_sharded(ctx, K_TOP, chunk=CHUNK, device=torch.device("cuda", device))
        return ctx.search(K_TOP, chunk=CHUNK)

    with mf.Context(prob, device=device) as ctx:
        for _ in range(args.warmup):
            step(ctx)
        step_ms, score_ms, launches, score_launches = [], [], 0, 0
        res = None
        with ClockSampler(device) as clk:
            if dist:
                dist.barrier()
            torch.cuda.synchronize(device)
            for _ in range(args.steps):
                flush.fill_(1.0)  # L2 flush outside the timed events
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                res = step(ctx)
                e1.record(stream)
                e1.synchronize()
                step_ms.append(e0.elapsed_time(e1))
                st = ctx.stats()
                score_ms.append(st["score_ms_last"])
                launches += st["kernel_launches_last"]
                score_launches += st["score_launches_last"]
            ctx_path = int(st["scoring_path"])
            torch.cuda.synchronize(device)
            if dist:
                dist.barrier()
        total_ms = float(sum(step_ms))
        if dist:
            t = torch.tensor([total_ms], device=f"cuda:{device}")
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            total_ms = float(t.item())
        value = n_cand * args.steps / (total_ms / 1e3)  # the whole space per step, over all ranks
        feasible_frac = res["count"] / n_cand

        # roofline of the scoring kernel: algorithmic FLOPs per launch / mean launch time
        fpc = flops_per_candidate(prob)
        per_launch_ms = float(sum(score_ms)) / max(score_launches, 1)
        lo, hi = shard.shard_range(n_cand, rank, world)
        per_launch_flops = fpc * (hi - lo) / (score_launches / args.steps)
        peaks, src = _peaks()
        achieved = per_launch_flops / (per_launch_ms / 1e3) / 1e12
        sgemm = fp32_peak(torch, device) if (rank == 0 and (prec == "fp32" or not args.no_stress)) else None
        if prec == "bf16":
            # launches of about a millisecond inside a step of tens: the burst peak applies
            peak = float(peaks["bf16_tflops"])
            roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                    "frac": achieved / peak, "frac_sustained": achieved / float(peaks["bf16_tflops_sustained"]),
                    "peak_source": f"{src} bf16 burst (sustained {peaks['bf16_tflops_sustained']})"}
        elif ctx_path == 2:  # the exact tensor-core variant
            roof = exact_roofline(achieved, sgemm)
        else:
            roof = {"bound": "fp32", "achieved": achieved, "peak": sgemm, "unit": "TFLOP/s",
                    "frac": achieved / sgemm if sgemm else None,
                    "peak_source": "measured cuBLAS fp32 GEMM (TF32 off), this run"}
        roof.update({"traffic": _traffic(prec), "kernel": "scoring kernel (one launch per 2^24 candidates)",
                     "flops_per_candidate": fpc, "launch_ms": per_launch_ms})

        # end to end through the C ABI from host buffers: create (uploads) + search + result
        e2e_ms = []
        for _ in range(max(2, min(args.steps, 5))):
            torch.cuda.synchronize(device)
            t0 = time.perf_counter()
            with mf.Context(prob, device=device) as c2:
                step(c2)
                st2 = c2.stats()
            e2e_ms.append(1e3 * (time.perf_counter() - t0))
        e2e_med = statistics.median(e2e_ms)
        if dist:
            t = torch.tensor([e2e_med], device=f"cuda:{device}")
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e2e_med = float(t.item())
        e2e = {"value": n_cand / (e2e_med / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(st2["h2d_bytes_create"]),
               "d2h_bytes_per_step": int(st2["d2h_bytes_last"]),
               "how": "mf_create from host arrays + mf_search_exhaustive + mf_destroy, host wall clock, median"}

    stress = stress_throughput(mf, torch, device) if rank == 0 and not args.no_stress else None
    tight = tight_throughput(mf, torch, device) if rank == 0 and not args.no_stress else None
    exact = exact_throughput(mf, torch, device, sgemm) if rank == 0 and not args.no_stress and prec == "bf16" \
        else None
    fixed = fixed_context_throughput(mf, torch, device) if rank == 0 and not args.no_stress else None
    ga = ga_latency(mf, torch, device, args.ga_decisions) if rank == 0 else None
    paper_ga = paper_ga_latency(mf, torch, device, args.ga_decisions) if rank == 0 else None
    base = cpu_baseline(W.large(precision="fp32")) if (rank == 0 and world == 1 and not args.no_cpu) else None
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
                "scaling": "strong", "vs_baseline": None, "dtype": "bf16" if prec == "bf16" else "f32",
                "data": "synthetic", "config": dict(workload_config(prec), parallelism=(
                    f"index-range split over {world} GPUs + all-gather of the k best" if world > 1 else "1 GPU")),
                "roofline": roof,
                "cpu_baseline": base, "e2e": e2e, "gpu_launches": launches, "clocks": clk.summary(),
                "feasible_fraction": feasible_frac, "best": {"idx": res["best_idx"], "J": res["best_score"],
                                                             "count": res["count"]},
                "ga": ga, "paper_ga": paper_ga, "stress": stress, "fixed_context": fixed,
                "tight": tight, "exact_fp32": exact,
                "peaks": {"fp32_sgemm_tflops": sgemm, "fp32_sgemm_how": "cuBLAS fp32 GEMM 8192^3, TF32 off, "
                          "best of 5 (the fp32 CUDA-core roofline)"} if sgemm else None}
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--precision", default=os.environ.get("MF_BENCH_PRECISION", "bf16"),
                    choices=["bf16", "fp32"])
    ap.add_argument("--ga-decisions", type=int, default=10)
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU-baseline leg")
    ap.add_argument("--no-stress", action="store_true", help="skip the stress-workload line")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
