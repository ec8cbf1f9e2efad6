#!/usr/bin/env python
"""Benchmark of the IsoLoCo outer step (Alg. 2) on GB300.

Default workload: the ~180M LLaMA-style shape set with K = 8 fp32 worker
replicas resident in HBM (219,701,248 parameters, 86 matrices), synthetic
seeded inputs.  One step = one full outer step through the C ABI: K-way
pseudo-gradient reduction, Iso-C on every matrix (batched polar iteration on
tcgen05 tensor cores, sigma_bar by trace), Nesterov update of theta and B.

Prints ONE JSON line (rank 0).  Under torchrun every rank runs its own replica
of the workload on its own GPU (the outer step has no cross-GPU exchange when
all workers share one GPU): weak scaling, value = all ranks' parameters / time.

--impl reference times the fp64 CPU oracle on the host cores instead, on a
bounded sample of the same workload (the reference arm of this benchmark).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "IsoLoCo outer-step ms & params/s at ~180M shapes, K=8; % HBM / TC roofline"
UNIT = "params/s"


def cpu_model() -> str:
    """The host CPU's model string (x86 `model name`, or the Arm implementer / part ids)."""
    try:
        with open("/proc/cpuinfo") as f:
            info = f.read()
    except OSError:
        return "unknown"
    for line in info.splitlines():
        if line.lower().startswith("model name"):
            return line.split(":", 1)[1].strip()
    impl = part = None
    for line in info.splitlines():
        if line.startswith("CPU implementer") and impl is None:
            impl = line.split(":", 1)[1].strip()
        if line.startswith("CPU part") and part is None:
            part = line.split(":", 1)[1].strip()
    return f"arm implementer {impl} part {part}" if impl else "unknown"


def iters_by_shape(table, iters):
    """Polar iteration counts per matrix shape: {"rows x cols": {count: matrices}}."""
    out = {}
    mats = [(r, c) for (_, r, c) in table if c > 0]
    for (r, c), it in zip(mats, iters):
        d = out.setdefault(f"{r}x{c}", {})
        d[str(it)] = d.get(str(it), 0) + 1
    return out


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
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
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- multi-rank timing
def max_over_ranks(total_ms: float, dist, device) -> float:
    """The slowest rank's timed total (ms); the local value without a process group."""
    if dist is None:
        return total_ms
    import torch
    t = torch.tensor([total_ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world: int, params: int, steps: int, total_ms: float) -> float:
    """Whole-job throughput: every rank's parameters, every step, over the slowest rank's time."""
    return world * params * steps / (total_ms / 1000.0)


# --------------------------------------------------------------------------- accounting
GRAM_SIDE_RATIO = 8   # tall matrices with rows >= 8 * cols iterate on n x n matrices (the library's rule)


def gram_side(r, c, fast=False, full=False):
    """Whether the library runs this matrix's polar iteration on the Gram side."""
    return r >= GRAM_SIDE_RATIO * c and r >= 2 * BK and not fast and not full


def gemm_flops(table, diag, fast=False, full=False):
    """Algorithmic (single-pass) FLOPs of the polar GEMMs of one step, per phase, from
    the per-matrix iteration counts: a full Gram 2*r*n^2 per iteration (symmetry not
    discounted), G^2 = 2*n^3 per quintic step, an update 2*r*n^2 per iteration
    (r = long side, n = short side of the matrix).  The fast variant runs `it` quintic
    steps and no polish."""
    out = {"gram": 0.0, "poly": 0.0, "update": 0.0}
    mats = [(r, c) for (_, r, c) in table if c > 0]
    for (r, c), it, st in zip(mats, diag["iters"], diag["status"]):
        big, small = max(r, c), min(r, c)
        gram1, sq1 = 2.0 * big * small * small, 2.0 * small ** 3
        if it > 0 and gram_side(r, c, fast, full):
            # iteration 0's Gram (2 m n^2) and P_0; then per iteration W = A Z and G = Z^T W
            # (2 n^3 each), P (quintic steps) and Z P (2 n^3); finally Q = Delta Z (2 m n^2)
            converged = (st == 0)
            grams = it + (0 if converged else 1)
            quintic = it - (1 if converged else 0)
            out["gram"] += gram1 + (grams - 1) * 2 * sq1
            out["poly"] += quintic * sq1
            out["update"] += (it - 1) * sq1 + gram1
            continue
        if fast:
            out["gram"] += it * gram1
            out["poly"] += it * sq1
            out["update"] += it * gram1
            continue
        if it == 0:
            out["gram"] += gram1  # one Gram, then found zero
            continue
        converged = (st == 0)
        out["gram"] += (it + (0 if converged else 1)) * gram1
        out["poly"] += (it - (1 if converged else 0)) * sq1
        out["update"] += it * gram1
    return out


BM, BN, BK = 256, 256, 64   # output tile of one CTA pair (tcgen05 cta_group::2), stage depth


def _sym_tiles(n):
    tm_n, tn_n = -(-n // BM), -(-n // BN)
    c = 0
    for tm in range(tm_n):
        x = tm * BM - BN + 1
        c += tn_n - (0 if x <= 0 else -(-x // BN))
    return c


# The library's default precision schedule (the quintic steps whose GEMMs run one pass),
# as the library defines it: per schedule kind, [from, to) for the Gram and polynomial and
# for the update.  Standard schedule: rectangular matrices; deep: near-square ones.
DEFAULT_SCHEDULE = {"std": {"gp": (1, 6), "upd": (2, 6)}, "deep": {"gp": (9, 11), "upd": (10, 11)}}
NO_DEMOTION = {"std": {"gp": (0, 0), "upd": (0, 0)}, "deep": {"gp": (0, 0), "upd": (0, 0)}}


def gemm_exec_flops(table, diag, fast=False, full=False, sched=None):
    """Tensor-core FLOPs the GEMM launches execute per phase: 2*BM*BN*K_padded per
    computed tile and per 16-bit pass, symmetric Grams/G^2 on their upper-triangle tiles
    only.  Passes: 3 at iteration 0 and in the polish update; elsewhere 2, or 1 for the
    steps the precision schedule `sched` (default: the library's) runs single-pass; 3
    everywhere with `full` (full precision, the clip variants) and in the fast variant.
    A Gram in the single-pass range runs one pass only while the matrix's previous residual
    is large (the library's rule); this count takes every such Gram as single-pass, a lower
    bound on the executed FLOPs."""
    sched = DEFAULT_SCHEDULE if sched is None else sched
    out = {"gram": 0.0, "poly": 0.0, "update": 0.0}
    mats = [(r, c) for (_, r, c) in table if c > 0]
    for (r, c), it, st in zip(mats, diag["iters"], diag["status"]):
        big, n = max(r, c), min(r, c)
        kpad_big, kpad_n = -(-big // BK) * BK, -(-n // BK) * BK
        gram1 = _sym_tiles(n) * BM * BN * 2.0 * kpad_big
        poly1 = _sym_tiles(n) * BM * BN * 2.0 * kpad_n
        upd1 = (-(-r // BM)) * (-(-c // BN)) * BM * BN * 2.0 * kpad_n
        if it > 0 and gram_side(r, c, fast, full):
            sq_all = (-(-n // BM)) * (-(-n // BN)) * BM * BN * 2.0 * kpad_n   # every tile of an n x n product
            converged = (st == 0)
            grams = it + (0 if converged else 1)
            quintic = it - (1 if converged else 0)
            # iteration 0: Gram and P_0 three passes; later W and G three passes, P two,
            # Z P two (three in the polish); the final Delta Z three
            out["gram"] += 3 * gram1 + (grams - 1) * 3 * (sq_all + poly1)
            out["poly"] += (3 * poly1 + 2 * poly1 * (quintic - 1)) if quintic >= 1 else 0.0
            out["update"] += 2 * sq_all * max(0, quintic - 1) + (3 * sq_all if converged and it > 1 else 0.0) + 3 * upd1
            continue
        if fast:   # `it` quintic steps, every one with three passes; no polish
            out["gram"] += 3 * gram1 * it
            out["poly"] += 3 * poly1 * it
            out["update"] += 3 * upd1 * it
            continue
        if it == 0:
            out["gram"] += 3 * gram1
            continue
        kind = sched["deep" if abs(r - c) * 16 < n else "std"]
        converged = (st == 0)
        quintic = it - (1 if converged else 0)   # steps 0 .. quintic - 1, then the polish

        def passes(k, rng):
            if k == 0 or full:
                return 3
            return 1 if rng[0] <= k < rng[1] else 2
        # the Gram of iteration t leads to step t (t quintic steps taken before it)
        for t in range(it + (0 if converged else 1)):
            out["gram"] += passes(t, kind["gp"]) * gram1
        for k in range(quintic):
            out["poly"] += passes(k, kind["gp"]) * poly1
            out["update"] += passes(k, kind["upd"]) * upd1
        if converged:
            out["update"] += 3 * upd1          # the polish
    return out


def stream_bytes(table, K, replica_bytes):
    n = sum(r * (c or 1) for (_, r, c) in table)
    n2 = sum(r * c for (_, r, c) in table if c > 0)
    return {
        "reduce": (K * replica_bytes + 4) * n + 4 * n,   # replicas + theta in; Delta (hi/lo or fp32) out
        "apply": 8 * n + 4 * n + 8 * n,                   # theta, B, U-source in; theta, B out
        "trace": 8 * n2,                                  # Q and Delta hi/lo
        "algorithmic_step": (K * replica_bytes + 16) * n + 8 * n2,
    }


# Arithmetic of the IsoLoCo step: fp32 streaming (reduction, Nesterov), polar GEMMs on 16-bit
# tensor-core passes over hi/lo splits of fp32 operands with fp32 accumulation.
DTYPE_ISO = "f32 streaming; polar GEMMs as bf16/fp16 hi+lo split passes, f32 accumulate"

# DRAM bytes (read + write) of all k_gemm_split launches of one step, from ncu captures of
# the current kernel, (workload, fast_steps, spectrum_kind) -> figure: the 180M step's four
# shape buckets captured one at a time with ncu (dram__bytes_read.sum + dram__bytes_write.sum) and summed.
GEMM_TRAFFIC = {
    ("llama_180m_k8", 0, 0): {
        "bytes_per_step": 24.45e9,
        "note": "dram__bytes_read.sum + dram__bytes_write.sum of every k_gemm_split launch of one step, "
                "captured per shape bucket (square48, tall12, wide24, embed2) and summed; same unit as "
                "achieved (per step over all GEMM launches)"},
}


# --------------------------------------------------------------------------- CPU oracle arm
CPU_SAMPLE = ["layers.0.attn_norm", "layers.0.wq", "layers.0.wk", "layers.0.ffn_norm", "layers.0.w_gate", "layers.0.w_up",
              "layers.0.w_down"]
REF_SAMPLE = ["layers.0.attn_norm", "layers.0.wq", "layers.0.ffn_norm"]


def oracle_sample_run(workload: str, names, seed: int = 0):
    """Runs the oracle's outer step on a sample of the workload's tensors, with the
    workload's generator recipe (CPU generator).  Returns (params, seconds)."""
    import oracle
    from paper_2607_03011_gb300 import workloads as W
    base = W.SPECS[workload]
    shapes = [s for s in base.shapes if s[0] in names]
    spec = W.custom_spec(shapes, K=base.K, rank=base.rank, shared_std=base.shared_std,
                         noise_std=base.noise_std, momentum_std=base.momentum_std,
                         replica_dtype=base.replica_dtype, name=base.name + "_sample")
    wl = W.make_workload(spec, seed=seed, device="cpu")
    reps = W.replicas_as_numpy(wl.replicas)
    th, b = wl.theta.numpy(), wl.momentum.numpy()
    t0 = time.perf_counter()
    oracle.isoloco_outer_step(wl.table, th, b, reps, alpha=base.alpha, eta=base.outer_lr, mu=base.momentum)
    dt = time.perf_counter() - t0
    return wl.N, dt, "+".join(f"{n}:{r}x{c}" if c else f"{n}:{r}" for (n, r, c) in shapes)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    cores = oracle.num_threads()
    times, nparams, desc = [], 0, ""
    for i in range(args.warmup + args.steps):
        nparams, dt, desc = oracle_sample_run(args.workload, REF_SAMPLE, seed=i)
        if i >= args.warmup:
            times.append(dt)
    ms = 1000.0 * sum(times) / len(times)
    value = nparams / (ms / 1000.0)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.workload, "sample": desc, "sample_params": nparams},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "cpu_model": cpu_model(),
                             "sample": f"oracle outer step on {desc} ({nparams} params) per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# --------------------------------------------------------------------------- DiLoCo arm
AGG_CODE = {"mean": 0, "ties": 1, "dare": 2}
AGG_KERNELS = {"mean": "k_diloco", "ties": "k_ties_bracket (one pass) + k_ties_merge", "dare": "k_dare"}


def diloco_bytes(agg, N, K, eb):
    """Algorithmic HBM bytes of one DiLoCo step per phase: the streaming pass reads theta,
    B and the K replicas and writes theta and B; TIES's trim reads theta and the replicas
    once (the bracket pass; the sample and the candidate selection are small)."""
    out = {"diloco": (16 + K * eb) * N}
    if agg == "ties":
        out["trim"] = (4 + K * eb) * N
    return out


def oracle_merging_sample(workload: str, names, agg: str, sparsity: float, seed: int = 0):
    """The oracle's DiLoCo step with a merging rule on a sample of the workload's tensors
    (TIES trims within the sample).  Returns (params, seconds, description)."""
    import oracle
    from oracle import merging
    from paper_2607_03011_gb300 import workloads as W
    base = W.SPECS[workload]
    shapes = [s for s in base.shapes if s[0] in names]
    spec = W.custom_spec(shapes, K=base.K, rank=base.rank, shared_std=base.shared_std,
                         noise_std=base.noise_std, momentum_std=base.momentum_std,
                         replica_dtype=base.replica_dtype, name=base.name + "_sample")
    wl = W.make_workload(spec, seed=seed, device="cpu")
    reps = W.replicas_as_numpy(wl.replicas)
    th, b = wl.theta.numpy(), wl.momentum.numpy()
    t0 = time.perf_counter()
    if agg == "mean":
        oracle.diloco_outer_step(th, b, reps, eta=base.outer_lr, mu=base.momentum)
    else:
        merging.merged_outer_step(th, b, reps, agg, sparsity=sparsity, seed=1, eta=base.outer_lr,
                                  mu=base.momentum)
    dt = time.perf_counter() - t0
    return wl.N, dt, "+".join(f"{n}:{r}x{c}" if c else f"{n}:{r}" for (n, r, c) in shapes)


def run_diloco(args, torch, isoloco, wl, plan, world, rank, local, dist, barrier):
    """Times diloco_outer_step (Alg. 1) with the chosen merging rule on the workload."""
    spec = wl.spec
    agg = args.aggregator
    opts = isoloco.make_opts(outer_lr=spec.outer_lr, momentum=spec.momentum, aggregator=AGG_CODE[agg],
                             sparsity=args.sparsity if agg != "mean" else 0.0, seed=1)
    theta0, mom0 = wl.theta.clone(), wl.momentum.clone()
    th, b = wl.theta, wl.momentum
    stream = torch.cuda.current_stream()

    def restore():
        th.copy_(theta0)
        b.copy_(mom0)

    for _ in range(args.warmup):
        restore()
        plan.diloco_outer_step(th, b, wl.replicas, opts)
    if plan.last_status() != 0:
        raise RuntimeError(f"warm-up step status {isoloco.STATUS_NAMES.get(plan.last_status())}")
    launches0 = plan.launches
    clocks = ClockSampler(local)
    torch.cuda.synchronize()
    barrier()
    clocks.start()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for i in range(args.steps):
        restore()
        ev[i][0].record(stream)
        plan.diloco_outer_step(th, b, wl.replicas, opts)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    status = plan.last_status()
    step_ms = [a.elapsed_time(z) for a, z in ev]
    total_ms = sum(step_ms)
    launches = plan.launches - launches0
    plan.profile(True)
    for i in range(args.steps):
        restore()
        plan.diloco_outer_step(th, b, wl.replicas, opts)
    torch.cuda.synchronize()
    prof = plan.profile_read()
    plan.profile(False)
    total_ms = max_over_ranks(total_ms, dist, "cuda")
    ms_per_step = total_ms / args.steps
    value = job_value(world, wl.N, args.steps, total_ms)

    # end to end: pinned host buffers copied in and out on the stream around the call
    e2e = None
    if not args.no_e2e and rank == 0:
        th_h, b_h = theta0.cpu().pin_memory(), mom0.cpu().pin_memory()
        reps_h = wl.replicas.cpu().pin_memory()
        th_d, b_d = torch.empty_like(th), torch.empty_like(b)
        reps_d = torch.empty_like(wl.replicas)
        e_ms = []
        for _ in range(1 + args.e2e_steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            th_d.copy_(th_h, non_blocking=True)
            b_d.copy_(b_h, non_blocking=True)
            reps_d.copy_(reps_h, non_blocking=True)
            plan.diloco_outer_step(th_d, b_d, reps_d, opts)
            th_h.copy_(th_d, non_blocking=True)
            b_h.copy_(b_d, non_blocking=True)
            e1.record(stream)
            e1.synchronize()
            e_ms.append(e0.elapsed_time(e1))
            th_h.copy_(theta0.cpu())
            b_h.copy_(mom0.cpu())
        e_ms = e_ms[1:]
        eb = wl.replicas.element_size()
        e2e = {"value": wl.N / (statistics.median(e_ms) / 1000.0), "unit": UNIT,
               "h2d_bytes_per_step": int(wl.N * (8 + wl.K * eb)), "d2h_bytes_per_step": int(wl.N * 8),
               "ms_per_step": statistics.median(e_ms),
               "api": "diloco_outer_step on device copies of pinned host buffers (copies on the same stream)"}
        del reps_h, reps_d

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0
    peaks, peak_src = load_peaks()
    hbm = peaks["hbm_gbs"]
    eb = wl.replicas.element_size()
    nb = diloco_bytes(agg, wl.N, wl.K, eb)
    phases = {}
    for ph, nbytes in nb.items():
        ms, n = prof[ph]
        gb = nbytes * args.steps / (ms / 1000.0) / 1e9 if ms > 0 else 0.0
        phases[ph] = {"achieved": gb, "frac": gb / hbm, "bytes_per_step": nbytes, "ms_per_step": ms / args.steps,
                      "launches_per_step": n / args.steps}
    dom = max(phases, key=lambda k: phases[k]["ms_per_step"])
    roofline = {"bound": "hbm", "kernel": {"diloco": "k_diloco" if agg == "mean" else
                                           ("k_ties_merge" if agg == "ties" else "k_dare"),
                                           "trim": "k_ties_bracket (+ sample and candidate selection)"}[dom],
                "achieved": phases[dom]["achieved"], "peak": hbm, "unit": "GB/s", "frac": phases[dom]["frac"],
                "traffic": None, "peak_source": f"{peak_src} hbm_gbs",
                "kernel_times": "per-phase CUDA events on the launch stream, in a profiled pass of the same "
                                "steps right after the timed region",
                "phases": phases}
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        import oracle
        oracle.build()
        nparams, dt, desc = oracle_merging_sample(args.workload, CPU_SAMPLE, agg, args.sparsity)
        cpu = {"value": nparams / dt, "unit": UNIT, "cores": 1, "kind": "oracle", "cpu_model": cpu_model(),
               "sample": f"oracle DiLoCo step ({agg}) on {desc} ({nparams} params, {dt:.1f} s), "
                         "same generator recipe"}
    line = {
        "metric": f"DiLoCo outer-step ({agg} aggregation) params/s at {args.workload}", "value": value,
        "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": args.workload, "params": wl.N, "K": wl.K, "aggregator": agg,
                   "sparsity": args.sparsity if agg != "mean" else 0.0,
                   "replica_dtype": str(wl.replicas.dtype).replace("torch.", ""),
                   "outer_lr": spec.outer_lr, "momentum": spec.momentum,
                   "l2": "inputs larger than L2 (K replicas = %.1f GB)" % (wl.replicas.numel() * eb / 1e9),
                   "timing": "sum of per-step CUDA-event intervals on the launch stream; theta/B restored "
                             "between steps outside the intervals",
                   "parallelism": f"replicas x{world}"},
        "status": isoloco.STATUS_NAMES.get(status, status),
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": int(launches),
        "clocks": clk, "step_ms": [round(x, 3) for x in step_ms],
    }
    print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


# --------------------------------------------------------------------------- GPU arm
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama_180m_k8")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--fast-steps", type=int, default=0,
                    help="time the fast variant of Sec. 4.3 (k fixed polar steps, rms sigma_bar); 0 = exact")
    ap.add_argument("--aggregator", default="iso_c", choices=["iso_c", "mean", "ties", "dare"],
                    help="iso_c: the IsoLoCo step (Alg. 2, default); mean / ties / dare: the DiLoCo step "
                         "(Alg. 1) with that merging rule (Sec. 3.2)")
    ap.add_argument("--sparsity", type=float, default=0.1, help="TIES / DARE sparsity (0.1: Sec. 5.1's best)")
    ap.add_argument("--spectrum", default="iso_c", choices=["iso_c", "clip_high", "clip_low", "svd"],
                    help="the IsoLoCo step's spectrum map (Sec. 4.5): every singular value to the mean (Iso-C), "
                         "or only those above (clip_high) / below (clip_low) it; svd: Iso-C with every singular "
                         "value computed (Alg. 2's SVD form)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    if args.impl == "reference":
        return run_reference(args)

    import torch

    from paper_2607_03011_gb300 import isoloco
    from paper_2607_03011_gb300 import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if dist is not None:
            dist.barrier()

    spec = W.SPECS[args.workload]
    wl = W.make_workload(spec, seed=rank, device="cuda")
    plan = isoloco.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    if args.aggregator != "iso_c":
        return run_diloco(args, torch, isoloco, wl, plan, world, rank, local, dist, barrier)
    spectrum_kind = {"iso_c": 0, "clip_high": 1, "clip_low": 2, "svd": 3}[args.spectrum]
    opts = isoloco.make_opts(spec.alpha, spec.outer_lr, spec.momentum, fast_steps=args.fast_steps,
                             spectrum_kind=spectrum_kind)
    theta0, mom0 = wl.theta.clone(), wl.momentum.clone()
    th, b = wl.theta, wl.momentum
    stream = torch.cuda.current_stream()

    def restore():
        th.copy_(theta0)
        b.copy_(mom0)

    for _ in range(args.warmup):
        restore()
        rc = plan.outer_step(th, b, wl.replicas, opts)
    if plan.last_status() not in (0,):
        raise RuntimeError(f"warm-up step status {isoloco.STATUS_NAMES.get(plan.last_status())}")

    # ---- timed region: K outer steps, each bracketed by CUDA events on the stream.
    launches0 = plan.launches
    clocks = ClockSampler(local)
    torch.cuda.synchronize()
    barrier()
    clocks.start()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for i in range(args.steps):
        restore()                       # outside the event pair: theta/B back to the step's inputs
        ev[i][0].record(stream)
        plan.outer_step(th, b, wl.replicas, opts)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    status = plan.last_status()
    step_ms = [a.elapsed_time(z) for a, z in ev]
    total_ms = sum(step_ms)
    launches = plan.launches - launches0
    diag = plan.read_diag()

    # ---- kernel times: the same K steps again with per-phase CUDA events (the library then
    # launches the polar iterations one by one, stopping once every matrix is done, since
    # events cannot sit inside its graph); the timed numbers above are without them
    plan.profile(True)
    for i in range(args.steps):
        restore()
        plan.outer_step(th, b, wl.replicas, opts)
    torch.cuda.synchronize()
    prof = plan.profile_read()
    plan.profile(False)
    total_ms = max_over_ranks(total_ms, dist, "cuda")
    ms_per_step = total_ms / args.steps
    value = job_value(world, wl.N, args.steps, total_ms)

    # ---- end-to-end through the host-buffer entry point (pinned host memory)
    e2e = None
    if not args.no_e2e and rank == 0:
        th_h = theta0.cpu().pin_memory()
        b_h = mom0.cpu().pin_memory()
        th0_h, b0_h = th_h.clone(), b_h.clone()
        reps_h = [wl.replicas[k].cpu().pin_memory() for k in range(wl.K)]
        plan.outer_step_host(th_h, b_h, reps_h, opts)    # first call allocates the staging buffers
        e_ms = []
        for _ in range(args.e2e_steps):
            th_h.copy_(th0_h)
            b_h.copy_(b0_h)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            rc = plan.outer_step_host(th_h, b_h, reps_h, opts)
            e1.record(stream)
            e1.synchronize()
            e_ms.append(e0.elapsed_time(e1))
        rep_bytes = wl.replicas.element_size()
        e2e = {"value": wl.N / (statistics.median(e_ms) / 1000.0), "unit": UNIT,
               "h2d_bytes_per_step": int(wl.N * (4 + 4 + wl.K * rep_bytes)),
               "d2h_bytes_per_step": int(wl.N * 8), "ms_per_step": statistics.median(e_ms),
               "api": "isoloco_outer_step_host",
               "link_h2d_bytes_per_step": int(wl.N * (4 + 4 + 4 + wl.K * rep_bytes)),
               "note": "pinned inputs: the reduce reads the replicas and theta in place over the host link, "
                       "theta and B are copied during the polar iteration (theta crosses the link twice)"}
        del reps_h

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0

    peaks, peak_src = load_peaks()
    fl = gemm_flops(wl.table, diag, fast=args.fast_steps > 0, full=spectrum_kind != 0)
    fl_rc = gemm_flops(wl.table, diag, fast=True if args.fast_steps > 0 else False, full=True)
    fx = gemm_exec_flops(wl.table, diag, fast=args.fast_steps > 0, full=spectrum_kind != 0)
    flops = sum(fl.values()) * args.steps
    xflops = sum(fx.values()) * args.steps
    gemm_ms = prof["gram"][0] + prof["poly"][0] + prof["update"][0]
    gemm_launches = prof["gram"][1] + prof["poly"][1] + prof["update"][1]
    tc_peak = peaks["bf16_tflops_sustained"]   # bf16 and fp16 share the dense tensor rate
    # the method's own FLOPs (4 m n^2 + 2 n^3 per quintic step, 4 m n^2 per polish) per second;
    # the split-precision passes the kernel executes are reported beside it
    achieved_tf = flops / (gemm_ms / 1000.0) / 1e12 if gemm_ms > 0 else 0.0
    executed_tf = xflops / (gemm_ms / 1000.0) / 1e12 if gemm_ms > 0 else 0.0
    sb = stream_bytes(wl.table, wl.K, wl.replicas.element_size())
    hbm = peaks["hbm_gbs"]

    def gbs(phase, nbytes):
        ms, n = prof[phase]
        return nbytes * args.steps / (ms / 1000.0) / 1e9 if ms > 0 else 0.0

    traffic = GEMM_TRAFFIC.get((args.workload, args.fast_steps, spectrum_kind))
    roofline = {"bound": "tensor", "kernel": "k_gemm_split (Gram, G^2 and update GEMMs)",
                "achieved": achieved_tf, "peak": tc_peak, "unit": "TFLOP/s",
                "frac": achieved_tf / tc_peak if tc_peak else None,
                "traffic": traffic["bytes_per_step"] if traffic else None,
                "traffic_note": traffic["note"] if traffic else "no DRAM capture of the current kernel",
                "peak_source": f"{peak_src} bf16_tflops_sustained (of measured: dense 16-bit tensor rate; the "
                               "kernel runs inside a 10-30 ms step, repeated)",
                "frac_of_burst": achieved_tf / peaks["bf16_tflops"] if peaks.get("bf16_tflops") else None,
                "counts": "algorithmic FLOPs of the polar GEMMs per step (fp32-equivalent products, full Gram: "
                          "4mn^2 + 2n^3 per quintic step, 4mn^2 per polish) over the GEMM launches' time",
                "kernel_times": "per-phase CUDA events on the launch stream, in a profiled pass of the "
                                "same steps right after the timed region",
                "algorithmic_tflop_per_step": flops / args.steps / 1e12,
                "rows_cols_tflop_per_step": sum(fl_rc.values()) / 1e12,
                "rows_cols_note": "the same iteration counts priced as if every matrix iterated on its rows x cols "
                                  "side (4mn^2 + 2n^3 per quintic step); the Gram-side matrices (rows >= 8 cols) do "
                                  "less work, which `algorithmic_tflop_per_step` counts",
                "executed_tensor_tflop_per_step": xflops / args.steps / 1e12,
                "executed_tflops": executed_tf,
                "frac_executed": executed_tf / tc_peak if tc_peak else None,
                "executed_note": "16-bit tensor passes the kernel runs (hi/lo splits: 2-3 passes per product), "
                                 "upper-triangle tiles of symmetric outputs",
                "gemm_ms_per_step": gemm_ms / args.steps, "gemm_launches_per_step": gemm_launches / args.steps}
    roofline_hbm = {
        "reduce": {"achieved": gbs("reduce", sb["reduce"]), "peak": hbm, "unit": "GB/s",
                   "frac": gbs("reduce", sb["reduce"]) / hbm, "bytes_per_launch": sb["reduce"],
                   "ms_per_step": prof["reduce"][0] / args.steps},
        "apply": {"achieved": gbs("apply", sb["apply"]), "peak": hbm, "unit": "GB/s",
                  "frac": gbs("apply", sb["apply"]) / hbm, "bytes_per_launch": sb["apply"],
                  "ms_per_step": prof["apply"][0] / args.steps},
        "trace": {"ms_per_step": prof["trace"][0] / args.steps, "fused": True,
                  "note": "tr(Q^T Delta) is summed in the epilogue of the GEMM that writes each matrix's final "
                          "Q (the polish update; the Gram side's Q = Delta Z), which reads Delta's planes "
                          "(4 B per matrix element) there; the trace pass itself only covers matrices with no "
                          "such GEMM (not converged) and is launch cost otherwise"},
        "peak_source": f"{peak_src} hbm_gbs",
    }
    phases_ms = {k: round(v[0] / args.steps, 4) for k, v in prof.items() if v[1]}
    phases_tflops = {k: round(fl[k] / (prof[k][0] / args.steps / 1000.0) / 1e12, 1)
                     for k in fl if prof[k][0] > 0}
    phases_exec = {k: round(fx[k] / (prof[k][0] / args.steps / 1000.0) / 1e12, 1)
                   for k in fx if prof[k][0] > 0}

    cpu = None
    if not args.no_cpu_baseline and world == 1:
        import oracle
        oracle.build()
        nparams, dt, desc = oracle_sample_run(args.workload, CPU_SAMPLE)
        cpu = {"value": nparams / dt, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
               "cpu_model": cpu_model(),
               "sample": f"fp64 oracle outer step on {desc} ({nparams} params, {dt:.1f} s), "
                         "same generator recipe"}

    iters = diag["iters"]
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": DTYPE_ISO, "data": "synthetic",
        "config": {"workload": args.workload, "params": wl.N, "K": wl.K, "matrices": plan.num_matrices,
                   "replica_dtype": str(wl.replicas.dtype).replace("torch.", ""),
                   "alpha": spec.alpha, "outer_lr": spec.outer_lr, "momentum": spec.momentum,
                   "l2": "inputs larger than L2 (K replicas = %.1f GB)" % (wl.replicas.numel() *
                                                                      wl.replicas.element_size() / 1e9),
                   "timing": "sum of per-step CUDA-event intervals on the launch stream; theta/B "
                             "restored between steps outside the intervals",
                   "parallelism": f"replicas x{world}",
                   "iso_c": ("exact polar, sigma_bar = tr(Q^T Delta)/r" if not args.fast_steps else
                             f"fast variant: {args.fast_steps} fixed polar steps, sigma_bar = ||Delta||_F/sqrt(r)"),
                   "spectrum": args.spectrum},
        "status": isoloco.STATUS_NAMES.get(status, status),
        "polar_iters": {"min": min(iters), "max": max(iters), "mean": sum(iters) / len(iters),
                        "by_shape": iters_by_shape(wl.table, iters)},
        "ms_step_median": statistics.median(step_ms), "ms_step_best": min(step_ms),
        "phases_ms_per_step": phases_ms, "phases_algorithmic_tflops": phases_tflops,
        "phases_executed_tflops": phases_exec,
        "roofline": roofline, "roofline_hbm": roofline_hbm,
        "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": int(launches),
        "clocks": clk, "step_ms": [round(x, 3) for x in step_ms],
    }
    print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
