"""Small, self-contained cases for profiling the library's kernels (e.g. under ncu).

    python -m paper_2607_03011_gb300.profile_cases step --workload square12 --steps 2
    python -m paper_2607_03011_gb300.profile_cases gemm --batch 48 --m 1024 --n 1024 --k 1024

`step` runs IsoLoCo outer steps through the C ABI on a named workload; `square48`
is the 48 square 1024 x 1024 matrices of the 180M recipe with K = 8 replicas
(1.6 GB of replicas: larger than L2, small enough for a full ncu capture), and
`square12` a quarter of it; with --per-launch the polar iterations are launched one
by one (phase profiling on) instead of as the library's CUDA graph, so that every
kernel is a plain launch.  `gemm` runs the split-precision GEMM entry point on random
inputs; `diloco` runs DiLoCo outer steps with a merging aggregator (Sec. 3.2), and
`step --spectrum 1|2` the clip variants of Sec. 4.5.
"""
from __future__ import annotations

import argparse

import torch

from . import isoloco
from . import workloads as W

EXTRA = {
    "square48": lambda: W.custom_spec([(f"w{i}", 1024, 1024) for i in range(48)], K=8, rank=32,
                                      shared_std=2e-5, noise_std=2e-5, momentum_std=2e-5, name="square48"),
    "square12": lambda: W.custom_spec([(f"w{i}", 1024, 1024) for i in range(12)], K=8, rank=32,
                                      shared_std=2e-5, noise_std=2e-5, momentum_std=2e-5, name="square12"),
    "tall4": lambda: W.custom_spec([("e", 32000, 1024), ("d0", 2816, 1024), ("d1", 2816, 1024), ("g", 1024, 2816)],
                                   K=8, rank=32, shared_std=2e-5, noise_std=2e-5, momentum_std=2e-5, name="tall4"),
}


def run_step(workload: str, steps: int, per_launch: bool = False, spectrum_kind: int = 0) -> None:
    spec = EXTRA[workload]() if workload in EXTRA else W.SPECS[workload]
    wl = W.make_workload(spec, seed=0, device="cuda")
    plan = isoloco.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    if per_launch:
        plan.profile(True)
    opts = isoloco.make_opts(spec.alpha, spec.outer_lr, spec.momentum, spectrum_kind=spectrum_kind)
    th0, b0 = wl.theta.clone(), wl.momentum.clone()
    for _ in range(steps):
        wl.theta.copy_(th0)
        wl.momentum.copy_(b0)
        plan.outer_step(wl.theta, wl.momentum, wl.replicas, opts)
    rc = plan.last_status()
    print("status", isoloco.STATUS_NAMES.get(rc, rc), "iters", sorted(set(plan.read_diag()["iters"])))
    if rc != 0:
        raise SystemExit(1)


def run_diloco(workload: str, steps: int, aggregator: int, sparsity: float) -> None:
    spec = EXTRA[workload]() if workload in EXTRA else W.SPECS[workload]
    wl = W.make_workload(spec, seed=0, device="cuda")
    plan = isoloco.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    opts = isoloco.make_opts(outer_lr=spec.outer_lr, momentum=spec.momentum, aggregator=aggregator,
                             sparsity=sparsity, seed=1)
    th0, b0 = wl.theta.clone(), wl.momentum.clone()
    for _ in range(steps):
        wl.theta.copy_(th0)
        wl.momentum.copy_(b0)
        plan.diloco_outer_step(wl.theta, wl.momentum, wl.replicas, opts)
    rc = plan.last_status()
    print("status", isoloco.STATUS_NAMES.get(rc, rc))
    if rc != 0:
        raise SystemExit(1)


def run_gemm(batch, m, n, k, a_mn, b_mn, reps, precision=0) -> None:
    g = torch.Generator(device="cuda").manual_seed(0)
    A = torch.randn((batch, k, m) if a_mn else (batch, m, k), device="cuda", generator=g)
    B = torch.randn((batch, k, n) if b_mn else (batch, n, k), device="cuda", generator=g)
    for _ in range(reps):
        isoloco.debug_gemm(A, B, a_mn, b_mn, m, n, k, precision=precision)
    torch.cuda.synchronize()
    print("gemm ok")


def main():
    ap = argparse.ArgumentParser()
    sub = ap.add_subparsers(dest="cmd", required=True)
    s = sub.add_parser("step")
    s.add_argument("--workload", default="square12")
    s.add_argument("--steps", type=int, default=2)
    s.add_argument("--per-launch", action="store_true")
    s.add_argument("--spectrum", type=int, default=0, help="0 Iso-C, 1 clip_high, 2 clip_low")
    dl = sub.add_parser("diloco")
    dl.add_argument("--workload", default="llama_180m_k8")
    dl.add_argument("--steps", type=int, default=2)
    dl.add_argument("--aggregator", type=int, default=1, help="0 mean, 1 TIES, 2 DARE")
    dl.add_argument("--sparsity", type=float, default=0.1)
    gm = sub.add_parser("gemm")
    gm.add_argument("--batch", type=int, default=48)
    gm.add_argument("--m", type=int, default=1024)
    gm.add_argument("--n", type=int, default=1024)
    gm.add_argument("--k", type=int, default=1024)
    gm.add_argument("--a-mn", type=int, default=0)
    gm.add_argument("--b-mn", type=int, default=0)
    gm.add_argument("--reps", type=int, default=2)
    gm.add_argument("--precision", type=int, default=0)
    a = ap.parse_args()
    if a.cmd == "step":
        run_step(a.workload, a.steps, a.per_launch, a.spectrum)
    elif a.cmd == "diloco":
        run_diloco(a.workload, a.steps, a.aggregator, a.sparsity)
    else:
        run_gemm(a.batch, a.m, a.n, a.k, a.a_mn, a.b_mn, a.reps, a.precision)


if __name__ == "__main__":
    main()
