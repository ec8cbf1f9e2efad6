"""Small, self-contained cases for profiling the library's kernels (e.g. under ncu).

    python -m paper_2607_03011_gb300.profile_cases step --workload square12 --steps 2
    python -m paper_2607_03011_gb300.profile_cases gemm --batch 48 --m 1024 --n 1024 --k 1024

`step` runs IsoLoCo outer steps through the C ABI on a named workload; `square48`
is the 48 square 1024 x 1024 matrices of the 180M recipe with K = 8 replicas
(1.6 GB of replicas: larger than L2, small enough for a full ncu capture), and
`square12` a quarter of it; `wide12` / `tall12` twelve 1024 x 2816 matrices (the shape of
w_gate and w_up) and twelve 2816 x 1024 ones (w_down); `wide24` the 24 w_gate / w_up matrices
and `embed2` the 32000 x 1024 embedding and head (with `square48` and `tall12`, the 180M
recipe's four shape buckets one at a time); with --per-launch the polar iterations are launched one
by one (phase profiling on) instead of as the library's CUDA graph, so that every
kernel is a plain launch.  `gemm` runs the split-precision GEMM entry point on random
inputs; `diloco` runs DiLoCo outer steps with a merging aggregator (Sec. 3.2), and
`step --spectrum 1|2` the clip variants of Sec. 4.5; `hostlink` measures the host link
(copy engines, and the host-buffer step's reduce reading pinned memory in place).
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
    "wide12": lambda: W.custom_spec([(f"d{i}", 1024, 2816) for i in range(12)], K=8, rank=32, shared_std=2e-5,
                                    noise_std=2e-5, momentum_std=2e-5, name="wide12"),
    "tall12": lambda: W.custom_spec([(f"g{i}", 2816, 1024) for i in range(12)], K=8, rank=32, shared_std=2e-5,
                                    noise_std=2e-5, momentum_std=2e-5, name="tall12"),
    "wide24": lambda: W.custom_spec([(f"u{i}", 1024, 2816) for i in range(24)], K=8, rank=32, shared_std=2e-5,
                                    noise_std=2e-5, momentum_std=2e-5, name="wide24"),
    "embed2": lambda: W.custom_spec([("embed", 32000, 1024), ("head", 32000, 1024)], K=8, rank=32, shared_std=2e-5,
                                    noise_std=2e-5, momentum_std=2e-5, name="embed2"),
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


def run_hostlink(gib: int, workload: str) -> None:
    """The host link: copy-engine transfers of a pinned buffer (one and four streams), and
    the library's reduce pass reading pinned replicas and theta in place
    (isoloco_outer_step_host, reduce phase timed by events)."""
    n = gib << 28  # floats
    h = torch.ones(n, dtype=torch.float32).pin_memory()
    d = torch.empty(n, dtype=torch.float32, device="cuda")
    streams = [torch.cuda.Stream() for _ in range(4)]

    def timed(fn, stream):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record(stream)
        fn()
        torch.cuda.synchronize()
        b.record(stream)
        b.synchronize()
        return a.elapsed_time(b)

    nbytes = n * 4
    for _ in range(2):
        with torch.cuda.stream(streams[0]):
            ms = timed(lambda: d.copy_(h, non_blocking=True), streams[0])
        print(f"H2D one stream: {nbytes / ms / 1e6:.1f} GB/s")
        with torch.cuda.stream(streams[0]):
            ms = timed(lambda: h.copy_(d, non_blocking=True), streams[0])
        print(f"D2H one stream: {nbytes / ms / 1e6:.1f} GB/s")

        def four():
            q = n // 4
            for i, s_ in enumerate(streams):
                with torch.cuda.stream(s_):
                    d[i * q:(i + 1) * q].copy_(h[i * q:(i + 1) * q], non_blocking=True)
        ms = timed(four, torch.cuda.current_stream())
        print(f"H2D four streams: {nbytes / ms / 1e6:.1f} GB/s")
    del h, d
    spec = EXTRA[workload]() if workload in EXTRA else W.SPECS[workload]
    wl = W.make_workload(spec, seed=0, device="cuda")
    plan = isoloco.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    th_h, b_h = wl.theta.cpu().pin_memory(), wl.momentum.cpu().pin_memory()
    reps_h = [wl.replicas[k].cpu().pin_memory() for k in range(wl.K)]
    opts = isoloco.make_opts(spec.alpha, spec.outer_lr, spec.momentum)
    plan.outer_step_host(th_h.clone().pin_memory(), b_h.clone().pin_memory(), reps_h, opts)
    plan.profile(True)
    for _ in range(2):
        plan.outer_step_host(th_h.clone().pin_memory(), b_h.clone().pin_memory(), reps_h, opts)
    ms = plan.profile_read()["reduce"][0] / 2
    rb = wl.N * (wl.K * wl.replicas.element_size() + 4)
    print(f"reduce pass reading pinned replicas and theta in place: {rb / 1e9:.2f} GB in {ms:.3f} ms = "
          f"{rb / ms / 1e6:.1f} GB/s")


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
    hl = sub.add_parser("hostlink")
    hl.add_argument("--gib", type=int, default=4)
    hl.add_argument("--workload", default="square12")
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
    elif a.cmd == "hostlink":
        run_hostlink(a.gib, a.workload)
    else:
        run_gemm(a.batch, a.m, a.n, a.k, a.a_mn, a.b_mn, a.reps, a.precision)


if __name__ == "__main__":
    main()
