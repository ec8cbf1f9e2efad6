"""CUDA path vs the fp64 oracle on the same seeded inputs, through the C ABI.

Tolerances (the method's targets): relative Frobenius error of every Iso-C
update alpha*sigma_bar*Q <= 2e-3, sigma_bar relative error <= 1e-4, elementwise
relative error <= 1e-5 on theta and momentum of the non-matrix tensors (with a
floor at the rms of the reference for entries that cancel).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03011_gb300 import workloads as W
from parity import check_step, elementwise_rel, oracle_fast_step, oracle_step, rel_fro

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def iso():
    from paper_2607_03011_gb300 import isoloco
    isoloco.lib()
    return isoloco


def run_gpu(iso, wl, alpha, eta, mu, reps=None, theta=None, mom=None, max_iter=0, reduce_mean=True,
            plan=None, fast_steps=0, **ablation):
    plan = plan or iso.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    th = (wl.theta if theta is None else theta).clone()
    b = (wl.momentum if mom is None else mom).clone()
    upd = torch.empty_like(th)
    rc = plan.outer_step(th, b, wl.replicas if reps is None else reps,
                         iso.make_opts(alpha, eta, mu, reduce_mean=reduce_mean, max_iter=max_iter, sync=True,
                                       fast_steps=fast_steps, **ablation),
                         update_out=upd)
    diag = plan.read_diag()
    return rc, th, b, upd, diag, plan


def compare(wl, rc, th, b, upd, diag, alpha, eta, mu, theta_in=None, mom_in=None, reps=None, only=None):
    assert rc == 0
    ref = oracle_step(wl.table, wl.theta if theta_in is None else theta_in,
                      wl.momentum if mom_in is None else mom_in, wl.replicas if reps is None else reps,
                      alpha, eta, mu, only=only)
    ref["theta_in"] = (wl.theta if theta_in is None else theta_in).double().cpu().numpy()
    mats = [i for i, t in enumerate(wl.table) if t[2] > 0]
    sig = diag["sigma_bar"]
    return check_step(wl.table, th.double().cpu().numpy(), b.double().cpu().numpy(),
                      upd.double().cpu().numpy(), sig, ref, only=only), ref


def test_tiny_two_steps(iso):
    """Tiny config: one outer step, then a second one reusing the momentum."""
    wl = W.make_workload("tiny", seed=0, device="cuda")
    sp = wl.spec
    rc, th, b, upd, diag, plan = run_gpu(iso, wl, sp.alpha, sp.outer_lr, sp.momentum)
    worst, ref = compare(wl, rc, th, b, upd, diag, sp.alpha, sp.outer_lr, sp.momentum)
    assert all(s == 0 for s in diag["status"])
    # step 2: each side regenerates replicas (seed 1) from its own theta and keeps its B
    th_o = torch.from_numpy(ref["theta"].astype(np.float32)).cuda()   # the oracle's own step-1 result
    b_o = torch.from_numpy(ref["momentum"].astype(np.float32))
    reps_g = W.make_replicas(sp, wl.table, th, seed=1)
    reps_o = W.make_replicas(sp, wl.table, th_o, seed=1)
    th2, b2 = th.clone(), b.clone()
    upd2 = torch.empty_like(th2)
    rc = plan.outer_step(th2, b2, reps_g, iso.make_opts(sp.alpha, sp.outer_lr, sp.momentum, sync=True),
                         update_out=upd2)
    assert rc == 0
    ref2 = oracle.isoloco_outer_step(wl.table, th_o.cpu().numpy(), b_o.numpy(), W.replicas_as_numpy(reps_o),
                                     alpha=sp.alpha, eta=sp.outer_lr, mu=sp.momentum)
    ref2["theta_in"] = th_o.double().cpu().numpy()
    check_step(wl.table, th2.double().cpu().numpy(), b2.double().cpu().numpy(), upd2.double().cpu().numpy(),
               plan.read_diag()["sigma_bar"], ref2)


@pytest.mark.parametrize("alpha,eta,mu", [(1.0, 1.8, 0.8), (0.5, 0.7, 0.0)])
def test_tiny_hyperparameters(iso, alpha, eta, mu):
    wl = W.make_workload("tiny", seed=3, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, alpha, eta, mu)
    compare(wl, rc, th, b, upd, diag, alpha, eta, mu)


RAGGED = [("a", 65, 130), ("b", 130, 65), ("c", 1, 9), ("d", 9, 1), ("e", 200, 3), ("f", 3, 200),
          ("g", 1, 1), ("v", 7, 0), ("h", 300, 257), ("w", 5, 0), ("i", 257, 300), ("j", 129, 129)]


def test_ragged_shapes_and_tails(iso):
    spec = W.custom_spec(RAGGED, K=3, rank=2, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=11, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9)
    compare(wl, rc, th, b, upd, diag, 1.0, 0.7, 0.9)


def test_gram_side_shapes(iso):
    """Tall matrices with rows >= 8 cols iterate on the Gram side (n x n matrices Z with
    G = Z^T A Z, then Q = Delta Z): odd and small n, several matrices in one bucket, a long
    4100 x 72, a 32000 x 256, bf16 replicas, and a zero pseudo-gradient in the bucket; the
    same inputs on the rows x cols path (full_precision = 1) as a cross-check."""
    shapes = [("a", 200, 3), ("b", 256, 16), ("c", 1024, 48), ("c2", 1024, 48), ("d", 2048, 33), ("e", 4100, 72),
              ("f", 32000, 256), ("z", 1024, 48), ("v", 17, 0)]
    for dtype in ("f32", "bf16"):
        spec = W.custom_spec(shapes, K=3, rank=2, replica_dtype=dtype, momentum_std=1e-4)
        wl = W.make_workload(spec, seed=51, device="cuda")
        npad = (wl.N + 63) // 64 * 64
        reps = torch.empty((wl.K, npad), dtype=wl.replicas.dtype, device="cuda")[:, :wl.N]
        reps.copy_(wl.replicas)
        o, r, c = wl.table[7]
        # Delta = 0 in the bucket (theta there made representable in the replicas' type first)
        wl.theta[o:o + r * c] = wl.theta[o:o + r * c].to(reps.dtype).float()
        reps[:, o:o + r * c] = wl.theta[o:o + r * c].to(reps.dtype)
        for fp in (0, 1):
            rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, reps=reps, full_precision=fp)
            worst, _ = compare(wl, rc, th, b, upd, diag, 1.0, 0.7, 0.9, reps=reps)
            o, r, c = wl.table[7]
            assert torch.count_nonzero(upd[o:o + r * c]) == 0
            print("Gram-side shapes", dtype, "rows x cols path" if fp else "Gram side", worst)


def test_split_k_gram(iso):
    """Tall-skinny matrices whose Gram takes several split-K passes."""
    spec = W.custom_spec([("t", 6000, 64), ("u", 64, 5000), ("v", 100, 0)], K=2, rank=3)
    wl = W.make_workload(spec, seed=2, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9)
    compare(wl, rc, th, b, upd, diag, 1.0, 0.7, 0.9)


def test_single_worker_and_sum_reduction(iso):
    spec = W.custom_spec([("m", 96, 64), ("v", 64, 0)], K=1, rank=2)
    wl = W.make_workload(spec, seed=4, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9)
    compare(wl, rc, th, b, upd, diag, 1.0, 0.7, 0.9)
    spec = W.custom_spec([("m", 96, 64), ("v", 64, 0)], K=4, rank=2)
    wl = W.make_workload(spec, seed=4, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, reduce_mean=False)
    assert rc == 0
    ref = oracle_step(wl.table, wl.theta, wl.momentum, wl.replicas, 1.0, 0.7, 0.9, reduce_mean=False)
    o, r, c = wl.table[0]
    assert rel_fro(upd[o:o + r * c].cpu().numpy(), ref["update"][o:o + r * c]) < 2e-3


def test_bf16_replicas(iso):
    spec = W.custom_spec([("m", 192, 128), ("n", 128, 320), ("v", 128, 0)], K=4, rank=3,
                         replica_dtype="bf16", shared_std=2e-3, noise_std=1e-3)
    wl = W.make_workload(spec, seed=8, device="cuda")
    assert wl.replicas.dtype == torch.bfloat16
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9)
    compare(wl, rc, th, b, upd, diag, 1.0, 0.7, 0.9)


def test_zero_pseudo_gradient(iso):
    spec = W.custom_spec([("m", 64, 48), ("v", 16, 0)], K=2, momentum_std=1e-3)
    wl = W.make_workload(spec, seed=1, device="cuda")
    reps = wl.theta.unsqueeze(0).repeat(2, 1)
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, reps=reps)
    assert rc == 0
    assert torch.count_nonzero(upd) == 0
    torch.testing.assert_close(b, 0.9 * wl.momentum, rtol=1e-6, atol=0)
    torch.testing.assert_close(th, wl.theta - 0.7 * 0.9 * (0.9 * wl.momentum), rtol=1e-6, atol=1e-9)
    assert diag["sigma_bar"] == [0.0]


def _zero_region(reps, theta, off, rows, cols, r0, r1, c0, c1):
    """Makes Delta_k = theta - theta_k exactly 0 on rows [r0, r1) x cols [c0, c1) of the
    matrix at `off`, for every worker k."""
    th = theta[off:off + rows * cols].view(rows, cols)
    for k in range(reps.shape[0]):
        reps[k, off:off + rows * cols].view(rows, cols)[r0:r1, c0:c1] = th[r0:r1, c0:c1].to(reps.dtype)


def _rank_deficient_case(iso, shapes, zeros, seed, **opts):
    """Runs a workload whose pseudo-gradients are exactly zero on the given regions
    (name -> rows [r0, r1) x cols [c0, c1)); returns (worst, per-matrix error, diag)."""
    spec = W.custom_spec(shapes, K=2, rank=4, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=seed, device="cuda")
    # a copy with the generator's row padding (every replica 16-byte aligned)
    npad = (wl.N + 63) // 64 * 64
    reps = torch.empty((wl.K, npad), dtype=wl.replicas.dtype, device="cuda")[:, :wl.N]
    reps.copy_(wl.replicas)
    t = {name: wl.table[i] for i, (name, _, _) in enumerate(shapes)}
    for name, (r0, r1, c0, c1) in zeros.items():
        o, r, c = t[name]
        _zero_region(reps, wl.theta, o, r, c, r0, r1, c0, c1)
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, reps=reps, **opts)
    assert rc == 0, iso.STATUS_NAMES.get(rc, rc)
    assert all(s == 0 for s in diag["status"])
    worst, ref = compare(wl, rc, th, b, upd, diag, 1.0, 0.7, 0.9, reps=reps)
    # the output is the partial isometry: exactly rho singular values, all alpha * sigma_bar
    u = upd.double().cpu().numpy()
    mats = [n for n, _, cc in shapes if cc > 0]
    for name, (r0, r1, c0, c1) in zeros.items():
        o, r, c = t[name]
        rank = min(r - (r1 - r0) if (c0, c1) == (0, c) else r, c - (c1 - c0) if (r0, r1) == (0, r) else c)
        sv = np.linalg.svd(u[o:o + r * c].reshape(r, c), compute_uv=False)
        assert np.all(np.abs(sv[:rank] / diag["sigma_bar"][mats.index(name)] - 1.0) < 5e-3), name
        assert np.all(sv[rank:] < 1e-6 * sv[0]), name
    return worst, diag


def test_rank_deficient_partial_isometry(iso):
    """Exactly rank-deficient pseudo-gradients (Alg. 2 / reading C3: Iso-C returns the
    partial isometry U_rho V_rho^T), with status OK.  The zeros are structural, as for
    embedding rows or input features that no worker's data touched, so the deficiency is
    exact on both sides.  Default precision where the zero lines lie on the side the Gram
    is formed over (columns of a tall or square matrix, rows of a wide one: they stay
    exactly zero), or are few: a tall matrix with 24 of 64 columns zero, a wide one with
    24 of 64 rows zero, 1024 x 1024 ones with 24 zero columns and with 24 zero rows (deep
    schedule), beside a full-rank matrix and a vector."""
    shapes = [("c40", 192, 64), ("wr", 64, 128), ("sqc", 1024, 1024), ("sq24", 1024, 1024), ("full", 96, 80),
              ("v", 33, 0)]
    zeros = {"c40": (0, 192, 40, 64), "wr": (40, 64, 0, 128), "sqc": (0, 1024, 1000, 1024),
             "sq24": (1000, 1024, 0, 1024)}
    worst, diag = _rank_deficient_case(iso, shapes, zeros, seed=21)
    print("rank-deficient (default precision) worst errors", worst, "iterations", diag["iters"])


def test_rank_deficient_many_zero_rows_full_precision(iso):
    """Zero lines on the long side in large numbers (a tall matrix with 5 nonzero rows, a
    wide one with 7 nonzero columns, a 1024 x 1024 one with 512 zero rows): with the
    two-pass steps the 11-bit operand turns the iterate's row space toward the zero
    directions (~2^-11 per step, up to ~1e-2 here), so these take full_precision = 1 (every
    step three passes), which meets the Iso-C tolerance."""
    shapes = [("r5", 128, 64), ("w7", 64, 128), ("sq512", 1024, 1024), ("c40", 192, 64), ("v", 17, 0)]
    zeros = {"r5": (5, 128, 0, 64), "w7": (0, 64, 7, 128), "sq512": (512, 1024, 0, 1024),
             "c40": (0, 192, 40, 64)}
    worst, diag = _rank_deficient_case(iso, shapes, zeros, seed=22, full_precision=1)
    print("rank-deficient (full precision) worst errors", worst, "iterations", diag["iters"])


def test_nonfinite_leaves_state_untouched(iso):
    spec = W.custom_spec([("m", 64, 48), ("v", 16, 0)], K=2, momentum_std=1e-3)
    wl = W.make_workload(spec, seed=1, device="cuda")
    reps = wl.replicas.clone()
    reps[1, 100] = float("nan")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, reps=reps)
    assert rc == iso.ERR_NONFINITE
    assert torch.equal(th, wl.theta) and torch.equal(b, wl.momentum)


def test_max_iter_reports_not_converged(iso):
    wl = W.make_workload("tiny", seed=0, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, max_iter=1)
    assert rc == iso.ERR_NOT_CONVERGED
    assert any(s == iso.ERR_NOT_CONVERGED for s in diag["status"])


@pytest.mark.parametrize("name, max_iter", [("tiny", 0), ("tiny", 1), ("gram_side_small", 0)])
def test_trace_is_tr_q_delta(iso, name, max_iter):
    """sigma_bar = tr(Q^T Delta) / r on both of its paths: summed in the epilogue of the GEMM that
    writes a converged matrix's Q (the polish update; the Gram side's Q = Delta Z), and by the
    separate trace pass for a matrix left unconverged (max_iter = 1).  Checked against the step's
    own output U = alpha sigma_bar Q: sigma_bar^2 = tr(U^T Delta) / (alpha r), Delta in fp64."""
    if name == "gram_side_small":
        spec = W.custom_spec([("e", 1024, 96), ("d", 600, 40), ("w", 200, 200)], K=2, rank=4,
                             shared_std=1e-3, noise_std=5e-4, momentum_std=0.0, name=name)
        wl = W.make_workload(spec, seed=3, device="cuda")
    else:
        wl = W.make_workload(name, seed=0, device="cuda")
    alpha = 0.5
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, alpha, 0.7, 0.9, max_iter=max_iter)
    assert rc in (0, iso.ERR_NOT_CONVERGED)
    delta = (wl.theta.double() - wl.replicas.double().mean(0)).cpu().numpy()
    u = upd.double().cpu().numpy()
    mats = [(o, r, c) for (o, r, c) in wl.table if c > 0]
    checked = 0
    for k, (o, r, c) in enumerate(mats):
        dm = delta[o:o + r * c].reshape(r, c)
        um = u[o:o + r * c].reshape(r, c)
        sb = float(diag["sigma_bar"][k])
        assert sb > 0.0, (name, max_iter, o, r, c)
        est = np.sqrt(max(0.0, float(np.sum(um * dm))) / (alpha * min(r, c)))
        assert abs(est / sb - 1.0) < 2e-4, (name, max_iter, r, c, est, sb)
        checked += 1
    assert checked == len(mats)


def test_deterministic(iso):
    wl = W.make_workload("tiny", seed=5, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    r1 = run_gpu(iso, wl, 1.0, 0.7, 0.9, plan=plan)
    r2 = run_gpu(iso, wl, 1.0, 0.7, 0.9, plan=plan)
    assert torch.equal(r1[1], r2[1]) and torch.equal(r1[2], r2[2]) and torch.equal(r1[3], r2[3])


def test_graph_loop_matches_per_launch_loop(iso):
    """The polar loop runs as one CUDA graph whose while-node stops once every matrix is
    done; under phase profiling it runs launch by launch instead.  Both give the same bits,
    the graph running at most one extra (empty) iteration, and a new max_iter rebuilds it."""
    spec = W.custom_spec(RAGGED, K=3, rank=2, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=11, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    for max_iter in (0, 20):
        l0 = plan.launches
        g = run_gpu(iso, wl, 1.0, 0.7, 0.9, plan=plan, max_iter=max_iter)
        lg = plan.launches - l0
        plan.profile(True)
        l0 = plan.launches
        h = run_gpu(iso, wl, 1.0, 0.7, 0.9, plan=plan, max_iter=max_iter)
        lh = plan.launches - l0
        plan.profile(False)
        assert g[0] == h[0] == 0
        assert torch.equal(g[1], h[1]) and torch.equal(g[2], h[2]) and torch.equal(g[3], h[3])
        assert g[4]["iters"] == h[4]["iters"] and g[4]["sigma_bar"] == h[4]["sigma_bar"]
        assert lh <= lg <= lh + lh // 2, (lg, lh)


# ---- the fast variant of Sec. 4.3: a fixed number of quintic steps, sigma_bar = ||Delta||_F / sqrt(r)

@pytest.mark.parametrize("steps", [5, 3, 8])
def test_fast_variant_ragged(iso, steps):
    """Odd and even step counts (Q in either ping-pong buffer), ragged tiles, 1-D tensors."""
    spec = W.custom_spec(RAGGED, K=3, rank=2, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=11, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, fast_steps=steps)
    assert rc == 0
    assert diag["iters"] == [steps] * len(diag["iters"]) and not any(diag["status"])
    ref = oracle_fast_step(wl.table, wl.theta, wl.momentum, wl.replicas, 1.0, 0.7, 0.9, steps)
    check_step(wl.table, th.double().cpu().numpy(), b.double().cpu().numpy(), upd.double().cpu().numpy(),
               diag["sigma_bar"], ref)


def test_fast_variant_tiny(iso):
    wl = W.make_workload("tiny", seed=0, device="cuda")
    sp = wl.spec
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, sp.alpha, sp.outer_lr, sp.momentum, fast_steps=5)
    assert rc == 0
    ref = oracle_fast_step(wl.table, wl.theta, wl.momentum, wl.replicas, sp.alpha, sp.outer_lr, sp.momentum, 5)
    check_step(wl.table, th.double().cpu().numpy(), b.double().cpu().numpy(), upd.double().cpu().numpy(),
               diag["sigma_bar"], ref)
    # the fast update is not the exact one: the rms proxy exceeds the mean singular value
    exact = run_gpu(iso, wl, sp.alpha, sp.outer_lr, sp.momentum)[4]
    assert all(f > e for f, e in zip(diag["sigma_bar"], exact["sigma_bar"]))


def test_fast_variant_180m_sampled(iso):
    """The benchmarked configuration at full size with the paper's 5 fixed steps."""
    sampled_parity(iso, "llama_180m_k8", ("layers.0.wq", "layers.5.w_gate", "layers.11.w_down"), fast_steps=5)


# ---- the ablations of Sec. 4.5 and App. B

ABLATIONS = [
    {"orth_target": 1},                                  # Iso-C of the Nesterov update P
    {"orth_target": 1, "momentum_kind": 1},              # ... with standard momentum (P = B')
    {"momentum_kind": 1},                                # standard momentum on Iso-C(Delta)
    {"scale_kind": 1},                                   # Muon's spectral scale sqrt(rows / cols)
    {"scale_kind": 1, "fast_steps": 5},                  # fixed steps + spectral scale (Muon-like)
    {"orth_target": 1, "fast_steps": 5},
    {"spectrum_kind": 1},                                # clip_high: s_i > sigma_bar -> sigma_bar
    {"spectrum_kind": 2},                                # clip_low: s_i < sigma_bar -> sigma_bar
    {"spectrum_kind": 1, "orth_target": 1},
]


@pytest.mark.parametrize("flags", ABLATIONS, ids=lambda f: "-".join(f"{k}{v}" for k, v in f.items()))
def test_ablation_variants(iso, flags):
    from oracle import variants
    spec = W.custom_spec(RAGGED, K=3, rank=2, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=11, device="cuda")
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.3, 0.7, 0.9, **flags)
    assert rc == 0
    ref = variants.isoloco_outer_step_variant(
        wl.table, wl.theta.cpu().numpy(), wl.momentum.cpu().numpy(), W.replicas_as_numpy(wl.replicas),
        alpha=1.3, eta=0.7, mu=0.9, **flags)
    ref["theta_in"] = wl.theta.double().cpu().numpy()
    sigma = diag["sigma_bar"]
    if flags.get("scale_kind"):
        # the spectral scale needs no sigma_bar, so the library does not compute it
        sigma = [s for s, (_, r, c) in zip(ref["sigma_bar"], wl.table) if c > 0]
        ref["sigma_bar"] = np.asarray(ref["sigma_bar"])
    check_step(wl.table, th.double().cpu().numpy(), b.double().cpu().numpy(), upd.double().cpu().numpy(),
               sigma, ref)


@pytest.mark.parametrize("kind", [1, 2])
def test_clip_180m_sampled(iso, kind):
    """clip_high / clip_low on the benchmarked configuration at full size."""
    sampled_parity(iso, "llama_180m_k8", ("layers.0.wq", "layers.5.w_gate", "layers.11.w_down", "head"),
                   spectrum_kind=kind)


@pytest.mark.parametrize("kind", [1, 2])
def test_clip_tiny_bf16_and_zero(iso, kind):
    """bf16 replicas; then replicas equal to theta (Delta = 0): U = 0, status OK."""
    from oracle import variants
    spec = W.custom_spec(W.tiny_shapes(), K=2, rank=4, replica_dtype="bf16", momentum_std=1e-4)
    wl = W.make_workload(spec, seed=21, device="cuda")
    rc, th, b, upd, diag, plan = run_gpu(iso, wl, 1.0, 0.7, 0.9, spectrum_kind=kind)
    assert rc == 0
    ref = variants.isoloco_outer_step_variant(
        wl.table, wl.theta.cpu().numpy(), wl.momentum.cpu().numpy(), W.replicas_as_numpy(wl.replicas),
        alpha=1.0, eta=0.7, mu=0.9, spectrum_kind=kind)
    ref["theta_in"] = wl.theta.double().cpu().numpy()
    check_step(wl.table, th.double().cpu().numpy(), b.double().cpu().numpy(), upd.double().cpu().numpy(),
               diag["sigma_bar"], ref)
    same = wl.theta.to(torch.bfloat16).float().to(torch.bfloat16).expand(wl.K, -1).contiguous()
    th0 = wl.theta.to(torch.bfloat16).float()
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, reps=same, theta=th0, plan=plan, spectrum_kind=kind)
    assert rc == 0 and float(upd.abs().max()) == 0.0


def test_clip_options_rejected(iso):
    wl = W.make_workload("tiny", seed=0, device="cuda")
    for flags in ({"spectrum_kind": 4}, {"spectrum_kind": -1}, {"spectrum_kind": 1, "fast_steps": 5},
                  {"spectrum_kind": 2, "scale_kind": 1}, {"spectrum_kind": 3, "fast_steps": 5}):
        with pytest.raises(iso.IsolocoError):
            run_gpu(iso, wl, 1.0, 0.7, 0.9, **flags)


def test_excluded_matrix_is_listed_as_1d(iso):
    """Sec. 4.5's exclusion of embedding/head from Iso-C: the caller lists the tensor as 1-D."""
    spec = W.custom_spec([("embed", 96, 64), ("w", 64, 48), ("head", 64, 96), ("norm", 64, 0)], K=2, rank=2)
    wl = W.make_workload(spec, seed=3, device="cuda")
    table = [(o, r * c, 0) if i in (0, 2) else (o, r, c) for i, (o, r, c) in enumerate(wl.table)]
    plan = iso.Plan(table, wl.N, wl.K)
    assert plan.num_matrices == 1
    rc, th, b, upd, diag, _ = run_gpu(iso, wl, 1.0, 0.7, 0.9, plan=plan)
    assert rc == 0
    ref = oracle_step(table, wl.theta, wl.momentum, wl.replicas, 1.0, 0.7, 0.9)
    ref["theta_in"] = wl.theta.double().cpu().numpy()
    check_step(table, th.double().cpu().numpy(), b.double().cpu().numpy(), upd.double().cpu().numpy(),
               diag["sigma_bar"], ref)


def test_diloco_outer_step(iso):
    spec = W.custom_spec(RAGGED, K=3, rank=2, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=6, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    th, b = wl.theta.clone(), wl.momentum.clone()
    assert plan.diloco_outer_step(th, b, wl.replicas, iso.make_opts(outer_lr=0.7, momentum=0.9, sync=True)) == 0
    ref = oracle.diloco_outer_step(wl.theta.cpu().numpy(), wl.momentum.cpu().numpy(),
                                   W.replicas_as_numpy(wl.replicas), eta=0.7, mu=0.9)
    assert elementwise_rel(th.cpu().numpy(), ref["theta"]) < 1e-5
    assert elementwise_rel(b.cpu().numpy(), ref["momentum"]) < 1e-5


def test_iso_c_merge(iso):
    spec = W.custom_spec([("m", 96, 64), ("n", 64, 160), ("v", 33, 0)], K=3, rank=2)
    wl = W.make_workload(spec, seed=9, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    out = torch.empty_like(wl.theta)
    assert plan.iso_c_merge(wl.theta, wl.replicas, 0.8, out) == 0
    assert plan.last_status() == 0
    ref = oracle.iso_c_merge(wl.table, wl.theta.cpu().numpy(), W.replicas_as_numpy(wl.replicas), alpha=0.8)
    for (o, r, c) in wl.table:
        sl = slice(o, o + r * (c or 1))
        got = out[sl].double().cpu().numpy() - wl.theta[sl].double().cpu().numpy()
        want = ref["out"][sl] - wl.theta[sl].double().cpu().numpy()
        assert rel_fro(got, want) < (2e-3 if c else 1e-5)


def test_host_buffer_entry_point(iso):
    wl = W.make_workload("tiny", seed=2, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    th, b = wl.theta.clone(), wl.momentum.clone()
    assert plan.outer_step(th, b, wl.replicas, iso.make_opts(sync=True)) == 0
    # pinned buffers: read in place by the reduce, theta / B copied during the polar iteration
    th_h = wl.theta.cpu().pin_memory()
    b_h = wl.momentum.cpu().pin_memory()
    reps_h = [wl.replicas[k].cpu().pin_memory() for k in range(wl.K)]
    assert plan.outer_step_host(th_h, b_h, reps_h, iso.make_opts()) == 0
    assert torch.equal(th_h, th.cpu()) and torch.equal(b_h, b.cpu())
    # pageable buffers: staged copies first
    th_p, b_p = wl.theta.cpu().clone(), wl.momentum.cpu().clone()
    reps_p = [wl.replicas[k].cpu().clone() for k in range(wl.K)]
    assert not th_p.is_pinned()
    assert plan.outer_step_host(th_p, b_p, reps_p, iso.make_opts()) == 0
    assert torch.equal(th_p, th.cpu()) and torch.equal(b_p, b.cpu())
    # pinned again, with the orthogonalise-P ablation (its reduce reads B in place too)
    th2, b2 = wl.theta.clone(), wl.momentum.clone()
    assert plan.outer_step(th2, b2, wl.replicas, iso.make_opts(sync=True, orth_target=1)) == 0
    th_h.copy_(wl.theta.cpu()); b_h.copy_(wl.momentum.cpu())
    assert plan.outer_step_host(th_h, b_h, reps_h, iso.make_opts(orth_target=1)) == 0
    assert torch.equal(th_h, th2.cpu()) and torch.equal(b_h, b2.cpu())


def sampled_parity(iso, workload, pick_names, fast_steps=0, **ablation):
    """A configuration at full size on the GPU (the launch configuration bench.py times),
    checked against the oracle on the sampled matrices plus every 1-D tensor (each matrix's
    Iso-C and each element's Nesterov step are independent of the others)."""
    wl = W.make_workload(workload, seed=0, device="cuda")
    sp = wl.spec
    rc, th, b, upd, diag, plan = run_gpu(iso, wl, sp.alpha, sp.outer_lr, sp.momentum, fast_steps=fast_steps,
                                         **ablation)
    assert rc == 0
    names = [s[0] for s in sp.shapes]
    pick = [names.index(n) for n in pick_names]
    pick += [i for i, s in enumerate(sp.shapes) if s[2] == 0]
    # the oracle gets only the sampled tensors, re-packed densely (host copies of the inputs)
    sub_table, parts, off = [], [], 0
    for i in pick:
        o, r, c = wl.table[i]
        n = r * (c or 1)
        sub_table.append((off, r, c))
        parts.append((o, n))
        off += n
    idx = torch.cat([torch.arange(o, o + n, device="cuda") for o, n in parts])
    if ablation:
        from oracle import variants
        ref = variants.isoloco_outer_step_variant(
            sub_table, wl.theta[idx].cpu().numpy(), wl.momentum[idx].cpu().numpy(),
            W.replicas_as_numpy(wl.replicas[:, idx]), alpha=sp.alpha, eta=sp.outer_lr, mu=sp.momentum,
            fast_steps=fast_steps, **ablation)
    elif fast_steps:
        ref = oracle_fast_step(sub_table, wl.theta[idx], wl.momentum[idx], wl.replicas[:, idx], sp.alpha,
                               sp.outer_lr, sp.momentum, fast_steps)
    else:
        ref = oracle.isoloco_outer_step(sub_table, wl.theta[idx].cpu().numpy(), wl.momentum[idx].cpu().numpy(),
                                        W.replicas_as_numpy(wl.replicas[:, idx]), alpha=sp.alpha,
                                        eta=sp.outer_lr, mu=sp.momentum)
    ref["theta_in"] = wl.theta[idx].double().cpu().numpy()
    mat_index = {p: j for j, p in enumerate([i for i, s in enumerate(sp.shapes) if s[2] > 0])}
    sig = [diag["sigma_bar"][mat_index[i]] for i in pick if sp.shapes[i][2] > 0]
    worst = check_step(sub_table, th[idx].double().cpu().numpy(), b[idx].double().cpu().numpy(),
                       upd[idx].double().cpu().numpy(), sig, ref)
    assert all(s == 0 for s in diag["status"])
    print(workload, "worst errors", worst, "iterations", sorted(set(diag["iters"])))
    del wl, th, b, upd, plan
    torch.cuda.empty_cache()


def test_llama_180m_k8_every_matrix(iso):
    """The benchmarked configuration (180M shapes, K = 8) in the launch configuration the
    bench times, checked against the oracle on every tensor: all 86 matrices (including the
    1024 x 1024 ones that need the most polar iterations) and every vector."""
    wl = W.make_workload("llama_180m_k8", seed=0, device="cuda")
    sp = wl.spec
    rc, th, b, upd, diag, plan = run_gpu(iso, wl, sp.alpha, sp.outer_lr, sp.momentum)
    assert rc == 0
    assert all(s == 0 for s in diag["status"])
    ref = oracle.isoloco_outer_step(wl.table, wl.theta.cpu().numpy(), wl.momentum.cpu().numpy(),
                                    W.replicas_as_numpy(wl.replicas), alpha=sp.alpha, eta=sp.outer_lr,
                                    mu=sp.momentum)
    ref["theta_in"] = wl.theta.double().cpu().numpy()
    u = upd.double().cpu().numpy()
    worst = check_step(wl.table, th.double().cpu().numpy(), b.double().cpu().numpy(), u, diag["sigma_bar"], ref)
    rows, mi = [], 0
    for pi, (o, r, c) in enumerate(wl.table):
        if not c:
            continue
        sl = slice(o, o + r * c)
        rows.append((rel_fro(u[sl], ref["update"][sl]), sp.shapes[pi][0], f"{r}x{c}", diag["iters"][mi]))
        mi += 1
    assert len(rows) == 86
    rows.sort(reverse=True)
    print("180M K=8, all 86 matrices: worst", worst)
    for e, name, shape, it in rows[:8]:
        print(f"  {name:18s} {shape:10s} iterations {it:2d}  Iso-C rel. Frobenius error {e:.3e}")
    # the matrices that need a second schedule round are among those checked
    slow = [x for x in rows if x[3] > 12]
    print("  matrices with more than 12 iterations:", [(x[1], x[3], f"{x[0]:.2e}") for x in slow])
    assert slow, "expected some 1024 x 1024 matrices to need a second schedule round"
    del wl, th, b, upd, plan
    torch.cuda.empty_cache()


def test_llama_180m_k16_every_square(iso):
    """180M shapes with K = 16: every 1024 x 1024 matrix (the ill-conditioned bucket) and
    one matrix of each other shape, plus every vector."""
    names = [s[0] for s in W.SPECS["llama_180m_k16"].shapes if s[1] == s[2]]
    sampled_parity(iso, "llama_180m_k16", tuple(names) + ("layers.7.w_up", "layers.0.w_down", "embed"))


@pytest.mark.parametrize("workload,pick", [
    ("llama_1b_k8", ("layers.0.wq", "layers.11.w_gate", "layers.23.w_down")),
    ("llama_3b_k4", ("layers.0.wv",)),   # bf16 replicas; 3072-wide matrices keep the oracle sample small
])
def test_larger_configs_sampled(iso, workload, pick):
    """The other configurations at full size (up to 3.4e9 parameters with 4 bf16 replicas),
    sampled matrices plus every 1-D tensor."""
    sampled_parity(iso, workload, pick)
