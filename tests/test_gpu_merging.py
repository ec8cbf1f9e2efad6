"""DiLoCo outer step with the merging aggregators of Sec. 3.2 (TIES, DARE): CUDA path vs
the oracle (oracle/merging.py) on the same seeded inputs, through the C ABI.

The momentum buffer starts at 0, so the new momentum B' = mu * 0 + U is the merged
direction U exactly.  The decisions are compared bit for bit: TIES's trim and sign
election through the zero and sign pattern of U (a mean of same-signed values, so it
cannot cancel), and with one worker the kept mask itself, for TIES and for DARE (whose U
at K > 1 is a sum of mixed signs that can cancel to 0 on one side only; a wrong drop
there moves U by |Delta_k| / K, far outside the value tolerance).  U = B' elementwise to
a relative 1e-5 (fp32 sums of at most K terms against fp64), and theta' to its own fp32
rounding plus 1e-5 of the update.

The oracle elects TIES's sign from the exact kept mass; the library sums in fp32, whose
result is within K 2^-24 sum_k |kept_k| of the exact mass.  Entries whose exact mass lies
inside that bound may elect either sign there: they are exempt from the sign check, and
their U must equal one of the two candidates the oracle gives (the disjoint mean of the
kept positive or of the kept negative values) or 0.  Every other entry is compared bit
for bit; the exempt count is printed.
"""
import numpy as np
import pytest
import torch

from oracle import merging
from paper_2607_03011_gb300 import workloads as W
from parity import elementwise_rel

pytestmark = pytest.mark.gpu

AGG = {"ties": 1, "dare": 2}
# ragged: N = 188375 (N mod 4 = 3, the scalar tail)
SHAPES = [("a", 65, 130), ("b", 130, 65), ("c", 1, 9), ("h", 300, 257), ("i", 257, 300), ("j", 129, 129),
          ("v", 7, 0), ("e", 200, 3), ("f", 3, 200), ("t", 3, 0)]


@pytest.fixture(scope="module")
def iso():
    from paper_2607_03011_gb300 import isoloco
    isoloco.lib()
    return isoloco


def run(iso, wl, agg, s, seed=1234, eta=0.7, mu=0.9, reduce_mean=True, plan=None):
    plan = plan or iso.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    th = wl.theta.clone()
    b = torch.zeros_like(th)
    rc = plan.diloco_outer_step(th, b, wl.replicas,
                                iso.make_opts(outer_lr=eta, momentum=mu, reduce_mean=reduce_mean, sync=True,
                                              aggregator=AGG[agg], sparsity=s, seed=seed))
    return rc, th, b


def ties_exempt(parts, K):
    """Entries whose exact kept mass lies within the fp32 election's rounding bound
    K 2^-24 sum_k |kept_k| of 0 (and that keep something)."""
    return (np.abs(parts["mass"]) <= K * 2.0 ** -24 * parts["abs_mass"]) & (parts["abs_mass"] > 0)


def ties_check(u_gpu, parts, K, where=""):
    """TIES's U against the oracle's exact election (module docstring); returns the number
    of entries exempt from the sign check."""
    u_ref = parts["update"]
    amb = ties_exempt(parts, K)
    ok = ~amb
    assert np.array_equal(u_gpu[ok] == 0, u_ref[ok] == 0), f"trim decisions differ{where}"
    assert np.array_equal(np.sign(u_gpu[ok]), np.sign(u_ref[ok])), f"elected signs differ{where}"
    assert elementwise_rel(u_gpu[ok], u_ref[ok]) < 1e-5
    if amb.any():
        ua = u_gpu[amb]
        rms = np.sqrt(np.mean(u_ref ** 2)) if u_ref.size else 0.0
        best = np.min(np.stack([np.abs(ua - parts["u_pos"][amb]) / np.maximum(np.abs(parts["u_pos"][amb]), rms),
                                np.abs(ua - parts["u_neg"][amb]) / np.maximum(np.abs(parts["u_neg"][amb]), rms),
                                np.abs(ua) / max(rms, 1e-300)]), axis=0)
        assert np.max(best) < 1e-5, f"an exempt entry is none of the election's candidates{where}"
    return int(amb.sum())


def check(th, b, ref, theta_in, agg, K):
    u_gpu = b.double().cpu().numpy()
    u_ref = ref["update"]
    if agg == "ties":
        nex = ties_check(u_gpu, ref["ties_parts"], K)
        print(f"TIES: {nex} of {u_gpu.size} entries within the fp32 election bound (exempt from the sign check)")
        # theta' follows U: compare it where the election is decided
        ok = ~ties_exempt(ref["ties_parts"], K)
        check_theta(th.double().cpu().numpy()[ok], ref["theta"][ok], theta_in[ok])
        return
    assert elementwise_rel(u_gpu, u_ref) < 1e-5
    check_theta(th.double().cpu().numpy(), ref["theta"], theta_in)


def check_theta(th_gpu, th_ref, theta_in):
    """theta' is stored in fp32: its error is its own rounding (<= 2^-24 |theta'|) plus the
    update's error (<= 1e-5 of the update, floored at the update's rms for entries whose
    sum over workers cancels, as in elementwise_rel)."""
    err = np.abs(th_gpu - th_ref)
    upd = np.abs(th_ref - theta_in)
    rms = np.sqrt(np.mean(upd ** 2))
    bound = 2.0 ** -24 * np.abs(th_ref) * 1.01 + 1e-5 * np.maximum(upd, rms) + 1e-30
    assert (err <= bound).all(), f"theta error {np.max(err / bound):.3g} x the bound"


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("agg,s", [("ties", 0.0), ("ties", 0.1), ("ties", 0.5), ("ties", 0.9), ("ties", 0.999),
                                   ("dare", 0.0), ("dare", 0.1), ("dare", 0.5), ("dare", 0.9)])
def test_ragged(iso, agg, s, dtype):
    spec = W.custom_spec(SHAPES, K=3, rank=2, replica_dtype=dtype)
    wl = W.make_workload(spec, seed=11, device="cuda")
    rc, th, b = run(iso, wl, agg, s)
    assert rc == 0
    th_in = wl.theta.cpu().numpy()
    ref = merging.merged_outer_step(th_in, np.zeros(wl.N, np.float32), W.replicas_as_numpy(wl.replicas),
                                    agg, sparsity=s, seed=1234, eta=0.7, mu=0.9)
    check(th, b, ref, th_in.astype(np.float64), agg, K=wl.K)


@pytest.mark.parametrize("agg,s", [("ties", 0.3), ("dare", 0.3)])
def test_single_worker_mask_is_exact(iso, agg, s):
    """K = 1: U = Delta on the kept entries (TIES: its own disjoint mean; DARE: rescaled),
    so U != 0 is the kept mask itself."""
    spec = W.custom_spec(SHAPES, K=1, rank=2)
    wl = W.make_workload(spec, seed=12, device="cuda")
    rc, th, b = run(iso, wl, agg, s, seed=99)
    assert rc == 0
    d = merging.task_vectors(wl.theta.cpu().numpy(), W.replicas_as_numpy(wl.replicas))
    mask = merging.ties_trim(d, s)[0][0] if agg == "ties" else merging.dare_mask(1, wl.N, s, 99)[0]
    got = (b.cpu().numpy() != 0)
    assert np.array_equal(got, mask & (d[0] != 0))
    if agg == "ties":
        assert got.sum() >= merging.ties_keep_count(wl.N, s)


def test_sum_reduction_and_sgd(iso):
    """DARE with reduce_mean = 0 (the sum) and TIES / DARE with mu = 0 (the SGD outer step
    of the paper's merging comparison)."""
    spec = W.custom_spec(SHAPES, K=4, rank=2)
    wl = W.make_workload(spec, seed=13, device="cuda")
    th_in = wl.theta.cpu().numpy()
    reps = W.replicas_as_numpy(wl.replicas)
    for agg, mean, mu in (("dare", False, 0.9), ("dare", True, 0.0), ("ties", True, 0.0)):
        rc, th, b = run(iso, wl, agg, 0.2, seed=5, mu=mu, reduce_mean=mean)
        assert rc == 0
        ref = merging.merged_outer_step(th_in, np.zeros(wl.N, np.float32), reps, agg, sparsity=0.2, seed=5,
                                        eta=0.7, mu=mu, reduce_mean=mean)
        check(th, b, ref, th_in.astype(np.float64), agg, K=wl.K)


@pytest.mark.parametrize("agg", ["ties", "dare"])
def test_mid_size_many_grid_strides(iso, agg):
    """N = 4.2e6 + 1001 (several grid-stride rounds of every pass; N mod 4 = 1), K = 5."""
    spec = W.custom_spec([("m", 2048, 2048), ("x", 1001, 0)], K=5, rank=8, shared_std=2e-5, noise_std=2e-5,
                         theta_std=0.02)
    wl = W.make_workload(spec, seed=14, device="cuda")
    rc, th, b = run(iso, wl, agg, 0.1, seed=3)
    assert rc == 0
    th_in = wl.theta.cpu().numpy()
    ref = merging.merged_outer_step(th_in, np.zeros(wl.N, np.float32), W.replicas_as_numpy(wl.replicas),
                                    agg, sparsity=0.1, seed=3, eta=0.7, mu=0.9)
    check(th, b, ref, th_in.astype(np.float64), agg, K=wl.K)


def test_bad_options_rejected(iso):
    spec = W.custom_spec(SHAPES, K=2, rank=2)
    wl = W.make_workload(spec, seed=15, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    th, b = wl.theta.clone(), wl.momentum.clone()
    for kw in ({"aggregator": 3}, {"aggregator": -1}, {"aggregator": 1, "sparsity": 1.0},
               {"aggregator": 2, "sparsity": -0.1}, {"aggregator": 2, "sparsity": float("nan")}):
        with pytest.raises(iso.IsolocoError):
            plan.diloco_outer_step(th, b, wl.replicas, iso.make_opts(sync=True, **kw))
    assert torch.equal(th, wl.theta) and torch.equal(b, wl.momentum)


def test_nonfinite_is_reported(iso):
    spec = W.custom_spec(SHAPES, K=2, rank=2)
    wl = W.make_workload(spec, seed=16, device="cuda")
    wl.replicas[1, 777] = float("nan")
    for agg in ("ties", "dare"):
        rc, _, _ = run(iso, wl, agg, 0.1)
        assert rc == iso.ERR_NONFINITE


@pytest.mark.parametrize("agg", ["ties", "dare"])
def test_llama_180m_k8_full(iso, agg):
    """The 180M-parameter, K = 8 workload at full size (the launch configuration the bench
    times with --aggregator), every entry compared; the oracle runs in chunks, with TIES's
    per-worker thresholds taken over the whole task vectors first."""
    wl = W.make_workload("llama_180m_k8", seed=0, device="cuda")
    s, seed = 0.1, 2024
    rc, th, b = run(iso, wl, agg, s, seed=seed, eta=wl.spec.outer_lr, mu=wl.spec.momentum)
    assert rc == 0
    n, K = wl.N, wl.K
    th_in = wl.theta.cpu().numpy()
    u_gpu = b.cpu().numpy()
    th_gpu = th.cpu().numpy()
    del th, b
    if agg == "ties":
        thr = np.empty(K, np.float32)
        for k in range(K):
            dk = merging.task_vectors(th_in, W.replicas_as_numpy(wl.replicas[k:k + 1]))
            thr[k] = merging.ties_thresholds(dk, s)[0]
            del dk
    step = 1 << 24
    exempt = 0
    for c0 in range(0, n, step):
        c1 = min(n, c0 + step)
        d = merging.task_vectors(th_in[c0:c1], W.replicas_as_numpy(wl.replicas[:, c0:c1]))
        ug = u_gpu[c0:c1].astype(np.float64)
        t_in = th_in[c0:c1].astype(np.float64)
        sel = slice(None)
        if agg == "ties":
            parts = merging.ties_merge(d, s, thr=thr, parts=True)
            u_ref = parts["update"]
            exempt += ties_check(ug, parts, K, where=f" in [{c0}, {c1})")
            sel = ~ties_exempt(parts, K)
        else:
            u_ref = merging.dare_merge(d, s, seed, n_total=n, idx=np.arange(c0, c1))
            assert elementwise_rel(ug, u_ref) < 1e-5
        t_ref = t_in - wl.spec.outer_lr * (u_ref + wl.spec.momentum * u_ref)
        check_theta(th_gpu[c0:c1].astype(np.float64)[sel], t_ref[sel], t_in[sel])
    if agg == "ties":
        print(f"TIES at 180M K=8: {exempt} of {n} entries within the fp32 election bound (exempt from the sign check)")
    del wl
    torch.cuda.empty_cache()


def test_dare_mask_at_k8_with_64bit_draw_numbers(iso):
    """Each worker's drop mask at K = 8 and N = 6e8 + 1 (draw numbers k * N + i + 1 up to
    4.8e9, past 2^32; N mod 4 = 1).  Delta_k = 2^(k - 20) everywhere, p = 1/2 and K = 8 make
    every scale a power of two, so U * 2^22 = sum of 2^k over the kept workers exactly: an
    8-bit record of the masks, compared at 2^20 sampled entries and the tail, and the
    per-worker drop rate over all entries."""
    K, n = 8, 600_000_001
    npad = (n + 63) // 64 * 64
    theta = torch.zeros(n, device="cuda")
    mom = torch.zeros(n, device="cuda")
    reps = torch.empty((K, npad), device="cuda")[:, :n]
    for k in range(K):
        reps[k].fill_(-(2.0 ** (k - 20)))
    plan = iso.Plan([], n, K)
    opts = iso.make_opts(outer_lr=0.7, momentum=0.9, sync=True, aggregator=2, sparsity=0.5, seed=0xC0FFEE)
    assert plan.diloco_outer_step(theta, mom, reps, opts) == 0
    del reps, theta
    bits = torch.round(mom * 2.0 ** 22).to(torch.int32)
    assert int(bits.min()) >= 0 and int(bits.max()) <= 255
    # the code is exact: U is a multiple of 2^-22
    assert torch.equal(bits.float() * 2.0 ** -22, mom)
    rng = np.random.default_rng(1)
    idx = np.concatenate([rng.integers(0, n, size=1 << 20), np.arange(n - 9, n)])
    got = bits[torch.from_numpy(idx).cuda()].cpu().numpy()
    want = merging.dare_mask(K, n, 0.5, 0xC0FFEE, idx=idx)
    code = (want * (1 << np.arange(K))[:, None]).sum(axis=0)
    assert np.array_equal(got, code)
    rate = [float(((bits >> k) & 1).float().mean()) for k in range(K)]
    assert all(abs(r - 0.5) < 5 * 0.5 / np.sqrt(n) for r in rate), rate


def test_ties_bracket_fallback_on_tied_magnitudes(iso):
    """|Delta_k| takes two values only, so the sampled bracket around the threshold holds
    about half of all entries and overflows its candidate segments: the trim falls back to
    the radix passes over the replicas, and the result is still the exact threshold's."""
    n, K = (1 << 22) + 5, 3
    g = torch.Generator(device="cuda").manual_seed(5)
    theta = torch.randn(n, device="cuda", generator=g) * 0.02
    npad = (n + 63) // 64 * 64
    reps = torch.empty((K, npad), device="cuda")[:, :n]
    for k in range(K):
        mag = torch.where(torch.rand(n, device="cuda", generator=g) < 0.5, 1e-3, 2e-3)
        sign = torch.where(torch.rand(n, device="cuda", generator=g) < 0.5, -1.0, 1.0)
        reps[k] = theta - sign * mag
    plan = iso.Plan([], n, K)
    th, b = theta.clone(), torch.zeros_like(theta)
    opts = iso.make_opts(outer_lr=0.7, momentum=0.9, sync=True, aggregator=1, sparsity=0.5)
    assert plan.diloco_outer_step(th, b, reps, opts) == 0
    th_in = theta.cpu().numpy()
    ref = merging.merged_outer_step(th_in, np.zeros(n, np.float32), [r.cpu().numpy() for r in reps], "ties",
                                    sparsity=0.5, eta=0.7, mu=0.9)
    check(th, b, ref, th_in.astype(np.float64), "ties", K=K)
