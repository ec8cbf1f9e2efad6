"""Comparison helpers shared by the GPU parity tests (oracle vs CUDA path)."""
import numpy as np

import oracle
from paper_2607_03011_gb300 import workloads as W


def oracle_step(table, theta, mom, reps, alpha, eta, mu, only=None, reduce_mean=True):
    """Runs the fp64 oracle on host copies of seeded inputs (never on CUDA outputs)."""
    th = theta.detach().cpu().numpy().astype(np.float32)
    b = mom.detach().cpu().numpy().astype(np.float32)
    r = W.replicas_as_numpy(reps)
    return oracle.isoloco_outer_step(table, th, b, r, alpha=alpha, eta=eta, mu=mu, only=only,
                                     reduce_mean=reduce_mean)


def oracle_fast_step(table, theta, mom, reps, alpha, eta, mu, steps, only=None):
    """The fast variant (Sec. 4.3) in fp64: the oracle's reduction, then its own fixed-step
    schedule (oracle/fast_ns.py) on every 2-D tensor and Nesterov."""
    from oracle import fast_ns
    th = theta.detach().cpu().numpy().astype(np.float32)
    b = mom.detach().cpu().numpy().astype(np.float32)
    delta = oracle.pseudo_gradient(th, W.replicas_as_numpy(reps), mode=0)
    ref = fast_ns.isoloco_outer_step_fast(table, th, b, delta, alpha, eta, mu, fast_ns.fast_schedule(steps),
                                          only=only)
    ref["theta_in"] = th.astype(np.float64)
    return ref


def rel_fro(a, b):
    a = np.asarray(a, np.float64); b = np.asarray(b, np.float64)
    nb = np.linalg.norm(b)
    return np.linalg.norm(a - b) / nb if nb > 0 else np.linalg.norm(a)


def elementwise_rel(a, b, floor_frac=1.0):
    """max |a-b| / max(|b|, floor) with floor = floor_frac * rms(b)."""
    a = np.asarray(a, np.float64); b = np.asarray(b, np.float64)
    floor = floor_frac * np.sqrt(np.mean(b * b)) if b.size else 0.0
    den = np.maximum(np.abs(b), floor)
    den[den == 0] = 1.0
    return float(np.max(np.abs(a - b) / den)) if a.size else 0.0


def check_step(table, gpu_theta, gpu_mom, gpu_upd, gpu_sigma, ref, only=None,
               tol_iso=2e-3, tol_sigma=1e-4, tol_1d=1e-5):
    """Asserts the tolerances of the outer step; returns a summary dict of the worst errors."""
    worst = {"iso_rel_fro": 0.0, "sigma_rel": 0.0, "theta_1d": 0.0, "mom_1d": 0.0, "theta_2d_rel_fro": 0.0}
    mi = 0
    for pi, (o, r, c) in enumerate(table):
        n = r * (c if c else 1)
        sl = slice(o, o + n)
        if only is not None and pi not in only:
            if c:
                mi += 1
            continue
        if c:
            e = rel_fro(gpu_upd[sl], ref["update"][sl])
            assert e <= tol_iso, (pi, r, c, e)
            s_ref = ref["sigma_bar"][pi]
            es = abs(gpu_sigma[mi] - s_ref) / s_ref if s_ref else abs(gpu_sigma[mi])
            assert es <= tol_sigma, (pi, r, c, es)
            dth = rel_fro(gpu_theta[sl] - ref["theta_in"][sl], ref["theta"][sl] - ref["theta_in"][sl])
            worst["iso_rel_fro"] = max(worst["iso_rel_fro"], e)
            worst["sigma_rel"] = max(worst["sigma_rel"], es)
            worst["theta_2d_rel_fro"] = max(worst["theta_2d_rel_fro"], dth)
            mi += 1
        else:
            et = elementwise_rel(gpu_theta[sl], ref["theta"][sl])
            eb = elementwise_rel(gpu_mom[sl], ref["momentum"][sl])
            assert et <= tol_1d and eb <= tol_1d, (pi, et, eb)
            worst["theta_1d"] = max(worst["theta_1d"], et)
            worst["mom_1d"] = max(worst["mom_1d"], eb)
    return worst
