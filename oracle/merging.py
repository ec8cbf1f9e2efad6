"""fp64 oracle for the merging aggregators of Sec. 3.2 inside Alg. 1 (test infrastructure).

Sec. 3.2 turns DiLoCo's mean of the pseudo-gradients Delta_k = theta - theta_k into a
model-merging rule: the Delta_k play the task vectors and the outer step applies the merged
direction U with the outer optimiser (Nesterov; mu = 0 is the SGD step of Sec. 5.1).

* TIES (trim, elect sign, disjoint merge; Yadav et al. 2023, restated from its definition):
  - trim: each worker keeps its n_keep = N - floor(sparsity * N) largest magnitudes
    |Delta_k| over all N entries of its task vector; entries equal to the n_keep-th largest
    are kept too (ties kept);
  - elect: the sign of the total mass of the kept values, sign(sum_k kept_k), taken
    exactly: an fp64 sum decides every entry whose sum clears that sum's own rounding
    bound, and the few that do not are summed as exact rationals, so the election depends
    on neither the order of the workers nor a working precision;
  - merge: U = mean of the kept values whose sign is the elected one (fp64), 0 if the
    elected sign is 0.
* DARE (drop and rescale; Yu et al. 2024): each entry of each Delta_k is dropped with
  probability p and the rest scaled by 1 / (1 - p); then the mean (or sum) over workers as
  in Alg. 1.  The drop of entry i of worker k is decided by SplitMix64 (Steele, Lea and
  Flood 2014), written here from its published definition: output number n from state s is
  mix(s + n * 0x9E3779B97F4A7C15), and u = (output >> 40) * 2^-24; dropped when u < p,
  with n = k * N + i + 1.

Delta_k is the fp32 difference of the stored fp32 values (bf16 replicas upcast exactly),
as both sides read it.  Only ``tests/`` may import this module; it shares no code with the
CUDA library.

Parity status: pinned (``tests/test_oracle_merging.py``: SplitMix64 known answers, a
hand-worked TIES example, election by mass, ties at the threshold, reductions to the mean
at sparsity 0, DARE's drop rate and unbiasedness).
"""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np

from . import nesterov

GAMMA = 0x9E3779B97F4A7C15
MASK64 = (1 << 64) - 1


def splitmix64(state: int, n: int) -> int:
    """Output number n (n >= 1) of SplitMix64 from state ``state`` (plain Python ints)."""
    z = (state + n * GAMMA) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def splitmix64_array(state: int, n: np.ndarray) -> np.ndarray:
    """The same on a uint64 array of output numbers (numpy's uint64 arithmetic wraps)."""
    with np.errstate(over="ignore"):
        z = np.uint64(state) + np.asarray(n, dtype=np.uint64) * np.uint64(GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def _replica_f32(r: np.ndarray) -> np.ndarray:
    r = np.ascontiguousarray(r)
    if r.dtype == np.uint16:
        return (r.astype(np.uint32) << np.uint32(16)).view(np.float32)
    return r.astype(np.float32, copy=False)


def task_vectors(theta, replicas) -> np.ndarray:
    """Delta_k = theta - theta_k in fp32, shape [K, N]."""
    th = np.ascontiguousarray(theta, dtype=np.float32).ravel()
    return np.stack([th - _replica_f32(r).ravel() for r in replicas])


def ties_keep_count(n: int, sparsity: float) -> int:
    """Entries each worker keeps: N - floor(sparsity * N), sparsity as fp32."""
    return n - int(math.floor(float(np.float32(sparsity)) * n))


def ties_thresholds(d: np.ndarray, sparsity: float, n_total: int | None = None) -> np.ndarray:
    """Per worker, the n_keep-th largest |d_k| (the value at that position of the sorted
    magnitudes).  d [K, N] holds whole task vectors."""
    n = d.shape[1] if n_total is None else n_total
    keep = ties_keep_count(n, sparsity)
    return np.array([np.partition(np.abs(dk), n - keep)[n - keep] for dk in d], dtype=np.float32)


def ties_trim(d: np.ndarray, sparsity: float):
    """(mask [K, N], thresholds [K]): keep |d_k| >= the n_keep-th largest |d_k|."""
    thr = ties_thresholds(d, sparsity)
    return np.abs(d) >= thr[:, None], thr


def ties_elect(kept: np.ndarray) -> np.ndarray:
    """Elected sign per entry (-1, 0 or 1): the sign of the exact sum over workers of the
    kept fp32 values kept [K, N].  The fp64 sum of K fp32 values is within
    K * 2^-53 * sum|kept| of the exact one, so its sign is exact wherever it clears that
    bound; the remaining entries (exact or near-exact cancellations) are summed as
    rationals."""
    k64 = kept.astype(np.float64)
    s = k64.sum(axis=0)
    bound = kept.shape[0] * 2.0 ** -53 * np.abs(k64).sum(axis=0)
    gamma = np.sign(s)
    for i in np.nonzero((np.abs(s) <= bound) & (bound > 0))[0]:
        gamma[i] = np.sign(sum((Fraction(float(x)) for x in kept[:, i]), Fraction(0)))
    return gamma


def ties_merge(d: np.ndarray, sparsity: float, thr: np.ndarray | None = None, parts: bool = False):
    """TIES direction U in fp64 from fp32 task vectors d [K, N]; thr (per worker) given when
    d holds only some entries of the task vectors.  With parts=True also returns the
    disjoint means of the kept positive and kept negative values (the two values U can
    take), the kept mass sum_k kept_k and sum_k |kept_k| (fp64), for callers that check an
    election taken in a narrower precision."""
    if thr is None:
        thr = ties_thresholds(d, sparsity)
    kept = np.where(np.abs(d) >= np.asarray(thr, np.float32)[:, None], d, np.float32(0.0)).astype(np.float32)
    gamma = ties_elect(kept)
    k64 = kept.astype(np.float64)
    agree = (np.sign(k64) == gamma[None, :]) & (k64 != 0)
    cnt = agree.sum(axis=0)
    tot = np.where(agree, k64, 0.0).sum(axis=0)
    u = np.where(cnt > 0, tot / np.maximum(cnt, 1), 0.0)
    if not parts:
        return u
    pos, neg = k64 > 0, k64 < 0
    u_pos = np.where(pos, k64, 0.0).sum(axis=0) / np.maximum(pos.sum(axis=0), 1)
    u_neg = np.where(neg, k64, 0.0).sum(axis=0) / np.maximum(neg.sum(axis=0), 1)
    return {"update": u, "u_pos": u_pos, "u_neg": u_neg, "mass": k64.sum(axis=0),
            "abs_mass": np.abs(k64).sum(axis=0)}


def dare_mask(K: int, n: int, sparsity: float, seed: int, idx: np.ndarray | None = None) -> np.ndarray:
    """Kept entries [K, len(idx)] of task vectors of length n: u(k, i) >= p, u from
    SplitMix64 output k * n + i + 1 (idx: the entries, all by default)."""
    i = np.arange(n, dtype=np.uint64) if idx is None else np.asarray(idx, dtype=np.uint64)
    num = np.arange(K, dtype=np.uint64)[:, None] * np.uint64(n) + i[None, :] + np.uint64(1)
    z = splitmix64_array(int(seed) & 0xFFFFFFFF, num)
    u = (z >> np.uint64(40)).astype(np.float64) * 2.0 ** -24
    return u >= float(np.float32(sparsity))


def dare_merge(d: np.ndarray, sparsity: float, seed: int, reduce_mean: bool = True,
               n_total: int | None = None, idx: np.ndarray | None = None) -> np.ndarray:
    """DARE direction U in fp64 from fp32 task vectors d [K, len(idx)] (entries idx of task
    vectors of length n_total; all entries by default)."""
    K, n = d.shape
    p = float(np.float32(sparsity))
    m = dare_mask(K, n if n_total is None else n_total, sparsity, seed, idx)
    s = np.where(m, d.astype(np.float64), 0.0).sum(axis=0) / (1.0 - p)
    return s / K if reduce_mean else s


def merged_outer_step(theta, momentum, replicas, aggregator: str, sparsity: float = 0.0,
                      seed: int = 0, eta: float = 0.7, mu: float = 0.9, reduce_mean: bool = True):
    """Alg. 1's outer step with a merging aggregator ("ties" or "dare") in place of the
    mean.  Returns dict(theta, momentum, update) in fp64; for TIES also "ties_parts", the
    election's candidates and mass (``ties_merge(parts=True)``)."""
    d = task_vectors(theta, replicas)
    parts = None
    if aggregator == "ties":
        parts = ties_merge(d, sparsity, parts=True)
        u = parts["update"]
    elif aggregator == "dare":
        u = dare_merge(d, sparsity, seed, reduce_mean)
    else:
        raise ValueError(aggregator)
    th = np.asarray(theta, dtype=np.float32).astype(np.float64).ravel()
    b = np.asarray(momentum, dtype=np.float32).astype(np.float64).ravel()
    to, bo = nesterov(u, th, b, eta, mu)
    out = {"theta": to, "momentum": bo, "update": u}
    if parts is not None:
        out["ties_parts"] = parts
    return out
