"""Pins for the merging-aggregator oracle (oracle/merging.py, Sec. 3.2), CPU only.

TIES is pinned by a hand-worked example (trim, election and disjoint mean each change
its answer if dropped), an election that follows mass and not the count of workers, the
rule for magnitudes tied at the threshold, and its reduction to the plain mean when
nothing is trimmed and every worker agrees in sign.  DARE is pinned by the published
SplitMix64 outputs, its reduction to Alg. 1 at p = 0, its drop rate and the unbiasedness
of the rescale.
"""
import numpy as np
import pytest

import oracle
from oracle import merging


def test_splitmix64_known_answers():
    """First outputs of SplitMix64 from state 0, as listed with the generator's reference
    implementation (Steele, Lea and Flood 2014; Vigna's splitmix64.c)."""
    assert [merging.splitmix64(0, n) for n in (1, 2, 3)] == [
        0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    arr = merging.splitmix64_array(0, np.array([1, 2, 3], dtype=np.uint64))
    assert [int(x) for x in arr] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_splitmix64_array_matches_scalar():
    n = np.array([1, 7, 2**40 + 3, 2**63 - 1], dtype=np.uint64)
    arr = merging.splitmix64_array(12345, n)
    assert [int(x) for x in arr] == [merging.splitmix64(12345, int(v)) for v in n]


def _reps_from_deltas(d, theta=None):
    d = np.asarray(d, dtype=np.float32)
    th = np.zeros(d.shape[1], np.float32) if theta is None else np.asarray(theta, np.float32)
    return th, [(th - dk).astype(np.float32) for dk in d]


def test_ties_hand_worked():
    """K = 3, N = 4, sparsity 0.25 -> each worker keeps 3 entries.
    worker 0: [1, -2, 3, 0.5] -> [1, -2, 3, 0]; worker 1: [2, 1, -1, 0.1] -> [2, 1, -1, 0];
    worker 2: [-1, 3, 2, -0.2] -> [-1, 3, 2, 0].
    entry 0: 1 + 2 - 1 > 0 -> mean(1, 2) = 1.5; entry 1: -2 + 1 + 3 > 0 -> mean(1, 3) = 2;
    entry 2: 3 - 1 + 2 > 0 -> mean(3, 2) = 2.5; entry 3: nothing kept -> 0."""
    d = [[1, -2, 3, 0.5], [2, 1, -1, 0.1], [-1, 3, 2, -0.2]]
    th, reps = _reps_from_deltas(d)
    out = merging.merged_outer_step(th, np.zeros(4, np.float32), reps, "ties", sparsity=0.25, eta=1.0, mu=0.0)
    assert np.allclose(out["update"], [1.5, 2.0, 2.5, 0.0], rtol=0, atol=1e-15)
    assert np.allclose(out["theta"], [-1.5, -2.0, -2.5, 0.0], rtol=0, atol=1e-15)


def test_ties_elects_by_mass_not_count():
    """One large positive against two small negatives: the positive mass wins."""
    d = merging.task_vectors(*_reps_from_deltas([[3.0], [-1.0], [-1.0]]))
    assert merging.ties_merge(d, 0.0)[0] == 3.0
    d = merging.task_vectors(*_reps_from_deltas([[1.0], [-1.5], [-1.0]]))
    assert merging.ties_merge(d, 0.0)[0] == -1.25


def test_ties_exact_cancellation_gives_zero():
    d = merging.task_vectors(*_reps_from_deltas([[2.0, 1.0], [-2.0, 1.0]]))
    assert list(merging.ties_merge(d, 0.0)) == [0.0, 1.0]


def test_ties_election_is_exact_and_order_free():
    """The election is the sign of the exact kept mass.  [2^60, 1, -2^60] sums to 1 > 0,
    which an fp64 sum in this order misses (2^60 + 1 rounds to 2^60) and an fp32 running
    sum misses too; [1, 2^-30, -1] sums to 2^-30 > 0, lost by an fp32 running sum.  Every
    worker order gives the same sign and the same disjoint mean."""
    import itertools
    for col, want_sign in (([2.0 ** 60, 1.0, -(2.0 ** 60)], 1.0), ([1.0, 2.0 ** -30, -1.0], 1.0),
                           ([-(2.0 ** 60), -1.0, 2.0 ** 60], -1.0), ([3.0, -1.0, -2.0], 0.0)):
        for perm in itertools.permutations(col):
            kept = np.array(perm, np.float32)[:, None]
            assert merging.ties_elect(kept)[0] == want_sign
            u = merging.ties_merge(kept, 0.0)[0]
            pos = [x for x in col if x > 0]
            neg = [x for x in col if x < 0]
            want = np.mean(pos) if want_sign > 0 else (np.mean(neg) if want_sign < 0 else 0.0)
            assert u == want
    # fp32 running sums in worker order would elect 0 for the second column
    assert np.float32(np.float32(1.0) + np.float32(2.0 ** -30)) - np.float32(1.0) == 0.0


def test_ties_parts_hold_both_candidates():
    d = np.array([[1.0, -2.0, 0.5], [3.0, 1.0, -0.5], [-1.0, -4.0, 0.0]], np.float32)
    p = merging.ties_merge(d, 0.0, parts=True)
    assert np.allclose(p["u_pos"], [2.0, 1.0, 0.5]) and np.allclose(p["u_neg"], [-1.0, -3.0, -0.5])
    assert np.allclose(p["mass"], [3.0, -5.0, 0.0]) and np.allclose(p["abs_mass"], [5.0, 7.0, 1.0])
    assert list(p["update"]) == [2.0, -3.0, 0.0]


def test_ties_keeps_ties_at_threshold():
    """n_keep = 3 of [2, -2, 1, -1]: the 3rd largest magnitude is 1, so all four stay."""
    d = merging.task_vectors(*_reps_from_deltas([[2.0, -2.0, 1.0, -1.0]]))
    mask, thr = merging.ties_trim(d, 0.25)
    assert thr[0] == 1.0 and mask.all()
    assert list(merging.ties_merge(d, 0.25)) == [2.0, -2.0, 1.0, -1.0]


@pytest.mark.parametrize("n,s,keep", [(4, 0.25, 3), (10, 0.1, 9), (10, 0.95, 1), (7, 0.0, 7), (1000, 0.5, 500)])
def test_ties_keep_count(n, s, keep):
    assert merging.ties_keep_count(n, s) == keep
    d = np.random.default_rng(n).standard_normal((2, n)).astype(np.float32)
    mask, _ = merging.ties_trim(d, s)
    assert list(mask.sum(axis=1)) == [keep, keep]          # distinct magnitudes
    # the kept ones are the largest
    for k in range(2):
        assert np.abs(d[k][mask[k]]).min() >= np.abs(d[k][~mask[k]]).max(initial=0)


def test_ties_without_trim_and_agreeing_signs_is_the_mean():
    rng = np.random.default_rng(3)
    th = (0.02 * rng.standard_normal(500)).astype(np.float32)
    sign = np.where(rng.random(500) < 0.5, -1.0, 1.0)
    reps = [(th - sign * (1e-3 + 1e-3 * rng.random(500))).astype(np.float32) for _ in range(4)]
    mom = (1e-4 * rng.standard_normal(500)).astype(np.float32)
    ties = merging.merged_outer_step(th, mom, reps, "ties", sparsity=0.0)
    dil = oracle.diloco_outer_step(th, mom, reps, eta=0.7, mu=0.9)
    # Delta_k is taken in fp32 here (the precision of the trim and sign decisions) and
    # exactly in the Alg. 1 oracle: one fp32 rounding of a 1e-3 difference apart
    assert np.abs(ties["theta"] - dil["theta"]).max() < 1e-9
    assert np.abs(ties["momentum"] - dil["momentum"]).max() < 1e-9


def test_dare_p0_is_alg1():
    rng = np.random.default_rng(5)
    th = (0.02 * rng.standard_normal(333)).astype(np.float32)
    reps = [(th - 1e-3 * rng.standard_normal(333)).astype(np.float32) for _ in range(3)]
    mom = (1e-4 * rng.standard_normal(333)).astype(np.float32)
    for mean in (True, False):
        dare = merging.merged_outer_step(th, mom, reps, "dare", sparsity=0.0, seed=9, reduce_mean=mean)
        dil = oracle.diloco_outer_step(th, mom, reps, eta=0.7, mu=0.9, reduce_mean=mean)
        assert np.abs(dare["theta"] - dil["theta"]).max() < 3e-9
        assert np.abs(dare["momentum"] - dil["momentum"]).max() < 3e-9


@pytest.mark.parametrize("p", [0.1, 0.5, 0.9])
def test_dare_drop_rate_and_unbiased_rescale(p):
    K, n = 4, 50_000
    m = merging.dare_mask(K, n, p, seed=77)
    rate = 1.0 - m.mean()
    assert abs(rate - p) < 5 * np.sqrt(p * (1 - p) / (K * n))
    # a constant task vector c: E[U] = c
    d = np.full((K, n), 0.5, np.float32)
    u = merging.dare_merge(d, p, seed=77)
    assert abs(u.mean() - 0.5) < 5 * 0.5 * np.sqrt(p / ((1 - p) * K * n))
    # each U is c * (kept count) / (K (1 - p))
    assert np.allclose(u, 0.5 * m.sum(axis=0) / (K * (1 - float(np.float32(p)))), rtol=1e-15)


def test_dare_mask_depends_on_seed_worker_and_entry():
    a = merging.dare_mask(2, 4096, 0.5, seed=1)
    b = merging.dare_mask(2, 4096, 0.5, seed=2)
    assert (a != b).mean() > 0.4
    assert (a[0] != a[1]).mean() > 0.4
    # entry i of worker k uses output number k * N + i + 1
    z = merging.splitmix64(1, 1 * 4096 + 10 + 1)
    assert a[1, 10] == ((z >> 40) * 2.0 ** -24 >= 0.5)
