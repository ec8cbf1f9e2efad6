"""Workspace bounds check (stands in for a memory checker): every region of a plan's
device workspace sits between guard bytes (isoloco_check_guards).  After steps on ragged
shapes, split-K Grams, bf16 replicas, every variant (fast, clip, exact SVD, ablations), the
merging aggregators, the merge and the host-buffer entry point, no kernel has written past
either end of any region.  A planted change of one guard byte on the host is caught."""
import pytest
import torch

from paper_2607_03011_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SHAPES = [("a", 65, 130), ("b", 130, 65), ("c", 1, 9), ("h", 300, 257), ("i", 257, 300), ("j", 129, 129),
          ("e", 200, 3), ("f", 3, 200), ("t", 4100, 72), ("v", 7, 0), ("w", 3, 0)]


@pytest.fixture(scope="module")
def iso():
    from paper_2607_03011_gb300 import isoloco
    isoloco.lib()
    return isoloco


def guards_ok(iso, plan):
    rc = plan.check_guards()
    assert rc == 0, iso.last_error()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_guards_after_every_variant(iso, dtype):
    spec = W.custom_spec(SHAPES, K=3, rank=2, replica_dtype=dtype, momentum_std=1e-4)
    wl = W.make_workload(spec, seed=41, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K, wl.replicas.dtype)
    variants = [{}, {"fast_steps": 5}, {"spectrum_kind": 1}, {"spectrum_kind": 2}, {"spectrum_kind": 3},
                {"orth_target": 1}, {"momentum_kind": 1}, {"scale_kind": 1}, {"full_precision": 1},
                {"precision_schedule": -1}, {"reduce_mean": False}]
    for kw in variants:
        th, b = wl.theta.clone(), wl.momentum.clone()
        upd = torch.empty_like(th)
        assert plan.outer_step(th, b, wl.replicas, iso.make_opts(sync=True, **kw), update_out=upd) == 0, kw
        guards_ok(iso, plan)
    for agg in (0, 1, 2):
        th, b = wl.theta.clone(), wl.momentum.clone()
        assert plan.diloco_outer_step(th, b, wl.replicas, iso.make_opts(sync=True, aggregator=agg,
                                                                        sparsity=0.3, seed=2)) == 0
        guards_ok(iso, plan)
    out = torch.empty_like(wl.theta)
    plan.iso_c_merge(wl.theta, wl.replicas, 0.7, out)
    torch.cuda.synchronize()
    guards_ok(iso, plan)
    if dtype == "f32":
        th_h = wl.theta.cpu().pin_memory()
        b_h = wl.momentum.cpu().pin_memory()
        reps_h = [wl.replicas[k].cpu().pin_memory() for k in range(wl.K)]
        assert plan.outer_step_host(th_h, b_h, reps_h, iso.make_opts()) == 0
        guards_ok(iso, plan)


def test_guards_at_full_size(iso):
    """The benchmarked 180M, K = 8 step (every bucket, split-K embedding Grams) and its
    exact-SVD variant."""
    wl = W.make_workload("llama_180m_k8", seed=0, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    for kw in ({}, {"spectrum_kind": 3}):
        th, b = wl.theta.clone(), wl.momentum.clone()
        assert plan.outer_step(th, b, wl.replicas, iso.make_opts(sync=True, **kw)) == 0
        guards_ok(iso, plan)
    del wl, plan
    torch.cuda.empty_cache()


def test_planted_guard_change_is_caught(iso):
    spec = W.custom_spec([("m", 64, 48), ("v", 16, 0)], K=2)
    wl = W.make_workload(spec, seed=1, device="cuda")
    plan = iso.Plan(wl.table, wl.N, wl.K)
    th, b = wl.theta.clone(), wl.momentum.clone()
    assert plan.outer_step(th, b, wl.replicas, iso.make_opts(sync=True)) == 0
    guards_ok(iso, plan)
    for region, after in ((0, 1), (3, 0)):
        p2 = iso.Plan(wl.table, wl.N, wl.K)
        assert iso.lib().isoloco_debug_touch_guard(p2._h, region, after) == 0
        assert p2.check_guards() == iso.ERR_GUARD
        assert ("past its end" if after else "before its start") in iso.last_error()
        p2.close()
