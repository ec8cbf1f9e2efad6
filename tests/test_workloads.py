"""Seeded synthetic inputs: shapes, sizes, determinism and the low-rank-plus-noise structure."""
import numpy as np
import torch

from paper_2607_03011_gb300 import workloads as W


def test_shape_sets_sizes():
    assert W.n_params(W.SPECS["llama_180m_k8"].shapes) == 219_701_248
    assert sum(1 for s in W.SPECS["llama_180m_k8"].shapes if s[2] > 0) == 86
    assert W.n_params(W.SPECS["llama_1b_k8"].shapes) == 1_364_295_680
    assert W.n_params(W.SPECS["llama_3b_k4"].shapes) == 3_367_673_856
    assert W.SPECS["llama_3b_k4"].replica_dtype == "bf16" and W.SPECS["llama_3b_k4"].K == 4
    t = W.param_table(W.SPECS["tiny"].shapes)
    assert t[0] == (0, 64, 64) and t[-1][2] == 0


def test_determinism_and_seeds():
    a = W.make_workload("tiny", seed=0)
    b = W.make_workload("tiny", seed=0)
    c = W.make_workload("tiny", seed=1)
    assert torch.equal(a.replicas, b.replicas) and torch.equal(a.theta, b.theta)
    assert not torch.equal(a.replicas, c.replicas)


def test_pseudo_gradient_structure():
    wl = W.make_workload("tiny", seed=0)
    spec = wl.spec
    off, r, c = wl.table[0]
    th = wl.theta[off:off + r * c].double().reshape(r, c)
    deltas = [th - wl.replicas[k, off:off + r * c].double().reshape(r, c) for k in range(wl.K)]
    # shared part: rank 4 with entries of std shared_std; noise: std noise_std per worker
    diff = (deltas[0] - deltas[1]).numpy()
    assert abs(diff.std() / (np.sqrt(2) * spec.noise_std) - 1) < 0.05
    mean = ((deltas[0] + deltas[1]) / 2).numpy()
    s = np.linalg.svd(mean, compute_uv=False)
    assert s[:4].min() > 3 * s[4]          # four dominant directions
    assert abs(wl.theta.std().item() / 0.02 - 1) < 0.05


def test_bf16_replicas():
    spec = W.custom_spec([("m", 16, 8), ("v", 8, 0)], K=3, replica_dtype="bf16")
    wl = W.make_workload(spec, seed=3)
    assert wl.replicas.dtype == torch.bfloat16 and wl.replicas.shape == (3, 136)
    reps = W.replicas_as_numpy(wl.replicas)
    assert reps[0].dtype == np.uint16
    back = (reps[0].astype(np.uint32) << 16).view(np.float32)
    np.testing.assert_array_equal(back, wl.replicas[0].float().numpy())
