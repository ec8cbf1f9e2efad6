"""Seeded synthetic workloads for the outer step: shape sets and input generators.

This module builds inputs only; it holds none of the outer step's arithmetic.
Both the CUDA path and the fp64 oracle read the tensors it returns.

Shape sets (parameter tables of LLaMA-style decoders, plus the tiny test set):

* ``tiny``: matrices 64x64, 64x256, 256x64, 128x64 and vectors of 64 and 256.
* ``llama_180m``: d_model 1024, 12 layers (Wq/Wk/Wv/Wo 1024x1024, SwiGLU
  W_gate/W_up 1024x2816 and W_down 2816x1024, two RMSNorm vectors of 1024),
  embedding and untied head 32000x1024 -- N = 219,701,248 parameters.
* ``llama_1b``: d_model 2048, 24 layers, SwiGLU 5632, vocabulary 32000.
* ``llama_3b``: d_model 3072, 28 layers, SwiGLU 8192, vocabulary 32000.

The paper trains "178M" LLaMA-2 style models (Sec. 3.1); the table here has an
untied head and no final norm, which is what the 219.7M count reflects.

Generator (per parameter of shape m x n; 1-D tensors use a shared vector):

    theta_global ~ N(0, 0.02^2)
    L   = A B^T * (s_shared / sqrt(r)),  A ~ N(0,1)^{m x r}, B ~ N(0,1)^{n x r}
    E_k ~ N(0, s_noise^2)  independently per worker k
    theta_k = round(theta_global - (L + E_k))   (fp32, or bf16 replicas)

so the per-worker pseudo-gradients theta_global - theta_k share a rank-r part
plus independent noise.  The momentum buffer is zero (tiny) or i.i.d.
N(0, s^2), a stand-in for the momentum carried from an earlier step.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import torch

# (name, rows, cols); cols == 0 marks a 1-D tensor of `rows` elements.
Shape = Tuple[str, int, int]


def llama_shapes(d_model: int, n_layers: int, d_ff: int, vocab: int = 32000) -> List[Shape]:
    shapes: List[Shape] = [("embed", vocab, d_model)]
    for layer in range(n_layers):
        p = f"layers.{layer}."
        shapes += [
            (p + "attn_norm", d_model, 0),
            (p + "wq", d_model, d_model),
            (p + "wk", d_model, d_model),
            (p + "wv", d_model, d_model),
            (p + "wo", d_model, d_model),
            (p + "ffn_norm", d_model, 0),
            (p + "w_gate", d_model, d_ff),
            (p + "w_up", d_model, d_ff),
            (p + "w_down", d_ff, d_model),
        ]
    shapes.append(("head", vocab, d_model))
    return shapes


def tiny_shapes() -> List[Shape]:
    return [("w0", 64, 64), ("w1", 64, 256), ("w2", 256, 64), ("w3", 128, 64),
            ("v0", 64, 0), ("v1", 256, 0)]


@dataclasses.dataclass(frozen=True)
class WorkloadSpec:
    name: str
    shapes: Tuple[Shape, ...]
    K: int
    rank: int
    shared_std: float          # std of the entries of the shared low-rank part
    noise_std: float           # std of each worker's independent noise
    momentum_std: float        # 0 -> zero momentum buffer
    replica_dtype: str = "f32"  # "f32" or "bf16"
    alpha: float = 1.0
    outer_lr: float = 0.7
    momentum: float = 0.9
    theta_std: float = 0.02


def _s(rel: float = 1e-3, theta_std: float = 0.02) -> float:
    return rel * theta_std


SPECS = {
    "tiny": WorkloadSpec("tiny", tuple(tiny_shapes()), K=2, rank=4, shared_std=1e-3,
                         noise_std=5e-4, momentum_std=0.0),
    "llama_180m_k8": WorkloadSpec("llama_180m_k8", tuple(llama_shapes(1024, 12, 2816)), K=8,
                                  rank=32, shared_std=_s(), noise_std=_s(), momentum_std=_s()),
    "llama_180m_k16": WorkloadSpec("llama_180m_k16", tuple(llama_shapes(1024, 12, 2816)), K=16,
                                   rank=32, shared_std=_s(), noise_std=_s(), momentum_std=_s()),
    "llama_1b_k8": WorkloadSpec("llama_1b_k8", tuple(llama_shapes(2048, 24, 5632)), K=8,
                                rank=32, shared_std=_s(), noise_std=_s(), momentum_std=_s()),
    "llama_3b_k4": WorkloadSpec("llama_3b_k4", tuple(llama_shapes(3072, 28, 8192)), K=4,
                                rank=64, shared_std=_s(), noise_std=_s(), momentum_std=_s(),
                                replica_dtype="bf16"),
}


def param_table(shapes: Sequence[Shape]) -> List[Tuple[int, int, int]]:
    """Dense flat layout: [(offset, rows, cols)] in order, no padding."""
    table, off = [], 0
    for _, r, c in shapes:
        table.append((off, r, c))
        off += r * (c if c > 0 else 1)
    return table


def n_params(shapes: Sequence[Shape]) -> int:
    return sum(r * (c if c > 0 else 1) for _, r, c in shapes)


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    table: List[Tuple[int, int, int]]
    theta: torch.Tensor        # [N] fp32
    momentum: torch.Tensor     # [N] fp32
    replicas: torch.Tensor     # [K, N] fp32 or bf16
    seed: int

    @property
    def N(self) -> int:
        return self.theta.numel()

    @property
    def K(self) -> int:
        return self.replicas.shape[0]


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _shared_part(spec: WorkloadSpec, table, device, g: torch.Generator) -> torch.Tensor:
    """Flat vector of the shared (rank-r) part of every parameter."""
    N = n_params(spec.shapes)
    out = torch.empty(N, dtype=torch.float32, device=device)
    for (off, r, c) in table:
        if c > 0:
            rk = min(spec.rank, r, c)
            a = torch.randn(r, rk, generator=g, device=device, dtype=torch.float32)
            b = torch.randn(c, rk, generator=g, device=device, dtype=torch.float32)
            out[off:off + r * c] = (a @ b.T).reshape(-1) * (spec.shared_std / math.sqrt(rk))
        else:
            out[off:off + r] = torch.randn(r, generator=g, device=device) * spec.shared_std
    return out


def make_replicas(spec: WorkloadSpec, table, theta: torch.Tensor, seed: int,
                  K: Optional[int] = None) -> torch.Tensor:
    """theta_k = theta - (shared + noise_k) for k = 0..K-1, rounded to the replica dtype."""
    device = theta.device
    K = spec.K if K is None else K
    g = _gen(device, seed * 7919 + 17)
    shared = _shared_part(spec, table, device, g)
    dt = torch.bfloat16 if spec.replica_dtype == "bf16" else torch.float32
    # rows padded to 64 elements so every replica starts 16-byte aligned
    n = theta.numel()
    reps = torch.empty((K, (n + 63) // 64 * 64), dtype=dt, device=device)[:, :n]
    for k in range(K):
        gk = _gen(device, seed * 1_000_003 + 1000 + k)
        noise = torch.randn(theta.numel(), generator=gk, device=device) * spec.noise_std
        reps[k] = (theta - (shared + noise)).to(dt)
        del noise
    return reps


def make_workload(name_or_spec, seed: int = 0, device="cpu", K: Optional[int] = None) -> Workload:
    spec = SPECS[name_or_spec] if isinstance(name_or_spec, str) else name_or_spec
    table = param_table(spec.shapes)
    N = n_params(spec.shapes)
    g = _gen(device, seed)
    theta = torch.randn(N, generator=g, device=device) * spec.theta_std
    if spec.momentum_std > 0:
        mom = torch.randn(N, generator=g, device=device) * spec.momentum_std
    else:
        mom = torch.zeros(N, device=device)
    reps = make_replicas(spec, table, theta, seed, K)
    return Workload(spec, table, theta, mom, reps, seed)


def custom_spec(shapes: Sequence[Shape], K: int, rank: int = 4, shared_std: float = 1e-3,
                noise_std: float = 5e-4, momentum_std: float = 0.0, replica_dtype: str = "f32",
                name: str = "custom", **hp) -> WorkloadSpec:
    return WorkloadSpec(name, tuple(shapes), K=K, rank=rank, shared_std=shared_std,
                        noise_std=noise_std, momentum_std=momentum_std,
                        replica_dtype=replica_dtype, **hp)


def replicas_as_numpy(replicas: torch.Tensor):
    """Host copies for the oracle: float32 arrays, or uint16 arrays of bf16 bits."""
    r = replicas.detach().cpu()
    if r.dtype == torch.bfloat16:
        return [x.view(torch.int16).numpy().view("uint16") for x in r]
    return [x.numpy() for x in r]
