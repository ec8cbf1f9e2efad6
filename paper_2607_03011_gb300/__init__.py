"""GB300-native IsoLoCo / DiLoCo outer step (arXiv 2607.03011).

The outer step of IsoLoCo (Alg. 2) and DiLoCo (Alg. 1) on one GB300: K worker
replicas resident in HBM, a K-way pseudo-gradient reduction, Iso-C on every
2-D tensor through a batched Newton-Schulz-type polar factor on tcgen05 tensor
cores, and a fused Nesterov update.  The compute runs in the hand-written CUDA
library ``libisoloco`` behind the C ABI declared in ``include/isoloco.h``;
``paper_2607_03011_gb300.isoloco`` is the thin Python binding over it.

Importing this package loads nothing; the CUDA library is opened on first use
and its absence is an error (there is no CPU fallback).
"""

__all__ = ["isoloco", "workloads"]


def __getattr__(name):
    if name in __all__:
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
