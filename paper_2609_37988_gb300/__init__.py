"""GB300-native compressed-KV decode attention (KV-Kaizen, arxiv 2609.37988).

The product is ``libkvk.so`` (C ABI in ``include/kvk.h``): quantise/truncate
on write and split-K decode attention over per-layer compressed caches, as
hand-written sm_103a kernels.  ``cache.Cache`` is a thin PyTorch wrapper
(device memory and streams only); ``workloads`` draws seeded synthetic
inputs; ``build`` compiles the library.
"""
import importlib

__all__ = ["cache", "workloads", "build"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
