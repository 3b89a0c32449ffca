"""GB300 (sm_103a) implementation of memoized DNN mutation testing.

The method: Ghanbari, Greenman, Tavakkol, Ahmed, "Provably Lossless Acceleration of
DNN Mutation Testing via Memoization" (PACMSE/ISSTA 2026), Algorithm 1.

  mure            ctypes binding of the CUDA library (include/mure.h)
  workloads       seeded synthetic networks, inputs and mutant tables
  build           nvcc build of the library
"""
from . import workloads  # noqa: F401  (pure numpy, no library load)

__all__ = ["workloads", "mure", "build"]


def __getattr__(name):
    if name in ("mure", "build"):
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
