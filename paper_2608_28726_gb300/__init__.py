"""GB300 (sm_103a) data path of the Pro-Router token-aware verifier.

The compute lives in ``libprorouter.so`` (hand-written CUDA kernels behind a
C ABI, declared in ``include/pro_router.h``); ``binding`` is a thin ctypes
layer with the same call names, and ``workloads`` draws seeded synthetic
inputs.  Importing this package loads nothing; ``binding`` fails loudly when
the library has not been built.
"""
__all__ = ["binding", "workloads"]
