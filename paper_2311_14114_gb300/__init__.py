"""GB300-native (sm_103a) implementation of SONIQ's inference hot path
(arXiv 2311.14114): per-channel two-level mixed-precision quantized matmul,
GEMV and implicit-GEMM convolution behind a C-ABI library (``include/soniq.h``).

``paper_2311_14114_gb300.soniq`` is the thin ctypes binding over
``libsoniq.so``; ``paper_2311_14114_gb300.workloads`` draws seeded synthetic
inputs.  Importing this package does not load the CUDA library; the binding
loads it on first use and raises if it is missing.
"""

__all__ = ["soniq", "workloads"]


def __getattr__(name):
    if name in __all__:
        import importlib
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
