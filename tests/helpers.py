"""Shared test helpers: tolerance of the fp16 outputs and small adapters that
run one workload through the CUDA path (C-ABI) and through the oracle."""
import numpy as np

import oracle


def y_tolerance(y_ref64: np.ndarray, terms64: np.ndarray) -> np.ndarray:
    """Allowed |y_gpu - y_ref| per element.

    The kernels sum sum_g alpha_g * Acc_g in fp32 and round once to fp16; the
    reference rounds the fp64 value once.  The two can land on neighbouring
    fp16 values (<= 1 ulp <= 2^-10 |y|, below 1e-3 relative) and fp32 adds
    ~2^-23 of the summed magnitudes; where terms cancel, the floor
    1e-3 * 2^-10 * sum_g |alpha_g Acc_g| covers that, and 2^-24 covers the
    fp16 subnormal spacing."""
    return 1e-3 * np.maximum(np.abs(y_ref64), terms64 * 2.0 ** -10) + 2.0 ** -24


def assert_y_close(y_gpu, ref, terms, what=""):
    y = np.asarray(y_gpu, dtype=np.float64)
    y_ref = np.asarray(ref["Y16"], dtype=np.float64) if isinstance(ref, dict) else np.asarray(ref, np.float64)
    tol = y_tolerance(y_ref, terms)
    err = np.abs(y - y_ref)
    bad = err > tol
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outputs outside tolerance; "
                           f"max err {err.max():.3e} at {np.unravel_index(err.argmax(), err.shape)}")


def fp16_ulp_diff(a16, b16) -> int:
    """Largest distance in fp16 units in the last place between two fp16 arrays."""
    a = np.asarray(a16, dtype=np.float16).view(np.int16).astype(np.int64)
    b = np.asarray(b16, dtype=np.float16).view(np.int16).astype(np.int64)
    # map sign-magnitude to a monotone integer line
    a = np.where(a < 0, -(a & 0x7FFF), a)
    b = np.where(b < 0, -(b & 0x7FFF), b)
    return int(np.abs(a - b).max()) if a.size else 0
