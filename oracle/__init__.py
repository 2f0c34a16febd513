"""CPU oracle for SONIQ's inference hot path (arXiv 2311.14114).

TEST INFRASTRUCTURE ONLY: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The library under
``paper_2311_14114_gb300`` never imports it and shares no code with it.

The arithmetic lives in ``soniq_oracle.c`` (plain C, fp32 code decisions in the
paper's operation order, exact int64 dot products, fp64 epilogue).  This module
compiles it with gcc on first use and wraps it for numpy arrays.  The final
fp64 -> fp16 rounding is numpy's ``astype(float16)`` (round to nearest even).

Every function here cites the passage of the paper it follows; the pins that
tie it to something other than itself are in ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import ctypes
import os
import platform
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "soniq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, f"liboracle_{platform.machine()}.so")
_lock = threading.Lock()
_lib = None

_i32p = ctypes.POINTER(ctypes.c_int32)


def build(force: bool = False) -> str:
    """Compile the C oracle into a shared object (gcc, -O2, no FP contraction)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, f32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_float
            lib.orc_act_group_codes.argtypes = [i32, i32]
            lib.orc_act_group_codes.restype = i64
            lib.orc_weight_group_codes.argtypes = [i32, i32, i32]
            lib.orc_weight_group_codes.restype = i64
            lib.orc_row_bytes.argtypes = [P, P, i32, i32, i32]
            lib.orc_row_bytes.restype = i64
            lib.orc_act_scales.argtypes = [P, i64, i32, P, P, i32, P]
            lib.orc_weight_scales.argtypes = [P, i32, i32, i32, P, P, i32, P]
            lib.orc_act_code.argtypes = [f32, f32, i32]
            lib.orc_act_code.restype = i32
            lib.orc_weight_code.argtypes = [f32, f32, i32]
            lib.orc_weight_code.restype = i32
            lib.orc_act_codes.argtypes = [P, i64, i32, P, P, P, P, i32, P]
            lib.orc_weight_codes.argtypes = [P, i32, i32, i32, P, P, P, P, P]
            lib.orc_pack_block.argtypes = [P, i32, P]
            lib.orc_unpack_block.argtypes = [P, i32, P]
            lib.orc_pack_act_rows.argtypes = [P, i64, i32, P, P, i32, P]
            lib.orc_pack_weight_rows.argtypes = [P, i32, i32, i32, P, P, i32, P]
            lib.orc_gemm_acc.argtypes = [P, i32, P, i32, P, P, i64, P]
            lib.orc_conv_acc.argtypes = [P, i32, i32, i32, i32, P, i32, i32, i32, i32, i32,
                                         i32, i32, P, P, i64, P]
            lib.orc_epilogue.argtypes = [P, P, i64, i32, P, i32, P, P, P, P]
            lib.orc_pm1_code.argtypes = [f32]
            lib.orc_pm1_code.restype = i32
            lib.orc_sub_scales.argtypes = [P, i64, i32, P, P, i32, i32, i32, P]
            lib.orc_codes_variant.argtypes = [P, i64, i32, P, P, P, P, i32, i32, P, i32, P]
            lib.orc_gemm_acc_runs.argtypes = [P, i32, P, i32, P, i32, i32, P, i64, P]
            lib.orc_epilogue_runs.argtypes = [P, P, i64, i32, i32, P, i32, P, P, P, P, P]
            _lib = lib
    return _lib


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a, a.ctypes.data_as(ctypes.c_void_p)


def _pair(x):
    x = list(x) + [0] * (2 - len(x))
    return np.array(x[:2], dtype=np.int32)


# --------------------------------------------------------------------------
# Layout sizes (Fig. 2 caption and Sec. 4.1: group by bit width, pad each
# block to the vector width; the pad amount is this library's reading).
# --------------------------------------------------------------------------

def act_group_codes(count: int, pad_unit: int) -> int:
    return int(_load().orc_act_group_codes(int(count), int(pad_unit)))


def weight_group_codes(count: int, pad_unit: int, taps: int = 1) -> int:
    return int(_load().orc_weight_group_codes(int(count), int(pad_unit), int(taps)))


def row_bytes(count, bits, pad_unit: int, taps: int = 1, is_weight: bool = False) -> int:
    c, cp = _c(_pair(count), np.int32)
    b, bp = _c(_pair(bits), np.int32)
    return int(_load().orc_row_bytes(cp, bp, int(pad_unit), int(taps), int(is_weight)))


# --------------------------------------------------------------------------
# a1: group-wise max-abs scales (Sec. 3, step 1).
# --------------------------------------------------------------------------

def act_scales(A, perm, count, per_row: bool = False) -> np.ndarray:
    A, Ap = _c(A, np.float32)
    M, K = A.shape
    perm, pp = _c(perm, np.int32)
    cnt, cp = _c(_pair(count), np.int32)
    s = np.zeros((M, 2) if per_row else (2,), dtype=np.float32)
    _load().orc_act_scales(Ap, M, K, pp, cp, int(per_row), s.ctypes.data_as(ctypes.c_void_p))
    return s


def weight_scales(W, perm, count, per_row: bool = True) -> np.ndarray:
    """W is [N][K] or [N][taps][K] (fp32)."""
    W = np.asarray(W, dtype=np.float32)
    if W.ndim == 2:
        W = W[:, None, :]
    W, Wp = _c(W, np.float32)
    N, taps, K = W.shape
    perm, pp = _c(perm, np.int32)
    cnt, cp = _c(_pair(count), np.int32)
    s = np.zeros((N, 2), dtype=np.float32)
    _load().orc_weight_scales(Wp, N, taps, K, pp, cp, int(per_row), s.ctypes.data_as(ctypes.c_void_p))
    return s


# --------------------------------------------------------------------------
# a3: codes (Sec. 3 steps 2 and 3, Eq. (1)).
# --------------------------------------------------------------------------

def act_code(a: float, s: float, n: int) -> int:
    return int(_load().orc_act_code(float(a), float(s), int(n)))


def weight_code(w: float, s: float, n: int) -> int:
    return int(_load().orc_weight_code(float(w), float(s), int(n)))


def act_codes(A, perm, count, bits, s, per_row: bool = False) -> np.ndarray:
    A, Ap = _c(A, np.float32)
    M, K = A.shape
    perm, pp = _c(perm, np.int32)
    cnt, cp = _c(_pair(count), np.int32)
    b, bp = _c(_pair(bits), np.int32)
    s, sp = _c(s, np.float32)
    U = np.zeros((M, K), dtype=np.uint8)
    _load().orc_act_codes(Ap, M, K, pp, cp, bp, sp, int(per_row), U.ctypes.data_as(ctypes.c_void_p))
    return U


def weight_codes(W, perm, count, bits, s) -> np.ndarray:
    """Returns J[N][taps][K] (int8) for W [N][K] or [N][taps][K]."""
    W = np.asarray(W, dtype=np.float32)
    squeeze = W.ndim == 2
    if squeeze:
        W = W[:, None, :]
    W, Wp = _c(W, np.float32)
    N, taps, K = W.shape
    perm, pp = _c(perm, np.int32)
    cnt, cp = _c(_pair(count), np.int32)
    b, bp = _c(_pair(bits), np.int32)
    s, sp = _c(s, np.float32)
    J = np.zeros((N, taps, K), dtype=np.int8)
    _load().orc_weight_codes(Wp, N, taps, K, pp, cp, bp, sp, J.ctypes.data_as(ctypes.c_void_p))
    return J[:, 0, :] if squeeze else J


# --------------------------------------------------------------------------
# a2: packing.
# --------------------------------------------------------------------------

def pack_block(codes, n: int) -> np.ndarray:
    codes, cp = _c(codes, np.uint32)
    assert codes.shape == (32,)
    words = np.zeros(n, dtype=np.uint32)
    _load().orc_pack_block(cp, int(n), words.ctypes.data_as(ctypes.c_void_p))
    return words


def unpack_block(words, n: int) -> np.ndarray:
    words, wp = _c(words, np.uint32)
    assert words.shape == (n,)
    codes = np.zeros(32, dtype=np.uint32)
    _load().orc_unpack_block(wp, int(n), codes.ctypes.data_as(ctypes.c_void_p))
    return codes


def pack_act_rows(U, count, bits, pad_unit: int) -> np.ndarray:
    U, Up = _c(U, np.uint8)
    M, K = U.shape
    cnt, cp = _c(_pair(count), np.int32)
    b, bp = _c(_pair(bits), np.int32)
    rb = row_bytes(count, bits, pad_unit, 1, False)
    out = np.zeros((M, rb), dtype=np.uint8)
    _load().orc_pack_act_rows(Up, M, K, cp, bp, int(pad_unit), out.ctypes.data_as(ctypes.c_void_p))
    return out


def pack_weight_rows(J, count, bits, pad_unit: int) -> np.ndarray:
    J = np.asarray(J, dtype=np.int8)
    if J.ndim == 2:
        J = J[:, None, :]
    J, Jp = _c(J, np.int8)
    N, taps, K = J.shape
    cnt, cp = _c(_pair(count), np.int32)
    b, bp = _c(_pair(bits), np.int32)
    rb = row_bytes(count, bits, pad_unit, taps, True)
    out = np.zeros((N, rb), dtype=np.uint8)
    _load().orc_pack_weight_rows(Jp, N, taps, K, cp, bp, int(pad_unit), out.ctypes.data_as(ctypes.c_void_p))
    return out


# --------------------------------------------------------------------------
# a4 / a7: exact integer accumulators per group.
# --------------------------------------------------------------------------

def gemm_acc(U, J, count, rows=None) -> np.ndarray:
    """acc[2][len(rows)][N] (int64) for codes U[M][K] (uint8) and J[N][K] (int8)."""
    U, Up = _c(U, np.uint8)
    J, Jp = _c(J, np.int8)
    M, K = U.shape
    N = J.shape[0]
    rows = np.arange(M, dtype=np.int64) if rows is None else np.asarray(rows, dtype=np.int64)
    rows, rp = _c(rows, np.int64)
    cnt, cp = _c(_pair(count), np.int32)
    acc = np.zeros((2, rows.shape[0], N), dtype=np.int64)
    _load().orc_gemm_acc(Up, K, Jp, N, cp, rp, rows.shape[0], acc.ctypes.data_as(ctypes.c_void_p))
    return acc


def conv_out_hw(H, W, R, S, stride=(1, 1), pad=(1, 1)):
    return (H + 2 * pad[0] - R) // stride[0] + 1, (W + 2 * pad[1] - S) // stride[1] + 1


def conv_acc(U, img_shape, J, count, R, S, stride=(1, 1), pad=(1, 1), pix=None) -> np.ndarray:
    """U: [Nimg*H*W][K] pixel codes (NHWC rows); J: [Cout][R*S][K].
    Returns acc[2][len(pix)][Cout] for output pixel indices pix (all if None)."""
    Nimg, H, Wd = img_shape
    U, Up = _c(U, np.uint8)
    J, Jp = _c(J, np.int8)
    K = U.shape[1]
    Cout = J.shape[0]
    P, Q = conv_out_hw(H, Wd, R, S, stride, pad)
    pix = np.arange(Nimg * P * Q, dtype=np.int64) if pix is None else np.asarray(pix, dtype=np.int64)
    pix, pp = _c(pix, np.int64)
    cnt, cp = _c(_pair(count), np.int32)
    acc = np.zeros((2, pix.shape[0], Cout), dtype=np.int64)
    _load().orc_conv_acc(Up, Nimg, H, Wd, K, Jp, Cout, R, S, stride[0], stride[1], pad[0], pad[1],
                         cp, pp, pix.shape[0], acc.ctypes.data_as(ctypes.c_void_p))
    return acc


# --------------------------------------------------------------------------
# a5: epilogue in fp64, then RN to fp16 (numpy).
# --------------------------------------------------------------------------

def epilogue(acc, s_a, s_w, bits_a, bits_w, rows=None, s_a_per_row: bool = False) -> np.ndarray:
    acc, accp = _c(acc, np.int64)
    n_rows, N = acc.shape[1], acc.shape[2]
    rows = np.arange(n_rows, dtype=np.int64) if rows is None else np.asarray(rows, dtype=np.int64)
    rows, rp = _c(rows, np.int64)
    s_a, sap = _c(s_a, np.float32)
    s_w, swp = _c(s_w, np.float32)
    ba, bap = _c(_pair(bits_a), np.int32)
    bw, bwp = _c(_pair(bits_w), np.int32)
    Y = np.zeros((n_rows, N), dtype=np.float64)
    _load().orc_epilogue(accp, rp, n_rows, N, sap, int(s_a_per_row), swp, bap, bwp,
                         Y.ctypes.data_as(ctypes.c_void_p))
    return Y


def epilogue_terms(acc, s_a, s_w, bits_a, bits_w, rows=None, s_a_per_row: bool = False) -> np.ndarray:
    """Sum over groups of |alpha_g * Acc_g| (fp64): the cancellation floor used by
    the output tolerance."""
    # every alpha_g is non-negative (max-abs scales over positive level counts),
    # so sum_g |alpha_g * Acc_g| is the epilogue applied to |Acc_g|.
    return epilogue(np.abs(np.asarray(acc, dtype=np.int64)), s_a, s_w, bits_a, bits_w,
                    rows=rows, s_a_per_row=s_a_per_row)


# --------------------------------------------------------------------------
# End-to-end helpers (the steps above in order).
# --------------------------------------------------------------------------

def linear(A, W, perm, count, bits_a, bits_w, pad_unit=128, act_mode="tensor",
           s_a=None, w_per_row=True, rows=None):
    """Quantized linear layer, all steps: returns a dict with scales, codes, packed
    rows, accumulators, fp64 Y and fp16 Y (for the given output rows)."""
    A32 = np.asarray(A, dtype=np.float32)
    per_row = act_mode == "row"
    if act_mode == "calibrated":
        s_a = np.asarray(s_a, dtype=np.float32)
    else:
        s_a = act_scales(A32, perm, count, per_row=per_row)
    s_w = weight_scales(W, perm, count, per_row=w_per_row)
    U = act_codes(A32, perm, count, bits_a, s_a, per_row=per_row)
    J = weight_codes(W, perm, count, bits_w, s_w)
    Ap = pack_act_rows(U, count, bits_a, pad_unit)
    Wp = pack_weight_rows(J, count, bits_w, pad_unit)
    acc = gemm_acc(U, J, count, rows=rows)
    Y = epilogue(acc, s_a, s_w, bits_a, bits_w, rows=rows, s_a_per_row=per_row)
    return dict(s_a=s_a, s_w=s_w, U=U, J=J, Ap=Ap, Wp=Wp, acc=acc, Y64=Y,
                Y16=Y.astype(np.float16))


def conv2d(X, W, perm, count, bits_a, bits_w, R, S, stride=(1, 1), pad=(1, 1), pad_unit=32,
           act_mode="tensor", s_a=None, w_per_row=True, pix=None):
    """Quantized conv (NHWC X [Nimg][H][W][C], OHWI W [Cout][R*S][C]) as the same
    steps with im2col addressing."""
    X32 = np.asarray(X, dtype=np.float32)
    Nimg, H, Wd, C = X32.shape
    rows = X32.reshape(Nimg * H * Wd, C)
    if act_mode == "calibrated":
        s_a = np.asarray(s_a, dtype=np.float32)
    else:
        s_a = act_scales(rows, perm, count, per_row=False)
    s_w = weight_scales(W, perm, count, per_row=w_per_row)
    U = act_codes(rows, perm, count, bits_a, s_a, per_row=False)
    J = weight_codes(W, perm, count, bits_w, s_w)
    Xp = pack_act_rows(U, count, bits_a, pad_unit)
    Wp = pack_weight_rows(J, count, bits_w, pad_unit)
    acc = conv_acc(U, (Nimg, H, Wd), J, count, R, S, stride, pad, pix=pix)
    Y = epilogue(acc, s_a, s_w, bits_a, bits_w)
    return dict(s_a=s_a, s_w=s_w, U=U, J=J, Xp=Xp, Wp=Wp, acc=acc, Y64=Y,
                Y16=Y.astype(np.float16))


# --------------------------------------------------------------------------
# f3: variants (signed activations, one-bit +-1 groups, scale sub-groups along
# K), linear layers.  kind[g]: 0 unsigned activations (default), 1 signed
# activations (Eq. (1)), 2 +-1 codes on both sides (one-bit groups).
# --------------------------------------------------------------------------

def n_runs(count, sub_k: int) -> int:
    """Scale runs per group array width: the larger group's run count."""
    c = _pair(count)
    if sub_k <= 0:
        return 1
    return int(max(1, max((int(x) + sub_k - 1) // sub_k for x in c)))


def pm1_code(x: float) -> int:
    return int(_load().orc_pm1_code(float(x)))


def sub_scales(X, perm, count, sub_k: int, per_row: bool) -> np.ndarray:
    X, Xp = _c(X, np.float32)
    M, K = X.shape
    perm, pp = _c(perm, np.int32)
    cnt, cp = _c(_pair(count), np.int32)
    nb = n_runs(count, sub_k)
    s = np.zeros(((M if per_row else 1), 2, nb), dtype=np.float32)
    _load().orc_sub_scales(Xp, M, K, pp, cp, int(sub_k), nb, int(per_row), s.ctypes.data_as(ctypes.c_void_p))
    return s


def codes_variant(X, perm, count, bits, kind, sub_k: int, s, per_row: bool) -> np.ndarray:
    X, Xp = _c(X, np.float32)
    M, K = X.shape
    perm, pp = _c(perm, np.int32)
    cnt, cp = _c(_pair(count), np.int32)
    b, bp = _c(_pair(bits), np.int32)
    kd, kp = _c(_pair(kind), np.int32)
    s, sp = _c(s, np.float32)
    C = np.zeros((M, K), dtype=np.int32)
    _load().orc_codes_variant(Xp, M, K, pp, cp, bp, kp, int(sub_k), int(s.shape[-1]), sp, int(per_row),
                              C.ctypes.data_as(ctypes.c_void_p))
    return C


def code_patterns(C, count, bits, kind) -> np.ndarray:
    """The stored n-bit patterns of codes C (packed order): two's complement for
    signed codes, bit (c + 1) / 2 for +-1 codes, the code itself otherwise."""
    C = np.asarray(C, dtype=np.int64)
    out = np.zeros(C.shape, dtype=np.uint8)
    c0 = int(_pair(count)[0])
    for g, sl in enumerate((slice(0, c0), slice(c0, C.shape[1]))):
        n, k = int(_pair(bits)[g]), int(_pair(kind)[g])
        x = C[:, sl]
        out[:, sl] = ((x + 1) // 2) if k == 2 else (x & ((1 << n) - 1))
    return out


def gemm_acc_runs(U, J, count, sub_k: int, rows=None) -> np.ndarray:
    """acc[2][nb][len(rows)][N] (int64)."""
    U, Up = _c(U, np.int32)
    J, Jp = _c(J, np.int32)
    M, K = U.shape
    N = J.shape[0]
    nb = n_runs(count, sub_k)
    rows = np.arange(M, dtype=np.int64) if rows is None else np.asarray(rows, dtype=np.int64)
    rows, rp = _c(rows, np.int64)
    cnt, cp = _c(_pair(count), np.int32)
    acc = np.zeros((2, nb, rows.shape[0], N), dtype=np.int64)
    _load().orc_gemm_acc_runs(Up, K, Jp, N, cp, int(sub_k), nb, rp, rows.shape[0],
                              acc.ctypes.data_as(ctypes.c_void_p))
    return acc


def epilogue_runs(acc, s_a, s_w, bits_a, bits_w, kind, rows=None, s_a_per_row: bool = False) -> np.ndarray:
    acc, accp = _c(acc, np.int64)
    nb, n_rows, N = acc.shape[1], acc.shape[2], acc.shape[3]
    rows = np.arange(n_rows, dtype=np.int64) if rows is None else np.asarray(rows, dtype=np.int64)
    rows, rp = _c(rows, np.int64)
    s_a, sap = _c(s_a, np.float32)
    s_w, swp = _c(s_w, np.float32)
    ba, bap = _c(_pair(bits_a), np.int32)
    bw, bwp = _c(_pair(bits_w), np.int32)
    kd, kp = _c(_pair(kind), np.int32)
    Y = np.zeros((n_rows, N), dtype=np.float64)
    _load().orc_epilogue_runs(accp, rp, n_rows, N, nb, sap, int(s_a_per_row), swp, bap, bwp, kp,
                              Y.ctypes.data_as(ctypes.c_void_p))
    return Y


def linear_variant(A, W, perm, count, bits_a, bits_w, kind=(0, 0), sub_k: int = 0, act_mode="tensor",
                   pad_unit: int = 128, rows=None):
    """A linear layer under the f3 variants, all steps: scales per run, codes,
    stored patterns, packed rows, run accumulators, fp64 and fp16 outputs.
    Weights always take Eq. (1) (or +-1 in kind-2 groups) with per-row scales."""
    A32 = np.asarray(A, dtype=np.float32)
    W32 = np.asarray(W, dtype=np.float32)
    per_row = act_mode == "row"
    s_a = sub_scales(A32, perm, count, sub_k, per_row)
    s_w = sub_scales(W32, perm, count, sub_k, True)
    U = codes_variant(A32, perm, count, bits_a, kind, sub_k, s_a, per_row)
    wkind = [2 if k == 2 else 1 for k in _pair(kind)]
    J = codes_variant(W32, perm, count, bits_w, wkind, sub_k, s_w, True)
    Ap = pack_act_rows(code_patterns(U, count, bits_a, kind), count, bits_a, pad_unit)
    Wp = pack_act_rows(code_patterns(J, count, bits_w, wkind), count, bits_w, pad_unit)
    acc = gemm_acc_runs(U, J, count, sub_k, rows=rows)
    Y = epilogue_runs(acc, s_a, s_w, bits_a, bits_w, kind, rows=rows, s_a_per_row=per_row)
    Yt = epilogue_runs(np.abs(acc), s_a, s_w, bits_a, bits_w, kind, rows=rows, s_a_per_row=per_row)
    return dict(s_a=s_a, s_w=s_w, U=U, J=J, Ap=Ap, Wp=Wp, acc=acc, Y64=Y, Y16=Y.astype(np.float16), terms=Yt)
