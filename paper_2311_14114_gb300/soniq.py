"""ctypes binding of libsoniq.so (``include/soniq.h``).

Argument marshalling only: torch supplies device memory and the current CUDA
stream; every step of the quantize / pack / GEMM / conv path runs in the
library's CUDA kernels.  There is no fallback: if the library is missing or
no GPU is present the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libsoniq.so")

SONIQ_OK = 0
SONIQ_ERR_INVALID_ARG, SONIQ_ERR_UNSUPPORTED, SONIQ_ERR_ALIGNMENT, SONIQ_ERR_CUDA, SONIQ_ERR_TIMEOUT = 1, 2, 3, 4, 5
STATUS_NAMES = {0: "SONIQ_OK", 1: "SONIQ_ERR_INVALID_ARG", 2: "SONIQ_ERR_UNSUPPORTED",
                3: "SONIQ_ERR_ALIGNMENT", 4: "SONIQ_ERR_CUDA", 5: "SONIQ_ERR_TIMEOUT"}
SCALE_PER_TENSOR, SCALE_PER_ROW, SCALE_CALIBRATED = 0, 1, 2
OUT_F16, OUT_BF16 = 0, 1
FLAG_FORCE_GEMV, FLAG_FORCE_MMA, FLAG_FORCE_FUSED, FLAG_FORCE_STAGED = 1, 2, 4, 8
FLAG_FORCE_SKINNY, FLAG_TEST_DROP_ARRIVE = 16, 0x100
ACT_UNSIGNED, ACT_SIGNED, ACT_PM1 = 0, 1, 2
PATH_NAMES = {0: "CUDA-core GEMV", 1: "tensor-core fused kernel", 2: "tensor-core staged (expand + GEMM)",
              3: "tensor-core skinny (swap-AB)"}

EXPORTED = ["soniq_abi_version", "soniq_status_string", "soniq_group_codes",
            "soniq_packed_row_bytes", "soniq_scale_runs", "soniq_validate_layout", "soniq_launch_count",
            "soniq_pack_weights", "soniq_quantize_act", "soniq_quantize_act_scratch_bytes",
            "soniq_quantize_act_oneshot", "soniq_mp_gemm", "soniq_mp_gemm_path", "soniq_mp_gemm_scratch_bytes",
            "soniq_mp_conv2d", "soniq_mp_conv2d_scratch_bytes", "soniq_sync_status",
            "soniq_test_drop_barrier_arrival"]

_SCALE = {"tensor": SCALE_PER_TENSOR, "row": SCALE_PER_ROW, "calibrated": SCALE_CALIBRATED}


class SoniqError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}")


class CLayout(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("n_groups", ctypes.c_int32),
                ("count", ctypes.c_int32 * 2), ("bits_w", ctypes.c_int32 * 2),
                ("bits_a", ctypes.c_int32 * 2), ("perm", ctypes.c_void_p),
                ("pad_unit", ctypes.c_int32), ("act_kind", ctypes.c_int32 * 2), ("sub_k", ctypes.c_int32)]


class CNextLayer(ctypes.Structure):
    _fields_ = [("layout", ctypes.c_void_p), ("s_a", ctypes.c_void_p), ("Ap", ctypes.c_void_p)]


class CConvDesc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("H", ctypes.c_int32), ("W", ctypes.c_int32),
                ("C_out", ctypes.c_int32), ("R", ctypes.c_int32), ("S", ctypes.c_int32),
                ("stride_h", ctypes.c_int32), ("stride_w", ctypes.c_int32),
                ("pad_h", ctypes.c_int32), ("pad_w", ctypes.c_int32)]


_lib = None


def lib() -> ctypes.CDLL:
    """Loads libsoniq.so (built by ``paper_2311_14114_gb300.build``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libsoniq.so not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        P, i32, i64, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
        L.soniq_abi_version.restype = i32
        L.soniq_status_string.argtypes = [i32]
        L.soniq_status_string.restype = ctypes.c_char_p
        L.soniq_group_codes.argtypes = [P, i32, i32, i32]
        L.soniq_group_codes.restype = i64
        L.soniq_packed_row_bytes.argtypes = [P, i32, i32]
        L.soniq_packed_row_bytes.restype = i64
        L.soniq_scale_runs.argtypes = [P]
        L.soniq_scale_runs.restype = i32
        L.soniq_validate_layout.argtypes = [P, P]
        L.soniq_validate_layout.restype = i32
        L.soniq_launch_count.restype = i64
        L.soniq_pack_weights.argtypes = [P, P, i32, i32, i32, P, P, P]
        L.soniq_pack_weights.restype = i32
        L.soniq_quantize_act.argtypes = [P, P, i64, i32, P, P, P, ctypes.c_size_t, P]
        L.soniq_quantize_act.restype = i32
        L.soniq_quantize_act_scratch_bytes.argtypes = [P, i64, i32]
        L.soniq_quantize_act_scratch_bytes.restype = i64
        L.soniq_quantize_act_oneshot.argtypes = [P, P, i64, P, P, P]
        L.soniq_quantize_act_oneshot.restype = i32
        L.soniq_mp_gemm.argtypes = [P, P, P, i32, i64, P, P, i32, P, i32, P, u32, P, ctypes.c_size_t, P, P]
        L.soniq_mp_gemm.restype = i32
        L.soniq_mp_gemm_path.argtypes = [P, i64, i32, u32, ctypes.c_size_t]
        L.soniq_mp_gemm_path.restype = i32
        L.soniq_mp_gemm_scratch_bytes.argtypes = [P, i64, i32, u32]
        L.soniq_mp_gemm_scratch_bytes.restype = i64
        L.soniq_mp_conv2d.argtypes = [P, P, P, P, i32, P, P, P, i32, P, u32, P, ctypes.c_size_t, P, P]
        L.soniq_mp_conv2d.restype = i32
        L.soniq_mp_conv2d_scratch_bytes.argtypes = [P, P, u32]
        L.soniq_mp_conv2d_scratch_bytes.restype = i64
        L.soniq_sync_status.argtypes = [P]
        L.soniq_sync_status.restype = i32
        L.soniq_test_drop_barrier_arrival.argtypes = [i32]
        L.soniq_test_drop_barrier_arrival.restype = None
        _lib = L
    return _lib


def _check(status: int, where: str):
    if status != SONIQ_OK:
        raise SoniqError(status, where)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t: torch.Tensor, dtype, name: str):
    if not t.is_cuda or t.dtype != dtype or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA {dtype} tensor")


# Scratch buffers the binding hands to the library, one per (use, device,
# stream): calls on one stream run in order, so they may share it; calls on
# different streams get different buffers.  The quantize scratch (whose
# barrier must start at zero and which every completed call leaves zeroed) is
# never shared with the GEMM scratch (which the staged path overwrites).
# Each is zero-filled when created and grows by reallocation when a call
# needs more.
_scratch = {}


def _get_scratch(nbytes: int, device, stream, use: str) -> Optional[torch.Tensor]:
    if nbytes <= 0:
        return None
    s = torch.cuda.current_stream(device) if stream is None else stream
    key = (use, torch.device(device).index, s.cuda_stream)
    buf = _scratch.get(key)
    if buf is None or buf.numel() < nbytes:
        with torch.cuda.stream(s):
            buf = torch.zeros(((nbytes + 255) // 256) * 256, dtype=torch.uint8, device=device)
        _scratch[key] = buf
    return buf


def reset_scratch():
    """Zero every cached quantize scratch buffer (needed after a SONIQ_ERR_TIMEOUT)."""
    for key, buf in _scratch.items():
        if key[0] == "quantize":
            buf.zero_()


class Layout:
    """Per-layer precision layout: groups, bit widths, channel permutation.

    perm[j] is the original channel at packed position j; positions
    [0, count[0]) form the low-precision group 0.  The permutation is kept in
    device memory (the kernels gather through it).  act_kind (per group:
    ACT_UNSIGNED, ACT_SIGNED, ACT_PM1) and sub_k (scale runs along K) select
    the layout variants of soniq_layout."""

    def __init__(self, perm: Sequence[int], count: Sequence[int], bits_w: Sequence[int],
                 bits_a: Optional[Sequence[int]] = None, pad_unit: int = 128, device=None,
                 act_kind: Sequence[int] = (0, 0), sub_k: int = 0):
        bits_a = bits_w if bits_a is None else bits_a
        perm_t = torch.as_tensor(perm, dtype=torch.int32).contiguous()
        self.K = int(perm_t.numel())
        count = list(count) + [0] * (2 - len(count))
        self.count = [int(count[0]), int(count[1])]
        self.bits_w = [int(b) for b in list(bits_w)[:2]] + [1] * (2 - len(bits_w))
        self.bits_a = [int(b) for b in list(bits_a)[:2]] + [1] * (2 - len(bits_a))
        self.pad_unit = int(pad_unit)
        n_groups = 2 if self.count[1] > 0 else 1
        self.act_kind = [int(k) for k in list(act_kind)[:2]] + [0] * (2 - len(act_kind))
        self.sub_k = int(sub_k)
        host = CLayout(self.K, n_groups, (ctypes.c_int32 * 2)(*self.count),
                       (ctypes.c_int32 * 2)(*self.bits_w), (ctypes.c_int32 * 2)(*self.bits_a),
                       None, self.pad_unit, (ctypes.c_int32 * 2)(*self.act_kind), self.sub_k)
        _check(lib().soniq_validate_layout(ctypes.byref(host),
                                           perm_t.numpy().ctypes.data_as(ctypes.c_void_p)),
               "soniq_validate_layout")
        self.perm_host = perm_t.numpy().copy()
        self.perm = perm_t.to(device if device is not None else "cuda")
        host.perm = ctypes.c_void_p(self.perm.data_ptr())
        self.c = host

    def row_bytes(self, is_weight: bool = False, taps: int = 1) -> int:
        v = lib().soniq_packed_row_bytes(ctypes.byref(self.c), int(is_weight), int(taps))
        if v < 0:
            raise SoniqError(1, "soniq_packed_row_bytes")
        return int(v)

    def group_codes(self, g: int, is_weight: bool = False, taps: int = 1) -> int:
        return int(lib().soniq_group_codes(ctypes.byref(self.c), int(g), int(is_weight), int(taps)))

    def scale_runs(self) -> int:
        """Scale entries per (row, group): soniq_scale_runs."""
        return int(lib().soniq_scale_runs(ctypes.byref(self.c)))

    def scale_shape(self, rows: Optional[int]) -> tuple:
        """Shape of a scale array: [rows][2] or [2], with a run axis when sub_k > 0."""
        tail = (2,) if self.sub_k == 0 else (2, self.scale_runs())
        return tail if rows is None else (rows,) + tail


def next_layer_row_order(next_layout: Layout):
    """Row order of a layer whose epilogue quantizes for `next_layout`
    (soniq_next_layer): entry j is the output channel placed at column j, the
    next layer's packed position j, or -1 for a padding position (a zero row).
    Index bookkeeping on the host for the one-time arrangement of weights."""
    import numpy as np
    pa0 = next_layout.group_codes(0)
    pa1 = next_layout.group_codes(1)
    c0, c1 = next_layout.count
    order = np.full(pa0 + pa1, -1, dtype=np.int64)
    order[:c0] = next_layout.perm_host[:c0]
    order[pa0:pa0 + c1] = next_layout.perm_host[c0:c0 + c1]
    return order


class NextLayer:
    """The next layer's codes written by a GEMM / conv epilogue (soniq_next_layer)."""

    def __init__(self, layout: Layout, s_a: torch.Tensor, Ap: Optional[torch.Tensor] = None, M: Optional[int] = None):
        _need(s_a, torch.float32, "s_a")
        self.layout = layout
        self.s_a = s_a
        if Ap is None:
            Ap = torch.empty((M, layout.row_bytes(False)), dtype=torch.uint8, device=s_a.device)
        self.Ap = Ap
        self.c = CNextLayer(ctypes.cast(ctypes.byref(layout.c), ctypes.c_void_p), s_a.data_ptr(), Ap.data_ptr())


def pack_weights(layout: Layout, W: torch.Tensor, scale_mode: str = "row",
                 Wp: Optional[torch.Tensor] = None, s_w: Optional[torch.Tensor] = None,
                 stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """soniq_pack_weights.  W: fp32 [N][K] or [N][taps][K] on the GPU."""
    _need(W, torch.float32, "W")
    N = W.shape[0]
    taps = 1 if W.dim() == 2 else W.shape[1]
    if Wp is None:
        Wp = torch.empty((N, layout.row_bytes(True, taps)), dtype=torch.uint8, device=W.device)
    if s_w is None:
        s_w = torch.empty(layout.scale_shape(N), dtype=torch.float32, device=W.device)
    mode = {"row": SCALE_PER_ROW, "tensor": SCALE_PER_TENSOR}[scale_mode]
    _check(lib().soniq_pack_weights(ctypes.byref(layout.c), _ptr(W), N, taps, mode, _ptr(Wp),
                                    _ptr(s_w), _stream(stream)), "soniq_pack_weights")
    return Wp, s_w


def quantize_act(layout: Layout, A: torch.Tensor, scale_mode: str = "tensor",
                 s_a: Optional[torch.Tensor] = None, Ap: Optional[torch.Tensor] = None,
                 stream=None, scratch: Optional[torch.Tensor] = False) -> Tuple[torch.Tensor, torch.Tensor]:
    """soniq_quantize_act.  A: fp16 [M][K] on the GPU.  For scale_mode
    'calibrated', s_a ([2] fp32) is an input.  scratch: a zero-filled uint8
    CUDA tensor, None for no scratch (two-pass per-tensor path), or left out
    for the binding's per-stream buffer."""
    _need(A, torch.float16, "A")
    M = A.shape[0]
    mode = _SCALE[scale_mode]
    if s_a is None:
        if mode == SCALE_CALIBRATED:
            raise ValueError("calibrated mode needs s_a")
        s_a = torch.empty(layout.scale_shape(M if mode == SCALE_PER_ROW else None), dtype=torch.float32,
                          device=A.device)
    if Ap is None:
        Ap = torch.empty((M, layout.row_bytes(False)), dtype=torch.uint8, device=A.device)
    if scratch is False:
        need = int(lib().soniq_quantize_act_scratch_bytes(ctypes.byref(layout.c), M, mode))
        scratch = _get_scratch(need, A.device, stream, "quantize")
    nbytes = 0 if scratch is None else scratch.numel() * scratch.element_size()
    _check(lib().soniq_quantize_act(ctypes.byref(layout.c), _ptr(A), M, mode, _ptr(s_a), _ptr(Ap),
                                    _ptr(scratch), nbytes, _stream(stream)), "soniq_quantize_act")
    return Ap, s_a


def quantize_act_oneshot(layout: Layout, A: torch.Tensor, s_a: Optional[torch.Tensor] = None,
                         Ap: Optional[torch.Tensor] = None, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """soniq_quantize_act_oneshot: per-tensor quantize with fixed library scratch
    (no allocation, no two-pass fallback; oversize inputs raise)."""
    _need(A, torch.float16, "A")
    M = A.shape[0]
    if s_a is None:
        s_a = torch.empty((2,), dtype=torch.float32, device=A.device)
    if Ap is None:
        Ap = torch.empty((M, layout.row_bytes(False)), dtype=torch.uint8, device=A.device)
    _check(lib().soniq_quantize_act_oneshot(ctypes.byref(layout.c), _ptr(A), M, _ptr(s_a), _ptr(Ap),
                                            _stream(stream)), "soniq_quantize_act_oneshot")
    return Ap, s_a


def mp_gemm(layout: Layout, Ap: torch.Tensor, s_a: torch.Tensor, Wp: torch.Tensor,
            s_w: torch.Tensor, scale_mode: str = "tensor", out_dtype=torch.float16,
            Y: Optional[torch.Tensor] = None, acc_dbg: Optional[torch.Tensor] = None,
            flags: int = 0, stream=None, next: Optional[NextLayer] = None,
            write_y: bool = True) -> torch.Tensor:
    """soniq_mp_gemm: Y[M][N] = dequantized (A W^T) from packed codes; with
    `next`, the epilogue also writes the next layer's packed codes (next.Ap)."""
    M, N = Ap.shape[0], Wp.shape[0]
    if Y is None and write_y:
        Y = torch.empty((M, N), dtype=out_dtype, device=Ap.device)
    od = OUT_BF16 if (Y is not None and Y.dtype == torch.bfloat16) or (Y is None and out_dtype == torch.bfloat16) \
        else OUT_F16
    qflags = int(flags) | (FLAG_FORCE_STAGED if next is not None else 0)
    need = int(lib().soniq_mp_gemm_scratch_bytes(ctypes.byref(layout.c), M, N, qflags))
    scratch = _get_scratch(need, Ap.device, stream, "gemm")
    _check(lib().soniq_mp_gemm(ctypes.byref(layout.c), _ptr(Ap), _ptr(s_a), _SCALE[scale_mode], M,
                               _ptr(Wp), _ptr(s_w), N, _ptr(Y), od, _ptr(acc_dbg), int(flags),
                               _ptr(scratch), max(need, 0),
                               ctypes.byref(next.c) if next is not None else None, _stream(stream)),
           "soniq_mp_gemm")
    return Y


def gemm_path(layout: Layout, M: int, N: int, flags: int = 0) -> str:
    """soniq_mp_gemm_path: the kernel soniq_mp_gemm runs for these arguments."""
    need = max(int(lib().soniq_mp_gemm_scratch_bytes(ctypes.byref(layout.c), M, N, int(flags))), 0)
    p = int(lib().soniq_mp_gemm_path(ctypes.byref(layout.c), M, N, int(flags), need))
    if p < 0:
        raise SoniqError(SONIQ_ERR_INVALID_ARG, "soniq_mp_gemm_path")
    return PATH_NAMES.get(p, str(p))


def conv_desc(batch, H, W, C_out, R=3, S=3, stride=(1, 1), pad=(1, 1)) -> CConvDesc:
    return CConvDesc(batch, H, W, C_out, R, S, stride[0], stride[1], pad[0], pad[1])


def conv_out_hw(cd: CConvDesc) -> Tuple[int, int]:
    P = (cd.H + 2 * cd.pad_h - cd.R) // cd.stride_h + 1
    Q = (cd.W + 2 * cd.pad_w - cd.S) // cd.stride_w + 1
    return P, Q


def mp_conv2d(layout: Layout, cd: CConvDesc, Xp: torch.Tensor, s_a: torch.Tensor,
              Wp: torch.Tensor, s_w: torch.Tensor, scale_mode: str = "tensor",
              out_dtype=torch.float16, Y: Optional[torch.Tensor] = None,
              acc_dbg: Optional[torch.Tensor] = None, flags: int = 0, stream=None,
              next: Optional[NextLayer] = None, write_y: bool = True) -> torch.Tensor:
    """soniq_mp_conv2d: NHWC implicit-GEMM convolution from packed codes; with
    `next`, the epilogue also writes the next layer's packed codes."""
    P, Q = conv_out_hw(cd)
    if Y is None and write_y:
        Y = torch.empty((cd.batch, P, Q, cd.C_out), dtype=out_dtype, device=Xp.device)
    od = OUT_BF16 if (Y is not None and Y.dtype == torch.bfloat16) or (Y is None and out_dtype == torch.bfloat16) \
        else OUT_F16
    qflags = int(flags) | (FLAG_FORCE_STAGED if next is not None else 0)
    need = int(lib().soniq_mp_conv2d_scratch_bytes(ctypes.byref(layout.c), ctypes.byref(cd), qflags))
    scratch = _get_scratch(need, Xp.device, stream, "gemm")
    _check(lib().soniq_mp_conv2d(ctypes.byref(layout.c), ctypes.byref(cd), _ptr(Xp), _ptr(s_a),
                                 _SCALE[scale_mode], _ptr(Wp), _ptr(s_w), _ptr(Y), od,
                                 _ptr(acc_dbg), int(flags), _ptr(scratch), max(need, 0),
                                 ctypes.byref(next.c) if next is not None else None,
                                 _stream(stream)), "soniq_mp_conv2d")
    return Y


def sync_status(stream=None) -> int:
    """soniq_sync_status: waits for the stream, returns the status code.  After
    a timeout the binding's scratch buffers are zeroed again (the contract of
    the scratch-taking calls)."""
    st = int(lib().soniq_sync_status(_stream(stream)))
    if st == SONIQ_ERR_TIMEOUT:
        torch.cuda.synchronize()
        reset_scratch()
        torch.cuda.synchronize()
    return st


def test_drop_barrier_arrival(armed: bool = True):
    """soniq_test_drop_barrier_arrival (test hook)."""
    lib().soniq_test_drop_barrier_arrival(1 if armed else 0)


def launch_count() -> int:
    return int(lib().soniq_launch_count())
