"""The C-ABI library: it loads without a GPU, exports every symbol that
include/soniq.h declares, and rejects bad arguments on the host before any
CUDA call (so these run on CPU)."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    from paper_2311_14114_gb300 import build
    build.build()
    from paper_2311_14114_gb300 import soniq
    return soniq.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "soniq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(soniq_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_four_hot_path_calls():
    names = declared_functions()
    for f in ("soniq_pack_weights", "soniq_quantize_act", "soniq_mp_gemm", "soniq_mp_conv2d"):
        assert f in names


def test_library_exports_every_declared_symbol(L):
    from paper_2311_14114_gb300 import soniq
    names = declared_functions()
    for name in names:
        assert hasattr(L, name), name
    assert sorted(soniq.EXPORTED) == names
    assert L.soniq_abi_version() == 3


def _layout(soniq, K=300, count=(200, 100), bits=(3, 8), pad=128, perm=None, act_kind=(0, 0), sub_k=0):
    c = soniq.CLayout()
    c.act_kind[0], c.act_kind[1] = act_kind
    c.sub_k = sub_k
    c.K = K
    c.n_groups = 2 if count[1] else 1
    c.count[0], c.count[1] = count
    c.bits_w[0], c.bits_w[1] = bits
    c.bits_a[0], c.bits_a[1] = bits
    c.perm = perm
    c.pad_unit = pad
    return c


def test_row_bytes_match_oracle(L):
    from paper_2311_14114_gb300 import soniq
    rng = np.random.default_rng(0)
    for _ in range(40):
        K = int(rng.integers(1, 5000))
        c1 = int(rng.integers(0, K + 1))
        bits = [int(rng.integers(1, 9)), int(rng.integers(1, 9))]
        pad = int(rng.choice([32, 128]))
        taps = int(rng.choice([1, 9, 25]))
        lay = _layout(soniq, K, (K - c1, c1), bits, pad)
        for w in (0, 1):
            got = L.soniq_packed_row_bytes(ctypes.byref(lay), w, taps)
            want = oracle.row_bytes([K - c1, c1], bits, pad, taps if w else 1, bool(w))
            assert got == want


def test_validate_layout(L):
    from paper_2311_14114_gb300 import soniq
    perm = np.arange(300, dtype=np.int32)[::-1].copy()
    ok = _layout(soniq)
    assert L.soniq_validate_layout(ctypes.byref(ok), perm.ctypes.data_as(ctypes.c_void_p)) == 0
    bad = perm.copy()
    bad[5] = bad[6]
    assert L.soniq_validate_layout(ctypes.byref(ok), bad.ctypes.data_as(ctypes.c_void_p)) == 1
    for kw in (dict(count=(200, 99)), dict(bits=(0, 8)), dict(bits=(3, 9)), dict(pad=64)):
        lay = _layout(soniq, **kw)
        assert L.soniq_validate_layout(ctypes.byref(lay), None) == 1, kw


def test_host_side_argument_errors_need_no_gpu(L):
    from paper_2311_14114_gb300 import soniq
    lay = _layout(soniq, perm=ctypes.c_void_p(16))
    fake = ctypes.c_void_p(4096)
    # null output pointer
    assert L.soniq_pack_weights(ctypes.byref(lay), fake, 10, 1, 1, None, fake, None) == 1
    # misaligned packed weights
    assert L.soniq_pack_weights(ctypes.byref(lay), fake, 10, 1, 1, ctypes.c_void_p(4097 + 3), fake, None) == 3
    # bad scale mode
    assert L.soniq_quantize_act(ctypes.byref(lay), fake, 10, 7, fake, fake, None, 0, None) == 1
    # empty input is a no-op that touches nothing
    assert L.soniq_quantize_act(ctypes.byref(lay), None, 0, 0, None, None, None, 0, None) == 0
    # misaligned scratch
    assert L.soniq_quantize_act(ctypes.byref(lay), fake, 10, 0, fake, fake, ctypes.c_void_p(4100), 9000,
                                None) == 3
    assert L.soniq_mp_gemm(ctypes.byref(lay), None, None, 0, 0, None, None, 5, None, 0, None, 0, None, 0, None, None) == 0
    # both dispatch overrides at once
    assert L.soniq_mp_gemm(ctypes.byref(lay), fake, fake, 0, 4, fake, fake, 8, fake, 0, None, 3, None, 0, None, None) == 1
    # bad output dtype
    assert L.soniq_mp_gemm(ctypes.byref(lay), fake, fake, 0, 4, fake, fake, 8, fake, 9, None, 0, None, 0, None, None) == 1
    # conv: per-row activation scales are rejected (a dot product spans pixels)
    cd = soniq.conv_desc(1, 8, 8, 16)
    assert L.soniq_mp_conv2d(ctypes.byref(lay), ctypes.byref(cd), fake, fake, 1, fake, fake, fake, 0,
                             None, 0, None, 0, None, None) == 1
    # conv: filter larger than the padded image
    cd = soniq.conv_desc(1, 2, 2, 16, R=5, S=5, pad=(0, 0))
    assert L.soniq_mp_conv2d(ctypes.byref(lay), ctypes.byref(cd), fake, fake, 0, fake, fake, fake, 0,
                             None, 0, None, 0, None, None) == 1
    # K beyond the supported range
    big = _layout(soniq, K=70000, count=(70000, 0), bits=(2, 2), perm=ctypes.c_void_p(16))
    assert L.soniq_mp_gemm(ctypes.byref(big), fake, fake, 0, 4, fake, fake, 8, fake, 0, None, 0, None, 0, None, None) == 2
    # M beyond the 32-bit row coordinates
    assert L.soniq_mp_gemm(ctypes.byref(lay), fake, fake, 0, 2 ** 31, fake, fake, 8, fake, 0, None, 0, None, 0, None,
                           None) == 2
    assert L.soniq_mp_gemm_path(ctypes.byref(lay), 2 ** 31, 8, 0, 0) == -1
    assert L.soniq_mp_gemm_scratch_bytes(ctypes.byref(lay), 2 ** 31, 8, 0) == -1
    # conv geometry in 64-bit arithmetic: a pad that overflows 32 bits, and output rows past 2^31
    cd = soniq.conv_desc(1, 8, 8, 16, pad=(2 ** 30, 1))
    assert L.soniq_mp_conv2d(ctypes.byref(lay), ctypes.byref(cd), fake, fake, 0, fake, fake, fake, 0,
                             None, 0, None, 0, None, None) == 2
    cd = soniq.conv_desc(2 ** 20, 2 ** 10, 2 ** 10, 16)
    assert L.soniq_mp_conv2d(ctypes.byref(lay), ctypes.byref(cd), fake, fake, 0, fake, fake, fake, 0,
                             None, 0, None, 0, None, None) == 2
    assert L.soniq_mp_conv2d_scratch_bytes(ctypes.byref(lay), ctypes.byref(cd), 0) == -1
    # a negative pad is malformed
    cd = soniq.conv_desc(1, 8, 8, 16, pad=(-1, 1))
    assert L.soniq_mp_conv2d(ctypes.byref(lay), ctypes.byref(cd), fake, fake, 0, fake, fake, fake, 0,
                             None, 0, None, 0, None, None) == 1


def test_next_layer_descriptor_checks(L):
    """The quantize-in-epilogue descriptor is checked on the host: the output
    width must be the next layer's padded row length, outputs fp16."""
    from paper_2311_14114_gb300 import soniq
    lay = _layout(soniq, perm=ctypes.c_void_p(16))
    nxt_lay = _layout(soniq, K=40, count=(30, 10), bits=(2, 8), pad=32, perm=ctypes.c_void_p(16))
    fake = ctypes.c_void_p(4096)
    nxt = soniq.CNextLayer(ctypes.cast(ctypes.byref(nxt_lay), ctypes.c_void_p).value, 4096, 4096)
    # N = 64 = 32 + 32 (pad 32) is accepted up to the missing scratch; 8 is not the padded width
    assert L.soniq_mp_gemm(ctypes.byref(lay), fake, fake, 0, 300, fake, fake, 8, fake, 0, None, 0, None, 0,
                           ctypes.byref(nxt), None) == 1
    # bf16 outputs cannot feed the next layer's fp16 quantizer
    assert L.soniq_mp_gemm(ctypes.byref(lay), fake, fake, 0, 300, fake, fake, 64, fake, 1, None, 0, None, 0,
                           ctypes.byref(nxt), None) == 1
    # without staged scratch the fused epilogue is unavailable
    assert L.soniq_mp_gemm(ctypes.byref(lay), fake, fake, 0, 300, fake, fake, 64, fake, 0, None, 0, None, 0,
                           ctypes.byref(nxt), None) == 2


def test_scratch_size_queries(L):
    """The per-tensor quantize asks for a barrier and per-CTA maxima; the other
    activation modes ask for nothing; bad layouts give -1 (host only)."""
    from paper_2311_14114_gb300 import soniq
    lay = _layout(soniq, perm=ctypes.c_void_p(16))
    L.soniq_quantize_act_scratch_bytes.restype = ctypes.c_int64
    L.soniq_quantize_act_scratch_bytes.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32]
    assert L.soniq_quantize_act_scratch_bytes(ctypes.byref(lay), 1000, 0) == 256 + 8 * 1024
    assert L.soniq_quantize_act_scratch_bytes(ctypes.byref(lay), 1000, 1) == 0
    assert L.soniq_quantize_act_scratch_bytes(ctypes.byref(lay), 1000, 2) == 0
    assert L.soniq_quantize_act_scratch_bytes(ctypes.byref(lay), 1000, 9) == -1
    bad = _layout(soniq, count=(200, 99))
    assert L.soniq_quantize_act_scratch_bytes(ctypes.byref(bad), 1000, 0) == -1


def test_status_strings(L):
    L.soniq_status_string.restype = ctypes.c_char_p
    assert L.soniq_status_string(5) == b"device wait timed out"


def test_layout_variant_checks(L):
    """Host-side checks of the layout variants (signed activations, +-1 groups,
    scale runs): validation, run counts, and that only the staged path takes them."""
    from paper_2311_14114_gb300 import soniq
    perm = np.arange(300, dtype=np.int32)
    pp = perm.ctypes.data_as(ctypes.c_void_p)
    ok = _layout(soniq, act_kind=(1, 1))
    assert L.soniq_validate_layout(ctypes.byref(ok), pp) == 0
    assert L.soniq_scale_runs(ctypes.byref(ok)) == 1
    runs = _layout(soniq, sub_k=128)                          # PA = 256 and 128
    assert L.soniq_scale_runs(ctypes.byref(runs)) == 2
    assert L.soniq_scale_runs(ctypes.byref(_layout(soniq, sub_k=384))) == 1
    for bad in (_layout(soniq, act_kind=(2, 0)),              # +-1 needs one-bit codes
                _layout(soniq, act_kind=(3, 0)),
                _layout(soniq, sub_k=100),
                _layout(soniq, sub_k=-128)):
        assert L.soniq_validate_layout(ctypes.byref(bad), pp) == 1
    assert L.soniq_validate_layout(ctypes.byref(_layout(soniq, act_kind=(2, 0), bits=(1, 8))), pp) == 0
    assert L.soniq_validate_layout(ctypes.byref(_layout(soniq, act_kind=(1, 0), pad=32)), pp) == 2
    # staged path only, with its scratch; no GEMV / fused / skinny
    need = L.soniq_mp_gemm_scratch_bytes(ctypes.byref(runs), 16, 64, 0)
    assert need > 0
    assert L.soniq_mp_gemm_path(ctypes.byref(runs), 16, 64, 0, need) == 2
    assert L.soniq_mp_gemm_path(ctypes.byref(runs), 16, 64, 0, 0) == -1
    assert L.soniq_mp_gemm_path(ctypes.byref(runs), 16, 64, 16, need) == -1


def test_binding_refuses_to_run_without_the_library(monkeypatch):
    """No CPU fallback: without libsoniq.so every call of the binding raises."""
    from paper_2311_14114_gb300 import soniq
    monkeypatch.setattr(soniq, "_lib", None)
    monkeypatch.setattr(soniq, "LIB_PATH", os.path.join(ROOT, "no_such_dir", "libsoniq.so"))
    with pytest.raises(RuntimeError, match="not built"):
        soniq.lib()
    # the first call a user makes (a layout, validated by the library) raises too
    with pytest.raises(RuntimeError, match="not built"):
        soniq.Layout(np.arange(64, dtype=np.int32), [48, 16], [2, 8])
