"""GPU parity: the CUDA path (through the C-ABI) against the CPU oracle on the
same seeded inputs.  Packed bytes, scales and int32 accumulators must match
bit for bit; fp16 outputs within the tolerance of helpers.y_tolerance."""
import numpy as np
import pytest

import oracle
from helpers import assert_y_close, fp16_ulp_diff
from paper_2311_14114_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sq():
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


def _dev(x, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def run_linear(sq, d, pad=128, act_mode="tensor", s_a_cal=None, w_mode="row", flags=0,
               out_dtype=torch.float16, bits_a=None):
    bits_w = d["bits"]
    bits_a = bits_w if bits_a is None else bits_a
    lay = sq.Layout(d["perm"], d["count"], bits_w, bits_a, pad_unit=pad)
    A = _dev(d["A"])
    W = _dev(d["W"])
    Wp, s_w = sq.pack_weights(lay, W, scale_mode=w_mode)
    s_in = _dev(np.asarray(s_a_cal, np.float32)) if act_mode == "calibrated" else None
    Ap, s_a = sq.quantize_act(lay, A, scale_mode=act_mode, s_a=s_in)
    M, N = A.shape[0], W.shape[0]
    acc = torch.zeros((2, M, N), dtype=torch.int32, device="cuda")
    Y = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, scale_mode=act_mode, acc_dbg=acc, flags=flags,
                   out_dtype=out_dtype)
    assert sq.sync_status() == 0
    return dict(Ap=Ap.cpu().numpy(), s_a=s_a.cpu().numpy(), Wp=Wp.cpu().numpy(),
                s_w=s_w.cpu().numpy(), acc=acc.cpu().numpy(), Y=Y.float().cpu().numpy())


def check_linear(sq, d, pad=128, act_mode="tensor", s_a_cal=None, w_mode="row", flags=0,
                 rows=None, out_dtype=torch.float16, bits_a=None, what=""):
    bits_w = d["bits"]
    bits_a = bits_w if bits_a is None else bits_a
    g = run_linear(sq, d, pad, act_mode, s_a_cal, w_mode, flags, out_dtype, bits_a)
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], bits_a, bits_w, pad_unit=pad,
                      act_mode=act_mode, s_a=s_a_cal, w_per_row=(w_mode == "row"), rows=rows)
    assert np.array_equal(g["s_w"], r["s_w"]), what + " weight scales"
    assert np.array_equal(g["Wp"], r["Wp"]), what + " packed weights"
    assert np.array_equal(g["s_a"], r["s_a"]), what + " activation scales"
    assert np.array_equal(g["Ap"], r["Ap"]), what + " packed activations"
    sel = slice(None) if rows is None else rows
    acc_g = g["acc"][:, sel, :]
    assert np.array_equal(acc_g.astype(np.int64), r["acc"]), what + " int32 accumulators"
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], bits_a, bits_w, rows=rows,
                                  s_a_per_row=(act_mode == "row"))
    y_ref = r["Y64"].astype(np.float16) if out_dtype == torch.float16 else r["Y64"]
    if out_dtype == torch.bfloat16:
        # bf16 keeps 8 significant bits: one bf16 ulp is 2^-7 relative
        tol = 2.0 ** -7 * np.maximum(np.abs(r["Y64"]), terms * 2.0 ** -10) + 1e-30
        assert (np.abs(g["Y"][sel] - r["Y64"]) <= tol).all(), what + " bf16 output"
    else:
        assert_y_close(g["Y"][sel], y_ref, terms, what)
        # away from cancellation (|y| >= sum_g |alpha_g Acc_g| / 16) the fp32 sum is
        # far below an fp16 ulp, so the two roundings differ by at most one ulp
        keep = np.abs(r["Y64"]) >= terms / 16
        assert fp16_ulp_diff(g["Y"][sel].astype(np.float16)[keep], y_ref[keep]) <= 1
    return g, r


# ---------------------------------------------------------------------------
# quantize / pack kernels
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("bits", [(1, 4), (2, 8), (3, 6), (4, 5), (7, 8)])
@pytest.mark.parametrize("pad", [32, 128])
@pytest.mark.parametrize("mode", ["tensor", "row"])
def test_quantize_act_bytes(sq, bits, pad, mode):
    d = wl.random_linear(3 + bits[0], M=77, K=333, N=8, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=0.3, n_outliers=3)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=pad)
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]), scale_mode=mode)
    A32 = d["A"].astype(np.float32)
    s_ref = oracle.act_scales(A32, d["perm"], d["count"], per_row=(mode == "row"))
    U = oracle.act_codes(A32, d["perm"], d["count"], d["bits"], s_ref, per_row=(mode == "row"))
    assert np.array_equal(s_a.cpu().numpy(), s_ref)
    assert np.array_equal(Ap.cpu().numpy(), oracle.pack_act_rows(U, d["count"], d["bits"], pad))


def test_quantize_act_calibrated_clips(sq):
    d = wl.random_linear(9, M=40, K=256, N=8, bits_lo=2, bits_hi=8, frac_hi=0.25, n_outliers=2,
                         outlier_scale=10.0)
    s_cal = np.array([0.8, 3.0], np.float32)          # below the true max: inputs clip
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Ap, _ = sq.quantize_act(lay, _dev(d["A"]), scale_mode="calibrated", s_a=_dev(s_cal))
    U = oracle.act_codes(d["A"].astype(np.float32), d["perm"], d["count"], d["bits"], s_cal)
    assert (U[:, :d["count"][0]] == 3).any() and (U[:, d["count"][0]:] == 255).any()
    assert np.array_equal(Ap.cpu().numpy(), oracle.pack_act_rows(U, d["count"], d["bits"], 128))


@pytest.mark.parametrize("mode", ["tensor", "row"])
def test_quantize_act_bytes_full_warps(sq, mode):
    # enough rows that each warp stages 32 rows, plus a ragged last tile
    d = wl.random_linear(21, M=80011, K=64, N=8, bits_lo=3, bits_hi=8, frac_hi=0.3, n_outliers=2)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]), scale_mode=mode)
    A32 = d["A"].astype(np.float32)
    s_ref = oracle.act_scales(A32, d["perm"], d["count"], per_row=(mode == "row"))
    U = oracle.act_codes(A32, d["perm"], d["count"], d["bits"], s_ref, per_row=(mode == "row"))
    assert np.array_equal(s_a.cpu().numpy(), s_ref)
    assert np.array_equal(Ap.cpu().numpy(), oracle.pack_act_rows(U, d["count"], d["bits"], 32))


@pytest.mark.parametrize("s_cal", [(1.0, 3.7), (2.0 ** -70, 2.0 ** 70), (6.1e-5, 65504.0)])
def test_quantize_act_every_fp16_value(sq, s_cal):
    # every finite fp16 pattern (signed zeros, subnormals, the extremes) through Sec. 3 step 2
    h = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    h = h[(h & 0x7C00) != 0x7C00]
    K = 256
    pad = (-len(h)) % K
    A = np.concatenate([h, np.zeros(pad, np.uint16)]).view(np.float16).reshape(-1, K)
    rng = np.random.default_rng(5)
    perm = rng.permutation(K).astype(np.int32)
    count, bits = [160, 96], [4, 8]
    lay = sq.Layout(perm, count, bits, pad_unit=32)
    s = np.asarray(s_cal, np.float32)
    Ap, _ = sq.quantize_act(lay, _dev(A), scale_mode="calibrated", s_a=_dev(s))
    U = oracle.act_codes(A.astype(np.float32), perm, count, bits, s)
    assert np.array_equal(Ap.cpu().numpy(), oracle.pack_act_rows(U, count, bits, 32))


def test_quantize_act_unaligned_k(sq):
    # K % 8 != 0 takes the scalar staging path
    d = wl.random_linear(10, M=33, K=301, N=8, bits_lo=3, bits_hi=7, frac_hi=0.4)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], pad_unit=32)
    assert np.array_equal(s_a.cpu().numpy(), r["s_a"])
    assert np.array_equal(Ap.cpu().numpy(), r["Ap"])


@pytest.mark.parametrize("taps", [1, 9])
@pytest.mark.parametrize("mode", ["row", "tensor"])
@pytest.mark.parametrize("bits", [(1, 8), (3, 6), (4, 4), (2, 5)])
def test_pack_weights_bytes(sq, taps, mode, bits):
    rng = np.random.default_rng(taps * 10 + bits[0])
    K, N = 200, 45
    perm, count, _ = wl.assignment(rng, K, 0.3, 0)
    W = (rng.standard_normal((N, taps, K)) * 0.05).astype(np.float32)
    pad = 32 if taps > 1 else 128
    lay = sq.Layout(perm, count, bits, pad_unit=pad)
    Wp, s_w = sq.pack_weights(lay, _dev(W if taps > 1 else W[:, 0, :]), scale_mode=mode)
    s_ref = oracle.weight_scales(W, perm, count, per_row=(mode == "row"))
    J = oracle.weight_codes(W, perm, count, bits, s_ref)
    assert np.array_equal(s_w.cpu().numpy(), s_ref)
    assert np.array_equal(Wp.cpu().numpy(), oracle.pack_weight_rows(J, count, bits, pad))


# ---------------------------------------------------------------------------
# GEMM (tensor cores) and GEMV (CUDA cores)
# ---------------------------------------------------------------------------

GEMM_BITS = [(1, 4), (1, 8), (2, 6), (2, 8), (3, 5), (3, 8), (4, 4), (4, 6), (4, 8), (2, 2), (8, 8), (5, 7)]


# tensor-core paths: staged (expand into scratch, then GEMM) and fused (expand on chip)
STAGED, FUSED = 2 | 8, 2 | 4


@pytest.mark.parametrize("path", [STAGED, FUSED], ids=["staged", "fused"])
@pytest.mark.parametrize("bits", GEMM_BITS)
def test_gemm_small_all_bit_pairs(sq, bits, path):
    # several 128x128 tiles plus ragged tails in M, N and K
    d = wl.random_linear(100 + bits[0] * 10 + bits[1], M=300, K=333, N=264, bits_lo=bits[0],
                         bits_hi=bits[1], frac_hi=0.3, n_outliers=2)
    check_linear(sq, d, flags=path, what=f"gemm{bits}")


def test_gemm_paths_reported(sq):
    d = wl.random_linear(5, M=300, K=333, N=264, bits_lo=2, bits_hi=8, frac_hi=0.3)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    assert sq.gemm_path(lay, 300, 264, STAGED) == sq.PATH_NAMES[2]
    assert sq.gemm_path(lay, 300, 264) == sq.PATH_NAMES[1]          # small: the fused kernel
    assert sq.gemm_path(lay, 8192, 4096) == sq.PATH_NAMES[2]        # large: staged
    assert sq.gemm_path(lay, 300, 264, FUSED) == sq.PATH_NAMES[1]
    assert sq.gemm_path(lay, 8, 264) == sq.PATH_NAMES[0]


@pytest.mark.parametrize("pad", [32, 128])
@pytest.mark.parametrize("act_mode", ["tensor", "row", "calibrated"])
def test_gemm_modes(sq, pad, act_mode):
    d = wl.random_linear(7, M=200, K=500, N=136, bits_lo=2, bits_hi=8, frac_hi=0.25, n_outliers=4,
                         outlier_scale=10.0)
    cal = [1.5, 9.0] if act_mode == "calibrated" else None
    check_linear(sq, d, pad=pad, act_mode=act_mode, s_a_cal=cal, flags=2,
                 what=f"gemm pad{pad} {act_mode}")


def test_gemm_bf16_and_tensor_weight_scale(sq):
    d = wl.random_linear(8, M=150, K=256, N=128, bits_lo=3, bits_hi=6, frac_hi=0.2)
    check_linear(sq, d, w_mode="tensor", flags=2, out_dtype=torch.bfloat16, what="bf16")


@pytest.mark.parametrize("frac", [0.0, 1.0])
def test_gemm_single_group(sq, frac):
    d = wl.random_linear(11, M=130, K=256, N=130, bits_lo=2, bits_hi=8, frac_hi=frac)
    check_linear(sq, d, flags=2, what=f"single group frac={frac}")


def test_gemm_different_act_and_weight_bits(sq):
    d = wl.random_linear(12, M=140, K=300, N=128, bits_lo=2, bits_hi=7, frac_hi=0.3)
    check_linear(sq, d, bits_a=[3, 6], flags=2, what="bits_a != bits_w")


def test_gemm_tiny_k_and_one_row(sq):
    d = wl.random_linear(13, M=129, K=5, N=17, bits_lo=2, bits_hi=8, frac_hi=0.4)
    check_linear(sq, d, flags=2, what="K=5")


def test_gemm_zero_group(sq):
    d = wl.random_linear(14, M=130, K=256, N=128, bits_lo=4, bits_hi=8, frac_hi=0.25)
    d = dict(d)
    A = d["A"].copy()
    A[:, d["perm"][d["count"][0]:]] = 0
    d["A"] = A
    g, r = check_linear(sq, d, flags=2, what="zero group")
    assert not g["acc"][1].any()


@pytest.mark.parametrize("path", [STAGED, FUSED], ids=["staged", "fused"])
def test_gemm_exactness_segments(sq, path):
    """Worst-case 8-bit codes over a long K: every partial sum is the extreme
    255 * -128, so a single fp32 accumulator would leave the exact-integer
    range after 514 codes.  The segmented accumulation must stay exact."""
    K, M, N = 4096, 130, 136
    perm = np.arange(K, dtype=np.int32)
    count = [0, K]
    A = np.full((M, K), 2.0, np.float16)
    W = np.full((N, K), -0.5, np.float32)
    W[::3, :] = 0.5                          # j = 127 on some rows
    A[1::2, ::7] = 0                         # some rows with fewer terms
    d = dict(A=A, W=W, perm=perm, count=count, bits=[4, 8])
    g, r = check_linear(sq, d, flags=path, what="segments")
    assert np.abs(r["acc"]).max() > 2 ** 24


def test_gemm_8bit_many_tiles_repeatable(sq):
    """8-bit weight groups expand fastest, so their expander warps run furthest
    ahead of the TMA ring; repeated runs over many tiles must stay exact
    (regression: a ring slot handed back before its words were consumed)."""
    d = wl.random_linear(15, M=4096, K=1152, N=1024, bits_lo=4, bits_hi=8, frac_hi=1.0)
    rows = np.arange(0, 4096, 8)
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], rows=rows)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    for rep in range(6):
        acc = torch.zeros((2, 4096, 1024), dtype=torch.int32, device="cuda")
        sq.mp_gemm(lay, Ap, s_a, Wp, s_w, acc_dbg=acc, flags=2)
        assert sq.sync_status() == 0
        assert np.array_equal(acc.cpu().numpy()[:, rows].astype(np.int64), r["acc"]), f"rep {rep}"


@pytest.mark.parametrize("M", [1, 2, 3, 4, 7, 16])
@pytest.mark.parametrize("bits", [(3, 6), (1, 8), (4, 4)])
def test_gemv(sq, M, bits):
    d = wl.random_linear(200 + M, M=M, K=1000, N=333, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=0.15, n_outliers=2)
    check_linear(sq, d, what=f"gemv M={M}")


@pytest.mark.parametrize("M,flags", [(12, 0), (13, 0), (13, 1), (16, 1)])
def test_gemv_dispatch_threshold_and_forced(sq, M, flags):
    """Both sides of the GEMV / tensor-core dispatch threshold with default flags,
    and the GEMV forced above it, against the oracle (bytes, accumulators, fp16)."""
    d = wl.random_linear(210 + M, M=M, K=1000, N=333, bits_lo=3, bits_hi=6, frac_hi=0.15, n_outliers=2)
    check_linear(sq, d, flags=flags, what=f"gemv M={M} flags={flags}")


def test_gemv_row_scales_pad32(sq):
    d = wl.random_linear(300, M=5, K=700, N=99, bits_lo=2, bits_hi=8, frac_hi=0.2)
    check_linear(sq, d, pad=32, act_mode="row", what="gemv row scales")


@pytest.mark.parametrize("M", [1, 2])
@pytest.mark.parametrize("K,N,bits", [
    (32768, 2000, (6, 8)),   # 24+ KB rows: a CTA's rows run in several rounds through shared memory
    (4096, 7, (3, 6)),       # fewer rows than one 16-row piece
    (1000, 2431, (1, 5)),    # ragged pieces and a ragged last CTA, pad 32
])
def test_gemv_bulk_rounds_and_ragged_pieces(sq, M, K, N, bits):
    d = wl.random_linear(700 + M + N, M=M, K=K, N=N, bits_lo=bits[0], bits_hi=bits[1], frac_hi=0.3)
    check_linear(sq, d, pad=32 if K == 1000 else 128, what=f"gemv M={M} K={K} N={N}")


def test_gemv_matches_mma(sq):
    d = wl.random_linear(301, M=16, K=768, N=256, bits_lo=3, bits_hi=6, frac_hi=0.15)
    a = run_linear(sq, d, flags=1)
    b = run_linear(sq, d, flags=2)
    assert np.array_equal(a["acc"], b["acc"])


# ---------------------------------------------------------------------------
# implicit-GEMM convolution
# ---------------------------------------------------------------------------

def run_conv(sq, spec, pad_unit=32, flags=0):
    d = wl.make_conv(spec)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=pad_unit)
    X = _dev(d["X"]).reshape(-1, spec.C)
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Xp, s_a = sq.quantize_act(lay, X)
    cd = sq.conv_desc(spec.batch, spec.H, spec.W, spec.C_out, spec.R, spec.S, spec.stride, spec.pad)
    acc = torch.zeros((2, spec.M, spec.C_out), dtype=torch.int32, device="cuda")
    Y = sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, acc_dbg=acc, flags=flags)
    assert sq.sync_status() == 0
    return d, dict(Xp=Xp.cpu().numpy(), s_a=s_a.cpu().numpy(), Wp=Wp.cpu().numpy(),
                   s_w=s_w.cpu().numpy(), acc=acc.cpu().numpy(),
                   Y=Y.float().cpu().numpy().reshape(spec.M, spec.C_out))


def check_conv(sq, spec, pad_unit=32, pix=None, what="conv", flags=0):
    d, g = run_conv(sq, spec, pad_unit, flags)
    r = oracle.conv2d(d["X"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], spec.R, spec.S,
                      stride=spec.stride, pad=spec.pad, pad_unit=pad_unit, pix=pix)
    assert np.array_equal(g["s_a"], r["s_a"]) and np.array_equal(g["s_w"], r["s_w"])
    assert np.array_equal(g["Xp"], r["Xp"]), what + " packed pixels"
    assert np.array_equal(g["Wp"], r["Wp"]), what + " packed weights"
    sel = slice(None) if pix is None else pix
    assert np.array_equal(g["acc"][:, sel, :].astype(np.int64), r["acc"]), what + " accumulators"
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], d["bits"], d["bits"])
    assert_y_close(g["Y"][sel], r["Y16"], terms, what)


@pytest.mark.parametrize("flags", [8, 4], ids=["staged", "fused"])
@pytest.mark.parametrize("bits", [(4, 8), (1, 4), (2, 6)])
@pytest.mark.parametrize("geom", [((1, 1), (1, 1)), ((2, 2), (0, 0)), ((1, 2), (1, 0))])
def test_conv_small(sq, bits, geom, flags):
    stride, pad = geom
    spec = wl.ConvSpec("t", batch=3, H=9, W=7, C=70, C_out=40, R=3, S=3, stride=stride, pad=pad,
                       bits_lo=bits[0], bits_hi=bits[1], frac_hi=0.3, seed=bits[0] + 7 * stride[0])
    check_conv(sq, spec, what=f"conv{bits}{geom}", flags=flags)


def test_conv_1x1_and_5x5_pad128(sq):
    for R, pad in ((1, 0), (5, 2)):
        spec = wl.ConvSpec("t", batch=2, H=8, W=8, C=64, C_out=130, R=R, S=R, stride=(1, 1),
                           pad=(pad, pad), bits_lo=3, bits_hi=8, frac_hi=0.25, seed=R)
        check_conv(sq, spec, pad_unit=128, what=f"conv {R}x{R}")


def test_conv_wide_rows_gather_path(sq):
    # 128-pixel tiles of a 200-pixel-wide image need ~800 input pixels of 256+ bytes: more
    # than the shared-memory halo holds, so the kernel gathers each chunk's rows instead
    spec = wl.ConvSpec("t", batch=1, H=6, W=200, C=256, C_out=32, R=3, S=3, stride=(1, 1),
                       pad=(1, 1), bits_lo=6, bits_hi=8, frac_hi=0.5, seed=11)
    check_conv(sq, spec, what="conv wide rows")


def test_conv_tiles_span_many_images(sq):
    # 5x5 images: a 128-pixel tile covers parts of six images (halo over whole images)
    spec = wl.ConvSpec("t", batch=13, H=5, W=5, C=96, C_out=24, R=3, S=3, stride=(1, 1),
                       pad=(1, 1), bits_lo=2, bits_hi=7, frac_hi=0.4, seed=12)
    check_conv(sq, spec, what="conv small images")


# ---------------------------------------------------------------------------
# full-size workloads (sampled outputs where the oracle would be slow)
# ---------------------------------------------------------------------------

def _sample_rows(M, n, seed):
    rng = np.random.default_rng(seed)
    rows = np.unique(np.concatenate([[0, M - 1], rng.choice(M, n, replace=False)]))
    return rows.astype(np.int64)


def test_full_linear_64x512x512(sq):
    d = wl.make_linear(wl.LINEAR_SMALL)
    check_linear(sq, d, what="linear 64x512x512")


@pytest.mark.parametrize("flags", [8, 4], ids=["staged", "fused"])
@pytest.mark.parametrize("spec", [wl.CONV_RESNET, wl.CONV_RESNET_1B4B], ids=lambda s: s.name)
def test_full_conv_resnet(sq, spec, flags):
    pix = _sample_rows(spec.M, 600, 1)
    check_conv(sq, spec, pix=pix, what=spec.name, flags=flags)


def test_full_mlp_up(sq):
    d = wl.make_linear(wl.MLP_UP)
    check_linear(sq, d, rows=_sample_rows(wl.MLP_UP.M, 200, 2), what=wl.MLP_UP.name)


@pytest.mark.parametrize("M", [1, 4, 16])
def test_full_decode(sq, M):
    d = wl.make_linear(wl.DECODE[M])
    check_linear(sq, d, what=wl.DECODE[M].name)


SWEEP_POINTS = [(s.bits_lo, s.bits_hi, s.frac_hi) for s in wl.sweep_specs()]


@pytest.mark.parametrize("lo,hi,frac", SWEEP_POINTS, ids=lambda v: str(v))
def test_sweep_every_point_full_k(sq, lo, hi, frac):
    """Every (low bits, high bits, high fraction) point of the precision sweep at
    its full K = N = 4096, on 256 activation rows; sampled rows against the oracle."""
    spec = wl.LinearSpec("sweep", M=8192, K=4096, N=4096, bits_lo=lo, bits_hi=hi, frac_hi=frac)
    d = wl.make_linear(spec, M=256)
    check_linear(sq, d, rows=_sample_rows(256, 24, 4), what=f"sweep lo{lo} hi{hi} f{frac}")


@pytest.mark.parametrize("flags", [0, FUSED], ids=["default", "fused"])
@pytest.mark.parametrize("lo,hi,frac", [(1, 8, 1.0), (2, 4, 0.1), (3, 6, 0.5), (4, 8, 0.25)])
def test_full_sweep_points(sq, lo, hi, frac, flags):
    spec = wl.LinearSpec("sweep", M=8192, K=4096, N=4096, bits_lo=lo, bits_hi=hi, frac_hi=frac)
    d = wl.make_linear(spec)
    check_linear(sq, d, rows=_sample_rows(8192, 48, 3), what=f"sweep lo{lo} hi{hi} f{frac}", flags=flags)


# ---------------------------------------------------------------------------
# failure reporting without a GPU fault
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("path", [STAGED, FUSED], ids=["staged", "fused"])
def test_timeout_is_reported_and_context_survives(sq, path):
    d = wl.random_linear(400, M=300, K=1000, N=256, bits_lo=2, bits_hi=8, frac_hi=0.25)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    assert sq.sync_status() == 0
    sq.mp_gemm(lay, Ap, s_a, Wp, s_w, flags=path | sq.FLAG_TEST_DROP_ARRIVE)
    assert sq.sync_status() == 5            # SONIQ_ERR_TIMEOUT, then cleared
    assert sq.sync_status() == 0
    check_linear(sq, d, flags=path, what="after timeout")


def test_quantize_barrier_timeout_is_reported_and_scratch_recovers(sq):
    """The one-pass per-tensor quantize with caller scratch: a dropped barrier
    arrival (host-armed test hook) runs the other CTAs' bounded waits out; the
    call reports SONIQ_ERR_TIMEOUT, the binding zeroes its scratch as the
    contract asks, and the next calls are exact."""
    d = wl.random_linear(401, M=2000, K=640, N=8, bits_lo=3, bits_hi=8, frac_hi=0.3, n_outliers=2)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    A = _dev(d["A"])
    assert sq.sync_status() == 0
    sq.test_drop_barrier_arrival(True)
    sq.quantize_act(lay, A, "tensor")
    assert sq.sync_status() == sq.SONIQ_ERR_TIMEOUT
    assert sq.sync_status() == 0
    A32 = d["A"].astype(np.float32)
    s_ref = oracle.act_scales(A32, d["perm"], d["count"])
    Ap_ref = oracle.pack_act_rows(oracle.act_codes(A32, d["perm"], d["count"], d["bits"], s_ref),
                                  d["count"], d["bits"], 128)
    for _ in range(2):
        Ap, s_a = sq.quantize_act(lay, A, "tensor")
        assert sq.sync_status() == 0
        assert np.array_equal(s_a.cpu().numpy(), s_ref)
        assert np.array_equal(Ap.cpu().numpy(), Ap_ref)


@pytest.mark.parametrize("K", [512, 3000])
def test_quantize_per_tensor_without_scratch_two_pass(sq, K):
    """scratch = NULL takes the two-pass per-tensor path (max-abs pass, then quantize)."""
    d = wl.random_linear(402, M=500, K=K, N=8, bits_lo=2, bits_hi=8, frac_hi=0.3, n_outliers=2)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]), "tensor", scratch=None)
    assert sq.sync_status() == 0
    A32 = d["A"].astype(np.float32)
    s_ref = oracle.act_scales(A32, d["perm"], d["count"])
    Ap_ref = oracle.pack_act_rows(oracle.act_codes(A32, d["perm"], d["count"], d["bits"], s_ref),
                                  d["count"], d["bits"], 32)
    assert np.array_equal(s_a.cpu().numpy(), s_ref)
    assert np.array_equal(Ap.cpu().numpy(), Ap_ref)
