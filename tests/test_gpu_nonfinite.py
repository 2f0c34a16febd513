"""Non-finite inputs (NaN, +-inf) through every activation-quantize path, the
weight pack and the next-layer epilogue, against the oracle.

Sec. 3 steps 2-3 clip the rounded level to the code range, so under a finite
scale +inf takes the top code and -inf the bottom one.  A NaN quotient (a NaN
input, or inf / inf under a scale that an infinite input made infinite) lies
on neither side of the clip and gives code 0.  Max-abs scales skip NaN and
keep infinities.  Each case plants the three values at seeded positions of
both precision groups (or of chosen rows and groups, where a scale is taken
from the data) and compares scales and packed bytes bit for bit."""
import numpy as np
import pytest

import oracle
from paper_2311_14114_gb300 import workloads as wl
from test_gpu_fused_quant import _arrange_rows, _next_layout, _to_channels

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

NAN, INF = np.float16(np.nan), np.float16(np.inf)


@pytest.fixture(scope="module")
def sq():
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _plant(X, cells, values):
    """X[r, c] = v for each cell and value, cycling through the values."""
    X = X.copy()
    for i, (r, c) in enumerate(cells):
        X[r, c] = values[i % len(values)]
    return X


def _cells(rng, rows, channels, n):
    return list(zip(rng.integers(0, rows, n), rng.choice(channels, n)))


def _check_act(sq, lay, perm, count, bits, pad, A16, mode, s_cal=None, scratch=False, what=""):
    s_in = _dev(np.asarray(s_cal, np.float32)) if mode == "calibrated" else None
    Ap, s_a = sq.quantize_act(lay, _dev(A16), scale_mode=mode, s_a=s_in, scratch=scratch)
    assert sq.sync_status() == 0
    A32 = A16.astype(np.float32)
    if mode == "calibrated":
        s_ref = np.asarray(s_cal, np.float32)
    else:
        s_ref = oracle.act_scales(A32, perm, count, per_row=(mode == "row"))
        assert np.array_equal(s_a.cpu().numpy(), s_ref), what + ": scales"
    U = oracle.act_codes(A32, perm, count, bits, s_ref, per_row=(mode == "row"))
    assert np.array_equal(Ap.cpu().numpy(), oracle.pack_act_rows(U, count, bits, pad)), what + ": packed codes"
    return U


# (M, K): K = 256 stages rows for the bulk gather kernel; K = 301 (K % 8 != 0)
# takes the tiled kernel's scalar staging; K = 32768 rows do not fit the gather
# kernel's stages and take the tiled kernel's vector staging
@pytest.mark.parametrize("M,K", [(40, 256), (33, 301), (3, 32768)])
@pytest.mark.parametrize("bits", [(4, 8), (2, 6), (1, 3)])
def test_calibrated_scales_clip_infinities(sq, M, K, bits):
    rng = np.random.default_rng(M + K + bits[0])
    perm, count, _ = wl.assignment(rng, K, 0.3, 0)
    A = (rng.standard_normal((M, K)) * 0.7).astype(np.float16)
    A = _plant(A, _cells(rng, M, np.arange(K), 3 * 12), [NAN, INF, -INF])
    lay = sq.Layout(perm, count, list(bits), pad_unit=32)
    s_cal = [0.9, 1.7]
    U = _check_act(sq, lay, perm, count, list(bits), 32, A, "calibrated", s_cal, what=f"calibrated {M}x{K} {bits}")
    # +inf reached the top code in some group (the planted cells cover both)
    top = [(1 << b) - 1 for b in bits]
    pos_inf = np.isposinf(A.astype(np.float32))[:, perm]
    assert pos_inf.any()
    for g, lo, hi in ((0, 0, count[0]), (1, count[0], K)):
        assert (U[:, lo:hi][pos_inf[:, lo:hi]] == top[g]).all()


# per-tensor scales from the data: group 0 carries NaN (its scale stays finite,
# the NaN codes to 0 on the Markstein path), group 1 carries +-inf (its scale
# becomes inf, every code of the group 0).  Paths: one CTA (up to 16K values),
# the one-pass kernel (library scratch), the two passes (no scratch), and the
# two passes with the tiled kernel (K % 8 != 0).
@pytest.mark.parametrize("M,K,scratch", [(16, 256, False), (300, 256, False), (300, 256, None), (80, 301, None)],
                         ids=["one-cta", "one-pass", "two-pass", "two-pass-tiles"])
def test_tensor_scales_skip_nan_keep_inf(sq, M, K, scratch):
    rng = np.random.default_rng(M * 7 + K)
    perm, count, _ = wl.assignment(rng, K, 0.3, 0)
    A = (rng.standard_normal((M, K)) * 0.7).astype(np.float16)
    A = _plant(A, _cells(rng, M, perm[:count[0]], 9), [NAN])
    A = _plant(A, _cells(rng, M, perm[count[0]:], 4), [INF, -INF])
    lay = sq.Layout(perm, count, [3, 8], pad_unit=32)
    _check_act(sq, lay, perm, count, [3, 8], 32, A, "tensor", scratch=scratch, what=f"tensor {M}x{K}")


@pytest.mark.parametrize("M,K", [(40, 256), (33, 301)])
def test_row_scales_skip_nan_keep_inf(sq, M, K):
    rng = np.random.default_rng(M + 3 * K)
    perm, count, _ = wl.assignment(rng, K, 0.3, 0)
    A = (rng.standard_normal((M, K)) * 0.7).astype(np.float16)
    g0, g1 = perm[:count[0]], perm[count[0]:]
    A[1, g0[2]] = INF        # row 1, group 0: scale inf
    A[2, g1[1]] = NAN        # row 2, group 1: finite scale, the NaN codes to 0
    A[3, g1[4]] = -INF       # row 3, group 1: scale inf
    A[4, g0[0]] = NAN
    A[4, g0[5]] = -INF
    lay = sq.Layout(perm, count, [4, 8], pad_unit=32)
    _check_act(sq, lay, perm, count, [4, 8], 32, A, "row", what=f"row {M}x{K}")


@pytest.mark.parametrize("taps", [1, 9])
@pytest.mark.parametrize("mode", ["row", "tensor"])
def test_pack_weights_non_finite(sq, taps, mode):
    rng = np.random.default_rng(taps + (mode == "row"))
    K, N = 200, 45
    perm, count, _ = wl.assignment(rng, K, 0.3, 0)
    bits = [3, 6]
    W = (rng.standard_normal((N, taps, K)) * 0.05).astype(np.float32)
    g0, g1 = perm[:count[0]], perm[count[0]:]
    W[0, 0, g0[3]] = np.nan                  # finite scale: NaN codes to 0
    W[5, taps - 1, g1[1]] = np.nan
    if mode == "row":
        W[7, 0, g0[0]] = np.inf              # row 7, group 0: scale inf
        W[9, taps - 1, g1[2]] = -np.inf      # row 9, group 1: scale inf
    pad = 32 if taps > 1 else 128
    lay = sq.Layout(perm, count, bits, pad_unit=pad)
    Wp, s_w = sq.pack_weights(lay, _dev(W if taps > 1 else W[:, 0, :]), scale_mode=mode)
    assert sq.sync_status() == 0
    s_ref = oracle.weight_scales(W, perm, count, per_row=(mode == "row"))
    J = oracle.weight_codes(W, perm, count, bits, s_ref)
    assert np.array_equal(s_w.cpu().numpy(), s_ref)
    assert np.array_equal(Wp.cpu().numpy(), oracle.pack_weight_rows(J, count, bits, pad))


@pytest.mark.parametrize("mode", ["row", "tensor"])
def test_pack_weights_extreme_scales(sq, mode):
    """Row maxima from the smallest fp32 subnormal to 3e38: where RN(1/s) * 2^(n-1)
    overflows (scales under about 2^-121) every code takes the IEEE division;
    where 1/s is subnormal (scales over 2^126) the estimate stays inside the
    tie window.  Per tensor, all rows share the largest maximum of the tiny ones."""
    rng = np.random.default_rng(77 + (mode == "row"))
    K = 200
    perm, count, _ = wl.assignment(rng, K, 0.3, 0)
    bases = np.array([1.4e-45, 1e-42, 1e-40, 3e-39, 1.2e-38, 1e-37, 3.7e-37, 1e-36, 1e-30, 1.0, 1e30, 8.6e37,
                      1e38, 3e38], np.float64)
    if mode == "tensor":
        bases = bases[bases < 1e-35]
    N = len(bases) * 4
    W = (rng.uniform(-1.0, 1.0, (N, K)) * np.repeat(bases, 4)[:, None]).astype(np.float32)
    # exact ties at half-levels and the maxima themselves
    W[::4, :8] = (np.repeat(bases, 1)[:, None] * np.array([1, -1, 0.5, -0.5, 0.25, 0.75, 1 / 3, -1 / 7])).astype(
        np.float32)
    bits = [3, 8]
    lay = sq.Layout(perm, count, bits)
    Wp, s_w = sq.pack_weights(lay, _dev(W), scale_mode=mode)
    assert sq.sync_status() == 0
    W3 = W[:, None, :]
    s_ref = oracle.weight_scales(W3, perm, count, per_row=(mode == "row"))
    J = oracle.weight_codes(W3, perm, count, bits, s_ref)
    assert np.array_equal(s_w.cpu().numpy(), s_ref)
    assert np.array_equal(Wp.cpu().numpy(), oracle.pack_weight_rows(J, count, bits, 128))


@pytest.mark.parametrize("kind,sub_k,lo", [((1, 1), 0, 3), ((1, 0), 128, 3), ((0, 1), 256, 3), ((2, 1), 128, 1)])
@pytest.mark.parametrize("act_mode", ["tensor", "row"])
def test_variant_layouts_non_finite(sq, kind, sub_k, lo, act_mode):
    """Signed (Eq. (1)) and +-1 groups and scale runs: the run maxima skip NaN
    and keep infinities; signed codes of +-inf clip to the end levels under a
    finite scale, NaN codes to 0 (+-1 groups take -1 for NaN, as x >= 0 fails)."""
    d = wl.random_linear(1700 + 10 * kind[0] + kind[1] + sub_k, M=40, K=700, N=64, bits_lo=lo, bits_hi=6,
                         frac_hi=0.4)
    rng = np.random.default_rng(sub_k + kind[0])
    perm, count = d["perm"], d["count"]
    A = d["A"].copy()
    A = _plant(A, _cells(rng, A.shape[0], perm[:count[0]], 12), [NAN, INF, -INF])
    A[5, perm[count[0] + 3]] = NAN             # a finite-scale NaN in group 1
    W = d["W"].copy()
    W[2, perm[4]] = np.nan
    W[9, perm[count[0] + 1]] = np.nan
    W[11, perm[count[0] + 7]] = -np.inf         # row 11, group 1 (a run of it): scale inf
    lay = sq.Layout(perm, count, d["bits"], act_kind=kind, sub_k=sub_k)
    Wp, s_w = sq.pack_weights(lay, _dev(W))
    Ap, s_a = sq.quantize_act(lay, _dev(A), scale_mode=act_mode)
    assert sq.sync_status() == 0
    r = oracle.linear_variant(A, W, perm, count, d["bits"], d["bits"], kind=kind, sub_k=sub_k, act_mode=act_mode)
    s_a_ref = (r["s_a"] if sub_k else r["s_a"][..., 0]).reshape(tuple(s_a.shape))
    assert np.array_equal(s_a.cpu().numpy(), s_a_ref), "activation scales"
    assert np.array_equal(s_w.cpu().numpy(), r["s_w"].reshape(tuple(s_w.shape))), "weight scales"
    assert np.array_equal(Ap.cpu().numpy(), r["Ap"]), "packed activations"
    assert np.array_equal(Wp.cpu().numpy(), r["Wp"]), "packed weights"


def test_next_layer_codes_of_overflowed_outputs(sq):
    """Outputs beyond the fp16 range round to +-inf; the epilogue's next-layer
    codes of them are the top code and 0 under the calibrated scales, as the
    oracle's codes of those same fp16 outputs."""
    d = wl.random_linear(640, M=300, K=333, N=8, bits_lo=2, bits_hi=8, frac_hi=0.3)
    A = (d["A"].astype(np.float32) * 2000.0).astype(np.float16)
    K2 = 200
    lay2, perm2, count2 = _next_layout(sq, K2, [3, 6], 0.25, 32, seed=43)
    order = sq.next_layer_row_order(lay2)
    rng = np.random.default_rng(11)
    W = rng.standard_normal((K2, A.shape[1])).astype(np.float32)
    Wa = _arrange_rows(W, order)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(Wa))
    Ap, s_a = sq.quantize_act(lay, _dev(A))
    s2 = np.array([1.5, 40.0], np.float32)
    nxt = sq.NextLayer(lay2, _dev(s2), M=300)
    Y = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, next=nxt)
    assert sq.sync_status() == 0
    Y16 = Y.cpu().numpy()
    real = order >= 0
    assert np.isposinf(Y16[:, real]).any() and np.isneginf(Y16[:, real]).any()
    X2 = _to_channels(Y16, order, K2).astype(np.float32)
    U = oracle.act_codes(X2, perm2, count2, [3, 6], s2)
    assert np.array_equal(nxt.Ap.cpu().numpy(), oracle.pack_act_rows(U, count2, [3, 6], 32))
