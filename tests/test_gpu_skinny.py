"""The skinny swap-AB tensor-core kernel (M <= 32 activation rows; the weight
rows are the MMA's 128-row side and are converted from their packed form on
chip) against the oracle: packed bytes, scales and int32 accumulators bit for
bit, fp16 outputs within the output tolerance (Sec. 3 / Sec. 4.2 products and
decode rules, as for every other path).

The E4M3 groups run with offset-binary weights (j + 2^(n-1)) and take
2^(n-1) * sum(u) back per activation row; the fp16 groups run in exact
segments drained through a TMEM ring of 8 regions.  The extreme-code tests
drive both to their largest magnitudes, with enough segments to wrap the
ring twice."""
import numpy as np
import pytest

import oracle
from helpers import assert_y_close
from paper_2311_14114_gb300 import workloads as wl
from test_gpu_parity import check_linear, _dev

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

SKINNY = 16


@pytest.fixture(scope="module")
def sq():
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


@pytest.mark.parametrize("M", [1, 2, 5, 12, 16, 17, 31, 32])
@pytest.mark.parametrize("bits", [(3, 6), (2, 8), (4, 4), (1, 8)])
def test_skinny_parity(sq, M, bits):
    """Ragged K (333 channels over two groups) and ragged N (three row tiles,
    the last one short)."""
    d = wl.random_linear(900 + M + 10 * bits[0], M=M, K=333, N=300, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=0.3, n_outliers=2)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    assert sq.gemm_path(lay, M, 300, SKINNY).startswith("tensor-core skinny")
    check_linear(sq, d, flags=SKINNY, what=f"skinny M={M} bits={bits}")


@pytest.mark.parametrize("bits", [(5, 7), (4, 8), (1, 1), (8, 8)])
def test_skinny_other_bit_pairs(sq, bits):
    d = wl.random_linear(950 + bits[0], M=9, K=1000, N=257, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=0.25, n_outliers=2)
    check_linear(sq, d, flags=SKINNY, what=f"skinny bits={bits}")


def test_skinny_mixed_activation_and_weight_bits(sq):
    """Activation and weight widths differ per group (one group E4M3, one fp16)."""
    d = wl.random_linear(960, M=7, K=700, N=200, bits_lo=3, bits_hi=8, frac_hi=0.3)
    check_linear(sq, d, flags=SKINNY, bits_a=[4, 6], what="skinny mixed widths")


def test_skinny_row_scales_and_bf16(sq):
    d = wl.random_linear(961, M=20, K=512, N=384, bits_lo=2, bits_hi=8, frac_hi=0.2)
    check_linear(sq, d, flags=SKINNY, act_mode="row", what="skinny row scales")
    check_linear(sq, d, flags=SKINNY, out_dtype=torch.bfloat16, what="skinny bf16")


def test_skinny_single_group(sq):
    d = wl.random_linear(962, M=16, K=640, N=130, bits_lo=3, bits_hi=6, frac_hi=1.0)
    check_linear(sq, d, flags=SKINNY, what="skinny one group (fp16)")
    d = wl.random_linear(963, M=16, K=640, N=130, bits_lo=3, bits_hi=6, frac_hi=0.0)
    check_linear(sq, d, flags=SKINNY, what="skinny one group (E4M3)")


@pytest.mark.parametrize("M", [1, 4, 16])
def test_skinny_decode_full_size(sq, M):
    """The decode layer (N = 11008, K = 4096, 3/6 bits), every output."""
    spec = wl.DECODE[M]
    d = wl.make_linear(spec)
    check_linear(sq, d, flags=SKINNY, what=f"skinny decode M={M}")


def test_default_dispatch(sq):
    d = wl.random_linear(964, M=16, K=1000, N=333, bits_lo=3, bits_hi=6, frac_hi=0.15)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    assert sq.gemm_path(lay, 12, 333) == "CUDA-core GEMV"
    for M in (13, 16, 32):
        assert sq.gemm_path(lay, M, 333).startswith("tensor-core skinny")
    assert not sq.gemm_path(lay, 33, 333).startswith("tensor-core skinny")
    # pad-32 layouts whose activation groups are not 128-code chunks take another kernel
    lay32 = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    assert not sq.gemm_path(lay32, 16, 333).startswith("tensor-core skinny")
    check_linear(sq, d, pad=32, what="pad-32 layout at M = 16")


def _run_codes(sq, U, J, count, bits_a, bits_w):
    M, K = U.shape
    N = J.shape[0]
    perm = np.arange(K, dtype=np.int32)
    lay = sq.Layout(perm, count, bits_w, bits_a, pad_unit=128)
    Ap = _dev(oracle.pack_act_rows(U, count, bits_a, 128))
    Wp = _dev(oracle.pack_weight_rows(J, count, bits_w, 128))
    s_a = np.array([1.0, 0.5], np.float32)
    s_w = np.tile(np.array([[0.25, 0.125]], np.float32), (N, 1))
    acc = torch.zeros((2, M, N), dtype=torch.int32, device="cuda")
    Y = sq.mp_gemm(lay, Ap, _dev(s_a), Wp, _dev(s_w), acc_dbg=acc, flags=SKINNY)
    assert sq.sync_status() == 0
    r_acc = oracle.gemm_acc(U, J, count)
    y64 = oracle.epilogue(r_acc, s_a, s_w, bits_a, bits_w)
    terms = oracle.epilogue_terms(r_acc, s_a, s_w, bits_a, bits_w)
    return acc.cpu().numpy().astype(np.int64), Y.float().cpu().numpy(), r_acc, y64.astype(np.float16), terms


@pytest.mark.parametrize("na,nw", [(4, 4), (3, 4), (4, 2), (1, 1)])
def test_skinny_e4m3_extreme_codes(sq, na, nw):
    """Every activation code at its top and weights alternating the extremes
    over K = 65536: offset-binary products up to 15 * 15 and sums up to
    about 2^23.8 in one unsegmented fp32 job."""
    K, M, N = 65536, 16, 136
    U = np.full((M, K), (1 << na) - 1, np.uint8)
    U[3, : K // 3] = 0
    J = np.empty((N, K), np.int8)
    J[0::2] = (1 << (nw - 1)) - 1
    J[1::2] = -(1 << (nw - 1))
    g_acc, g_y, r_acc, y16, terms = _run_codes(sq, U, J, [K, 0], [na, 1], [nw, 1])
    assert np.array_equal(g_acc, r_acc)
    assert_y_close(g_y, y16, terms, f"skinny extreme E4M3 {na}/{nw}")


def test_skinny_fp16_segments_wrap_the_ring(sq):
    """An 8-bit group of 16384 codes at its extremes: 16 exact segments of 1024
    codes through 8 TMEM regions, beside a 4-bit E4M3 group at its extremes."""
    K0, K1 = 8192, 16384
    K, M, N = K0 + K1, 16, 130
    U = np.empty((M, K), np.uint8)
    U[:, :K0] = 15
    U[:, K0:] = 255
    U[1::2, K0:] = 0                      # rows whose centred fp16 values sit at the other extreme
    J = np.empty((N, K), np.int8)
    J[0::2, :K0] = 7
    J[1::2, :K0] = -8
    J[0::2, K0:] = -128
    J[1::2, K0:] = 127
    g_acc, g_y, r_acc, y16, terms = _run_codes(sq, U, J, [K0, K1], [4, 8], [4, 8])
    assert np.abs(r_acc[1]).max() > 2 ** 21
    assert np.array_equal(g_acc, r_acc)
    assert_y_close(g_y, y16, terms, "skinny segmented fp16 group")


def test_skinny_timeout_is_reported_and_context_survives(sq):
    d = wl.random_linear(970, M=16, K=1000, N=256, bits_lo=3, bits_hi=6, frac_hi=0.25)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    assert sq.sync_status() == 0
    sq.mp_gemm(lay, Ap, s_a, Wp, s_w, flags=SKINNY | sq.FLAG_TEST_DROP_ARRIVE)
    assert sq.sync_status() == 5            # SONIQ_ERR_TIMEOUT, then cleared
    assert sq.sync_status() == 0
    check_linear(sq, d, flags=SKINNY, what="skinny after timeout")
