"""Worst-case exactness of the integer dot products on the floating-point
tensor pipes (Sec. 3 "Enabling Low-Cost Fixed-Point Operations": integer-only
MACs; Sec. 4.2: unsigned x signed products into int32).

Groups whose codes are at most 4 bits wide run on the E4M3 pipe and
accumulate in fp32.  These tests drive every product to its largest
magnitude over the longest supported K (65536 codes), and drive partial sums
with random low bits through 2^20 ... 2^24 inside a K-chunk, so that any
accumulation narrower than fp32, or any rounding of a partial sum, shows up as
an accumulator that differs from the oracle's exact int64 sum.

The codes are chosen directly (the quantizer is tested elsewhere) and packed
by the oracle; the GPU accumulators (``acc_dbg``) and fp16 outputs are
compared with ``oracle.gemm_acc`` / ``oracle.epilogue`` bit for bit and within
the output tolerance."""
import numpy as np
import pytest

import oracle
from helpers import assert_y_close

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sq():
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _run_codes(sq, U, J, count, bits_a, bits_w, flags):
    """GEMM of given codes (U [M][K] uint8, J [N][K] int8, packed-position
    order) through the C-ABI; returns (gpu acc int64, gpu Y, oracle acc, oracle Y16, terms)."""
    M, K = U.shape
    N = J.shape[0]
    perm = np.arange(K, dtype=np.int32)
    lay = sq.Layout(perm, count, bits_w, bits_a, pad_unit=128)
    Ap = _dev(oracle.pack_act_rows(U, count, bits_a, 128))
    Wp = _dev(oracle.pack_weight_rows(J, count, bits_w, 128))
    s_a = np.array([1.0, 0.5], np.float32)
    s_w = np.tile(np.array([[0.25, 0.125]], np.float32), (N, 1))
    acc = torch.zeros((2, M, N), dtype=torch.int32, device="cuda")
    Y = sq.mp_gemm(lay, Ap, _dev(s_a), Wp, _dev(s_w), acc_dbg=acc, flags=flags)
    assert sq.sync_status() == 0
    r_acc = oracle.gemm_acc(U, J, count)
    y64 = oracle.epilogue(r_acc, s_a, s_w, bits_a, bits_w)
    terms = oracle.epilogue_terms(r_acc, s_a, s_w, bits_a, bits_w)
    return acc.cpu().numpy().astype(np.int64), Y.float().cpu().numpy(), r_acc, y64.astype(np.float16), terms


def _max_codes(M, N, K, na, nw):
    """Every activation code at its top, 2^na - 1; weight rows alternate the
    largest positive and the most negative code, so that the products are the
    extremes of both signed and offset-binary encodings."""
    U = np.full((M, K), (1 << na) - 1, np.uint8)
    J = np.empty((N, K), np.int8)
    J[0::2] = (1 << (nw - 1)) - 1
    J[1::2] = -(1 << (nw - 1))
    return U, J


PATHS = pytest.mark.parametrize("flags", [2 | 8, 2 | 4], ids=["staged", "fused"])


@PATHS
@pytest.mark.parametrize("na,nw", [(4, 4), (3, 4), (4, 3), (2, 4)])
@pytest.mark.parametrize("K", [65536, 65536 - 128 + 37])
def test_e4m3_group_all_extreme_products(sq, na, nw, K, flags):
    M, N = 130, 136                        # two row tiles and two column tiles, both ragged
    U, J = _max_codes(M, N, K, na, nw)
    U[5, : K // 3] = 0                     # a row whose sum stops growing early
    g_acc, g_y, r_acc, y16, terms = _run_codes(sq, U, J, [K, 0], [na, 1], [nw, 1], flags=flags)
    assert np.abs(r_acc).max() == K * ((1 << na) - 1) * (1 << (nw - 1))
    assert np.array_equal(g_acc, r_acc)
    assert_y_close(g_y, y16, terms, f"extreme E4M3 na={na} nw={nw} K={K}")


@PATHS
@pytest.mark.parametrize("K", [65536, 40000])
def test_e4m3_partial_sums_cross_2_20_to_2_24_mid_chunk(sq, K, flags):
    """Random codes from the top of the range: partial sums grow by about 100
    per code and carry random low bits, crossing 2^20, 2^21, ..., 2^24 at
    arbitrary points inside 128-code chunks."""
    rng = np.random.default_rng(11)
    M, N = 128, 256
    U = rng.integers(9, 16, size=(M, K), dtype=np.uint8)
    J = np.empty((N, K), np.int8)
    J[: N // 2] = rng.integers(4, 8, size=(N // 2, K), dtype=np.int8)      # positive sums
    J[N // 2:] = rng.integers(-8, -5, size=(N - N // 2, K), dtype=np.int8)  # negative sums
    g_acc, g_y, r_acc, y16, terms = _run_codes(sq, U, J, [K, 0], [4, 1], [4, 1], flags=flags)
    big = np.abs(r_acc[0])
    if K == 65536:
        assert big.max() > 2 ** 22
    assert np.array_equal(g_acc, r_acc)
    assert_y_close(g_y, y16, terms, f"E4M3 crossing K={K}")


@PATHS
def test_e4m3_and_fp16_groups_both_extreme(sq, flags):
    """A 4-bit group and an 8-bit group side by side, both at their extremes
    over a long K: the 8-bit group needs exact segments, the 4-bit one runs
    unsegmented on the E4M3 pipe."""
    K0, K1 = 32768, 8192
    K = K0 + K1
    M, N = 129, 130
    U = np.empty((M, K), np.uint8)
    U[:, :K0] = 15
    U[:, K0:] = 255
    J = np.empty((N, K), np.int8)
    J[0::2, :K0] = 7
    J[1::2, :K0] = -8
    J[0::2, K0:] = -128
    J[1::2, K0:] = 127
    g_acc, g_y, r_acc, y16, terms = _run_codes(sq, U, J, [K0, K1], [4, 8], [4, 8], flags=flags)
    assert np.abs(r_acc[1]).max() > 2 ** 24
    assert np.array_equal(g_acc, r_acc)
    assert_y_close(g_y, y16, terms, "E4M3 + fp16 extremes")
