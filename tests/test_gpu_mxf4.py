"""Groups of <= 2-bit codes on the block-scaled E2M1 tensor pipe
(tcgen05.mma kind::mxf4 with unit UE8M0 scales; E2M1 holds 0, 0.5, 1, 1.5, 2,
so a code c with |c| <= 4 is exact as c / 2 and the fp32 sums of the products
u j / 4 are exact), on the staged path with 240-column tiles.  Accumulators
bit for bit against the oracle's int64 sums (Sec. 3 / Sec. 4.2 decode), fp16
outputs within the output tolerance."""
import numpy as np
import pytest

import oracle
from helpers import assert_y_close
from paper_2311_14114_gb300 import workloads as wl
from test_gpu_parity import check_linear, _dev

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

STAGED = 2 | 8


@pytest.fixture(scope="module")
def sq():
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


@pytest.mark.parametrize("bits,frac", [((2, 8), 0.25), ((1, 8), 0.25), ((2, 4), 0.5), ((1, 2), 0.3),
                                       ((2, 2), 0.0), ((1, 6), 0.1), ((2, 6), 1.0), ((2, 4), 0.1)])
@pytest.mark.parametrize("shape", [(300, 2100, 470), (257, 3000, 465)])
def test_e2m1_groups(sq, bits, frac, shape):
    """Ragged M, K (groups not whole 256-code stages; K of at least 2048 codes,
    where the library takes E2M1) and N (two 240-column tiles, the second
    partial; widths that 240-column tiles would pad by more than 7 % keep
    E4M3)."""
    M, K, N = shape
    d = wl.random_linear(1300 + bits[0] + 10 * bits[1] + K, M=M, K=K, N=N, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=frac, n_outliers=2)
    check_linear(sq, d, flags=STAGED, what=f"e2m1 bits={bits} frac={frac} shape={shape}")


def test_e2m1_row_scales_and_bf16(sq):
    d = wl.random_linear(1350, M=200, K=2200, N=480, bits_lo=2, bits_hi=8, frac_hi=0.2)
    check_linear(sq, d, flags=STAGED, act_mode="row", what="e2m1 row scales")
    check_linear(sq, d, flags=STAGED, out_dtype=torch.bfloat16, what="e2m1 bf16")


def test_e2m1_sweep_shape_sampled_rows(sq):
    """The sweep point lo 2 / hi 8 / 25 % at full size (every column, sampled rows)."""
    spec = wl.LinearSpec("e2m1_sweep", M=8192, K=4096, N=4096, bits_lo=2, bits_hi=8, frac_hi=0.25)
    d = wl.make_linear(spec)
    check_linear(sq, d, rows=np.arange(0, 8192, 97), what="e2m1 sweep point")


@pytest.mark.parametrize("na,nw", [(2, 2), (1, 2), (2, 1), (1, 1)])
def test_e2m1_extreme_codes(sq, na, nw):
    """Every activation code at its top and weights alternating the extremes
    over K = 65536: |u j| up to 3 * 2 per product, sums up to 2^17.6 in one job."""
    K, M, N = 65536, 130, 470
    U = np.full((M, K), (1 << na) - 1, np.uint8)
    U[3, : K // 3] = 0
    J = np.empty((N, K), np.int8)
    J[0::2] = (1 << (nw - 1)) - 1
    J[1::2] = -(1 << (nw - 1))
    count = [K, 0]
    perm = np.arange(K, dtype=np.int32)
    lay = sq.Layout(perm, count, [nw, 1], [na, 1], pad_unit=128)
    Ap = _dev(oracle.pack_act_rows(U, count, [na, 1], 128))
    Wp = _dev(oracle.pack_weight_rows(J, count, [nw, 1], 128))
    s_a = np.array([1.0, 0.5], np.float32)
    s_w = np.tile(np.array([[0.25, 0.125]], np.float32), (N, 1))
    acc = torch.zeros((2, M, N), dtype=torch.int32, device="cuda")
    Y = sq.mp_gemm(lay, Ap, _dev(s_a), Wp, _dev(s_w), acc_dbg=acc, flags=STAGED)
    assert sq.sync_status() == 0
    r_acc = oracle.gemm_acc(U, J, count)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), r_acc)
    terms = oracle.epilogue_terms(r_acc, s_a, s_w, [na, 1], [nw, 1])
    assert_y_close(Y.float().cpu().numpy(), oracle.epilogue(r_acc, s_a, s_w, [na, 1], [nw, 1]).astype(np.float16),
                   terms, f"e2m1 extremes {na}/{nw}")

