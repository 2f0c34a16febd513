"""The lean epilogue of the staged tensor-core path: the kernel that runs when
no debug accumulators are requested.  On 256-column tiles with rows of at
least 3072 codes it is the 2-SM CTA-pair kernel (M = 256 MMAs over two CTAs'
shared-memory stages, each CTA's TMEM holding its own 128 rows); on shorter
rows, one CTA per tile.

Each case runs one layer twice, with and without `acc_dbg`.  Both epilogues
evaluate the same fp32 expression from the same exact integer group sums
(Sec. 3, "Enabling Low-Cost Fixed-Point Operations"), so the two outputs are
compared bit for bit; the lean outputs are also compared with the oracle
within the output tolerance.  Shapes cover an odd number of 128-row tiles
(the last pair's second CTA lies past M), ragged N and K, a segmented fp16
group, per-row activation scales, bf16 outputs, the full headline layer and
the ResNet convolution."""
import numpy as np
import pytest

import oracle
from helpers import assert_y_close
from paper_2311_14114_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

STAGED = 2 | 8


@pytest.fixture(scope="module")
def sq():
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _bits16(y):
    return y.contiguous().view(torch.int16).cpu().numpy()


def run_both(sq, d, flags=STAGED, act_mode="tensor", out_dtype=torch.float16):
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]), scale_mode=act_mode)
    M, N = d["A"].shape[0], d["W"].shape[0]
    assert sq.gemm_path(lay, M, N, flags).startswith("tensor-core staged")
    acc = torch.zeros((2, M, N), dtype=torch.int32, device="cuda")
    y_gen = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, scale_mode=act_mode, acc_dbg=acc, flags=flags, out_dtype=out_dtype)
    y_lean = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, scale_mode=act_mode, flags=flags, out_dtype=out_dtype)
    assert sq.sync_status() == 0
    return y_gen, y_lean


def check_lean(sq, d, rows=None, act_mode="tensor", out_dtype=torch.float16, flags=STAGED, what=""):
    y_gen, y_lean = run_both(sq, d, flags, act_mode, out_dtype)
    assert np.array_equal(_bits16(y_gen), _bits16(y_lean)), what + ": lean and general outputs differ"
    bits = d["bits"]
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], bits, bits, act_mode=act_mode, rows=rows)
    sel = slice(None) if rows is None else rows
    y = y_lean.float().cpu().numpy()[sel]
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], bits, bits, rows=rows,
                                  s_a_per_row=(act_mode == "row"))
    if out_dtype == torch.bfloat16:
        tol = 2.0 ** -7 * np.maximum(np.abs(r["Y64"]), terms * 2.0 ** -10) + 1e-30
        assert (np.abs(y - r["Y64"]) <= tol).all(), what + " bf16 output"
    else:
        assert_y_close(y, r["Y64"].astype(np.float16), terms, what)


@pytest.mark.parametrize("shape,bits,frac", [
    # 2-SM pairs (rows of at least 3072 codes)
    ((300, 3333, 264), (4, 8), 0.3),     # 3 row tiles: the second pair's rank-1 CTA lies past M
    ((513, 3100, 1100), (3, 6), 0.5),    # 5 column tiles, the last 76 wide
    ((257, 4096, 512), (4, 4), 0.0),     # one E4M3 group over K = 4096
    ((384, 4096, 256), (8, 8), 1.0),     # one fp16 group in four exact segments
    # 2-SM pairs on E2M1 layouts (240-column tiles, 120-row B halves)
    ((300, 3333, 470), (2, 8), 0.25),    # E2M1 beside fp16, the second column tile partial
    ((257, 4096, 480), (1, 4), 0.0),     # one E2M1 group
    ((640, 3500, 960), (2, 4), 0.1),     # E2M1 beside E4M3
    # one CTA per tile (shorter rows)
    ((300, 333, 264), (4, 8), 0.3),
    ((1000, 1000, 600), (2, 8), 0.25),
    ((513, 700, 1100), (3, 6), 0.5),
    ((384, 2048, 256), (8, 8), 1.0),     # one fp16 group in two exact segments
    ((640, 1536, 768), (1, 8), 0.1),
])
def test_lean_matches_general_and_oracle(sq, shape, bits, frac):
    M, K, N = shape
    d = wl.random_linear(1500 + M + K, M=M, K=K, N=N, bits_lo=bits[0], bits_hi=bits[1], frac_hi=frac,
                         n_outliers=2)
    check_lean(sq, d, what=f"lean {shape} {bits} {frac}")


def test_lean_row_scales_and_bf16(sq):
    d = wl.random_linear(1560, M=520, K=900, N=520, bits_lo=4, bits_hi=8, frac_hi=0.2)
    check_lean(sq, d, act_mode="row", what="lean row scales")
    check_lean(sq, d, out_dtype=torch.bfloat16, what="lean bf16")


def test_lean_headline_layer(sq):
    """8192 x 4096 x 4096, 4/8 bits, 25 % high: every output against the general
    epilogue, sampled rows against the oracle."""
    spec = wl.LinearSpec("sweep", M=8192, K=4096, N=4096, bits_lo=4, bits_hi=8, frac_hi=0.25)
    d = wl.make_linear(spec)
    rng = np.random.default_rng(5)
    rows = np.unique(np.concatenate([[0, 127, 128, 255, 256, 8191], rng.choice(8192, 40, replace=False)]))
    check_lean(sq, d, rows=rows.astype(np.int64), flags=0, what="lean headline")


def test_lean_resnet_conv(sq):
    spec = wl.CONV_RESNET
    d = wl.make_conv(spec)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    X = _dev(d["X"]).reshape(-1, spec.C)
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Xp, s_a = sq.quantize_act(lay, X)
    cd = sq.conv_desc(spec.batch, spec.H, spec.W, spec.C_out, spec.R, spec.S, spec.stride, spec.pad)
    acc = torch.zeros((2, spec.M, spec.C_out), dtype=torch.int32, device="cuda")
    y_gen = sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, acc_dbg=acc, flags=STAGED)
    y_lean = sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, flags=STAGED)
    assert sq.sync_status() == 0
    assert np.array_equal(_bits16(y_gen), _bits16(y_lean)), "conv: lean and general outputs differ"
    pix = np.arange(0, spec.M, 97)
    r = oracle.conv2d(d["X"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], spec.R, spec.S,
                      stride=spec.stride, pad=spec.pad, pad_unit=32, pix=pix)
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], d["bits"], d["bits"])
    y = y_lean.float().cpu().numpy().reshape(spec.M, spec.C_out)[pix]
    assert_y_close(y, r["Y16"], terms, "lean conv")
