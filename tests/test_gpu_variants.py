"""Layout variants on the GPU (staged tensor-core path) against the oracle:
signed activations (Eq. (1) applied to activations), one-bit +-1 groups
(Sec. 4.2 XNOR / POPCOUNT semantics), and scale runs along K (each run of
sub_k codes with its own scales and its own exact accumulator).  Scales and
packed bytes bit for bit, accumulators bit for bit (per run with sub_k),
fp16 outputs within the output tolerance."""
import numpy as np
import pytest

import oracle
from helpers import assert_y_close
from paper_2311_14114_gb300 import workloads as wl

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


def run_variant(sq, d, kind, sub_k, act_mode="tensor", rows=None):
    bits = d["bits"]
    lay = sq.Layout(d["perm"], d["count"], bits, act_kind=kind, sub_k=sub_k)
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]), scale_mode=act_mode)
    M, N = d["A"].shape[0], d["W"].shape[0]
    nb = lay.scale_runs()
    acc = torch.zeros((2, nb, M, N) if sub_k else (2, M, N), dtype=torch.int32, device="cuda")
    assert sq.gemm_path(lay, M, N).startswith("tensor-core staged")
    Y = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, scale_mode=act_mode, acc_dbg=acc)
    assert sq.sync_status() == 0
    r = oracle.linear_variant(d["A"], d["W"], d["perm"], d["count"], bits, bits, kind=kind, sub_k=sub_k,
                              act_mode=act_mode, rows=rows)
    sel = slice(None) if rows is None else rows
    s_a_ref = r["s_a"] if sub_k else r["s_a"][..., 0]
    s_a_ref = s_a_ref.reshape(tuple(s_a.shape))
    assert np.array_equal(s_a.cpu().numpy(), s_a_ref), "activation scales"
    assert np.array_equal(s_w.cpu().numpy(), r["s_w"].reshape(tuple(s_w.shape))), "weight scales"
    assert np.array_equal(Ap.cpu().numpy(), r["Ap"]), "packed activations"
    assert np.array_equal(Wp.cpu().numpy(), r["Wp"]), "packed weights"
    g_acc = acc.cpu().numpy().astype(np.int64)
    g_acc = g_acc[:, :, sel] if sub_k else g_acc[:, None, sel]
    assert np.array_equal(g_acc, r["acc"]), "run accumulators"
    assert_y_close(Y.float().cpu().numpy()[sel], r["Y64"].astype(np.float16), r["terms"],
                   f"variant kind={kind} sub_k={sub_k}")
    return r


@pytest.mark.parametrize("bits", [(4, 8), (3, 6), (2, 5), (1, 4)])
@pytest.mark.parametrize("act_mode", ["tensor", "row"])
def test_signed_activations(sq, bits, act_mode):
    d = wl.random_linear(1100 + bits[0], M=300, K=333, N=264, bits_lo=bits[0], bits_hi=bits[1], frac_hi=0.3,
                         n_outliers=2)
    r = run_variant(sq, d, (1, 1), 0, act_mode)
    assert (r["U"] < 0).any()


@pytest.mark.parametrize("bits,kind", [((1, 8), (2, 0)), ((1, 1), (2, 2)), ((1, 4), (2, 1)), ((3, 1), (0, 2))])
def test_pm1_groups(sq, bits, kind):
    d = wl.random_linear(1120 + bits[1], M=200, K=700, N=130, bits_lo=bits[0], bits_hi=bits[1], frac_hi=0.4)
    run_variant(sq, d, kind, 0)


@pytest.mark.parametrize("bits,kind,sub_k", [((4, 8), (0, 0), 128), ((2, 8), (1, 1), 256), ((1, 4), (2, 0), 128),
                                             ((3, 6), (0, 1), 384), ((4, 4), (0, 0), 512)])
@pytest.mark.parametrize("act_mode", ["tensor", "row"])
def test_scale_runs(sq, bits, kind, sub_k, act_mode):
    d = wl.random_linear(1140 + bits[0] + sub_k, M=257, K=1333, N=300, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=0.35, n_outliers=3)
    run_variant(sq, d, kind, sub_k, act_mode)


def test_scale_runs_large(sq):
    """A 2048 x 1024 x 4096 layer with 128-code runs (24 runs in the 4-bit group,
    8 in the 8-bit group per tile), sampled rows."""
    spec = wl.LinearSpec("runs", M=2048, K=4096, N=1024, bits_lo=4, bits_hi=8, frac_hi=0.25)
    d = wl.make_linear(spec)
    run_variant(sq, d, (0, 0), 128, rows=np.arange(0, 2048, 61))


def test_variant_errors(sq):
    d = wl.random_linear(1160, M=16, K=256, N=64, bits_lo=2, bits_hi=8, frac_hi=0.5)
    with pytest.raises(sq.SoniqError):                      # +-1 needs one-bit codes
        sq.Layout(d["perm"], d["count"], d["bits"], act_kind=(2, 0))
    with pytest.raises(sq.SoniqError):                      # runs are multiples of 128 codes
        sq.Layout(d["perm"], d["count"], d["bits"], sub_k=100)
    with pytest.raises(sq.SoniqError):                      # linear layers only (pad unit 128)
        sq.Layout(d["perm"], d["count"], d["bits"], act_kind=(1, 1), pad_unit=32)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], act_kind=(1, 1))
    with pytest.raises(sq.SoniqError) as ei:                 # weight scales per row only
        sq.pack_weights(lay, _dev(d["W"]), scale_mode="tensor")
    assert ei.value.status == sq.SONIQ_ERR_UNSUPPORTED
    with pytest.raises(sq.SoniqError) as ei:
        sq.quantize_act_oneshot(lay, _dev(d["A"]).half())
    assert ei.value.status == sq.SONIQ_ERR_UNSUPPORTED
    # 8-bit runs of 1024 codes could pass 2^24: refused
    lay = sq.Layout(d["perm"], d["count"], [8, 8], sub_k=1024)
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    with pytest.raises(sq.SoniqError) as ei:
        sq.mp_gemm(lay, Ap, s_a, Wp, s_w)
    assert ei.value.status == sq.SONIQ_ERR_UNSUPPORTED
    # convolutions keep the default layout
    lay = sq.Layout(d["perm"], d["count"], d["bits"], act_kind=(1, 1))
    X = _dev(np.zeros((1, 4, 4, 256), np.float16)).reshape(-1, 256)
    Xp, sx = sq.quantize_act(lay, X)
    cd = sq.conv_desc(1, 4, 4, 64, 1, 1, (1, 1), (0, 0))
    with pytest.raises(sq.SoniqError) as ei:
        sq.mp_conv2d(lay, cd, Xp, sx, Wp, s_w)
    assert ei.value.status == sq.SONIQ_ERR_UNSUPPORTED
    assert sq.sync_status() == 0
