"""Quantize-in-epilogue (Sec. 4.1: Conv2D + BatchNorm + Quantize fused on the
CPU back-end): a GEMM or convolution whose epilogue also writes the next
layer's packed activation codes with the next layer's calibrated scales.

Reading: the next layer quantizes the fp16 tensor this layer outputs, so each
output is rounded to fp16 before Sec. 3 step 2.  The GPU's fp16 outputs can
differ from the oracle's by one fp16 ulp where the fp32 and fp64 epilogues
round differently (the output tolerance allows that); a code can then differ
too.  The tests therefore check:
  * fused codes == soniq_quantize_act(calibrated) of the same call's own fp16
    outputs, bit for bit (the fused path reproduces the unfused one exactly);
  * fused codes == the oracle's codes of the oracle's fp16 outputs, for every
    32-code block all of whose 32 outputs agree with the oracle's; blocks with
    a differing output must be rare;
  * outputs and int32 accumulators against the oracle as everywhere else.
The layer's output columns are the next layer's packed positions (weights
arranged once by next_layer_row_order, zero rows at padding)."""
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


def _next_layout(sq, K2, bits2, frac2, pad2, seed):
    perm2, count2, _ = wl.assignment(np.random.default_rng(seed), K2, frac2, 0)
    return sq.Layout(perm2, count2, bits2, pad_unit=pad2), perm2, count2


def _arrange_rows(W, order):
    """Rows of W placed at the next layer's packed positions (zero rows at -1)."""
    Wa = np.zeros((len(order),) + W.shape[1:], dtype=W.dtype)
    Wa[order >= 0] = W[order[order >= 0]]
    return Wa


def _to_channels(Y16, order, K2):
    """The next layer's input in original channel order from packed-order outputs."""
    X2 = np.zeros((Y16.shape[0], K2), dtype=np.float16)
    X2[:, order[order >= 0]] = Y16[:, order >= 0]
    return X2


def _check_codes(sq, lay2, perm2, count2, bits2, pad2, s2, order, Ap2_gpu, Y16_gpu, Y16_ref, what):
    K2 = len(perm2)
    # the unfused path on the GPU's own outputs: identical bytes
    X2_gpu = _dev(_to_channels(Y16_gpu, order, K2))
    Ap_unfused, _ = sq.quantize_act(lay2, X2_gpu, "calibrated", s_a=_dev(s2))
    assert sq.sync_status() == 0
    assert np.array_equal(Ap2_gpu, Ap_unfused.cpu().numpy()), what + ": fused != unfused codes"
    # the oracle's codes of the oracle's outputs, block by block
    X2_ref = _to_channels(Y16_ref, order, K2).astype(np.float32)
    U = oracle.act_codes(X2_ref, perm2, count2, bits2, s2)
    Ap_ref = oracle.pack_act_rows(U, count2, bits2, pad2)
    same_y = (Y16_gpu.view(np.int16) == Y16_ref.view(np.int16))
    bad_blocks = 0
    off = 0
    for g in range(2):
        pa = lay2.group_codes(g)
        n = bits2[g]
        base = 0 if g == 0 else lay2.group_codes(0)
        for b in range(pa // 32):
            cols = slice(base + 32 * b, base + 32 * b + 32)
            byt = slice(off + 4 * n * b, off + 4 * n * (b + 1))
            differ = ~np.all(Ap2_gpu[:, byt] == Ap_ref[:, byt], axis=1)
            explained = ~np.all(same_y[:, cols], axis=1)
            assert not (differ & ~explained).any(), f"{what}: group {g} block {b} codes differ with equal outputs"
            bad_blocks += int(differ.sum())
        off += 4 * n * (pa // 32)
    assert bad_blocks <= max(2, Ap2_gpu.shape[0] // 50), f"{what}: {bad_blocks} blocks with differing outputs"


@pytest.mark.parametrize("bits2,pad2", [((2, 8), 128), ((3, 6), 32), ((4, 4), 32), ((1, 8), 128), ((5, 7), 32)])
def test_gemm_epilogue_writes_next_layer_codes(sq, bits2, pad2):
    d = wl.random_linear(600 + bits2[0], M=300, K=333, N=8, bits_lo=2, bits_hi=8, frac_hi=0.3, n_outliers=2)
    K2 = 200
    lay2, perm2, count2 = _next_layout(sq, K2, list(bits2), 0.25, pad2, seed=41 + bits2[1])
    order = sq.next_layer_row_order(lay2)
    rng = np.random.default_rng(7)
    W = (rng.standard_normal((K2, d["A"].shape[1])) * 0.05).astype(np.float32)
    Wa = _arrange_rows(W, order)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(Wa))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    s2 = np.array([0.9, 2.5], np.float32)                       # calibrated: some outputs clip
    nxt = sq.NextLayer(lay2, _dev(s2), M=300)
    acc = torch.zeros((2, 300, len(order)), dtype=torch.int32, device="cuda")
    Y = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, acc_dbg=acc, next=nxt)
    assert sq.sync_status() == 0
    r = oracle.linear(d["A"], Wa, d["perm"], d["count"], d["bits"], d["bits"])
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), r["acc"])
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], d["bits"], d["bits"])
    Y16 = Y.cpu().numpy()
    assert_y_close(Y16.astype(np.float64), r["Y16"], terms, "fused-quant GEMM outputs")
    _check_codes(sq, lay2, perm2, count2, list(bits2), pad2, s2, order, nxt.Ap.cpu().numpy(), Y16, r["Y16"],
                 f"gemm next {bits2} pad {pad2}")
    # without fp16 outputs the same codes come out
    nxt2 = sq.NextLayer(lay2, _dev(s2), M=300)
    sq.mp_gemm(lay, Ap, s_a, Wp, s_w, next=nxt2, write_y=False)
    assert sq.sync_status() == 0
    assert np.array_equal(nxt2.Ap.cpu().numpy(), nxt.Ap.cpu().numpy())


def test_gemm_epilogue_next_codes_large(sq):
    """The MLP up-projection shape feeding a 3072-channel next layer."""
    spec = wl.LinearSpec("mlp", M=2048, K=768, N=3072, bits_lo=2, bits_hi=8, frac_hi=0.2, n_outliers=8,
                         outlier_scale=20.0)
    d = wl.make_linear(spec)
    lay2, perm2, count2 = _next_layout(sq, 3072, [2, 8], 0.2, 128, seed=5)
    order = sq.next_layer_row_order(lay2)
    Wa = _arrange_rows(d["W"], order)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    Wp, s_w = sq.pack_weights(lay, _dev(Wa))
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    s2 = np.array([0.6, 1.8], np.float32)
    nxt = sq.NextLayer(lay2, _dev(s2), M=spec.M)
    Y = sq.mp_gemm(lay, Ap, s_a, Wp, s_w, next=nxt)
    assert sq.sync_status() == 0
    rows = np.arange(0, spec.M, 16)
    r = oracle.linear(d["A"], Wa, d["perm"], d["count"], d["bits"], d["bits"], rows=rows)
    Y16 = Y.cpu().numpy()
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], d["bits"], d["bits"], rows=rows)
    assert_y_close(Y16[rows].astype(np.float64), r["Y16"], terms, "mlp fused outputs")
    _check_codes(sq, lay2, perm2, count2, [2, 8], 128, s2, order, nxt.Ap.cpu().numpy()[rows], Y16[rows], r["Y16"],
                 "mlp next layer")


def test_conv_epilogue_writes_next_layer_codes(sq):
    spec = wl.ConvSpec("t", batch=3, H=9, W=7, C=70, C_out=40, R=3, S=3, stride=(1, 1), pad=(1, 1),
                       bits_lo=4, bits_hi=8, frac_hi=0.3, seed=3)
    d = wl.make_conv(spec)
    lay2, perm2, count2 = _next_layout(sq, 40, [2, 6], 0.3, 32, seed=9)
    order = sq.next_layer_row_order(lay2)
    Wa = _arrange_rows(d["W"], order)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    Wp, s_w = sq.pack_weights(lay, _dev(Wa))
    Xp, s_a = sq.quantize_act(lay, _dev(d["X"]).reshape(-1, spec.C))
    cd = sq.conv_desc(spec.batch, spec.H, spec.W, len(order))
    s2 = np.array([0.5, 1.5], np.float32)
    nxt = sq.NextLayer(lay2, _dev(s2), M=spec.M)
    Y = sq.mp_conv2d(lay, cd, Xp, s_a, Wp, s_w, next=nxt)
    assert sq.sync_status() == 0
    r = oracle.conv2d(d["X"], Wa, d["perm"], d["count"], d["bits"], d["bits"], 3, 3)
    Y16 = Y.cpu().numpy().reshape(spec.M, -1)
    terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], d["bits"], d["bits"])
    assert_y_close(Y16.astype(np.float64), r["Y16"], terms, "fused-quant conv outputs")
    _check_codes(sq, lay2, perm2, count2, [2, 6], 32, s2, order, nxt.Ap.cpu().numpy(), Y16, r["Y16"],
                 "conv next layer")


def test_next_layer_width_must_match(sq):
    d = wl.random_linear(610, M=300, K=128, N=100, bits_lo=2, bits_hi=8, frac_hi=0.3)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    lay2, _, _ = _next_layout(sq, 100, [2, 8], 0.3, 32, seed=1)
    Wp, s_w = sq.pack_weights(lay, _dev(d["W"]))                  # 100 rows, not the padded width
    Ap, s_a = sq.quantize_act(lay, _dev(d["A"]))
    nxt = sq.NextLayer(lay2, _dev(np.array([1.0, 1.0], np.float32)), M=300)
    with pytest.raises(sq.SoniqError) as ei:
        sq.mp_gemm(lay, Ap, s_a, Wp, s_w, next=nxt)
    assert ei.value.status == sq.SONIQ_ERR_INVALID_ARG
