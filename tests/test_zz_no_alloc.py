"""soniq_quantize_act_oneshot: the per-tensor quantize entry point that uses only
fixed library scratch.  It must give the same scales and packed bytes as
soniq_quantize_act in per-tensor mode, call after call (its grid barrier is
reused without clearing), and refuse inputs that do not fit on chip."""
import dataclasses

import numpy as np
import pytest

from paper_2311_14114_gb300 import workloads as wl

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sq():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2311_14114_gb300 import soniq
    soniq.lib()
    return soniq


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


@pytest.mark.gpu
def test_oneshot_matches_quantize_act_on_two_calls_in_a_row(sq):
    spec = wl.CONV_RESNET
    first = wl.make_conv(spec)
    second = wl.make_conv(dataclasses.replace(spec, seed=7))
    lay = sq.Layout(first["perm"], first["count"], first["bits"], pad_unit=32)
    for d in (first, second):
        X = _dev(d["X"]).reshape(-1, spec.C)
        Ap_ref, s_ref = sq.quantize_act(lay, X, "tensor")
        Ap, s_a = sq.quantize_act_oneshot(lay, X)
        assert sq.sync_status() == 0
        assert np.array_equal(s_a.cpu().numpy(), s_ref.cpu().numpy())
        assert np.array_equal(Ap.cpu().numpy(), Ap_ref.cpu().numpy())


@pytest.mark.gpu
def test_oneshot_refuses_inputs_that_do_not_fit(sq):
    d = wl.random_linear(3, M=4096, K=4096, N=8, bits_lo=2, bits_hi=8, frac_hi=0.25)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    with pytest.raises(sq.SoniqError) as ei:
        sq.quantize_act_oneshot(lay, _dev(d["A"]))
    assert ei.value.status == sq.SONIQ_ERR_UNSUPPORTED
