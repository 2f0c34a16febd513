"""soniq_quantize_act_oneshot: the per-tensor activation quantize for callers
that cannot allocate device memory or pass the library any of their own (for
example code that is handed only the layer's tensors by a runtime whose
allocator it cannot reach, or a real-time loop where cudaMalloc and the
synchronization it may bring are not allowed).  It keeps its grid barrier and
per-CTA maxima in a fixed static array of the library instead.

These tests call it through the C-ABI (the ctypes binding) and check that:
  * two calls in a row give the same scales and packed bytes as the existing
    entry point soniq_quantize_act in per-tensor mode (bit for bit, the
    tolerance every packed-byte test here uses), and as the CPU oracle;
  * inputs too large for its fixed on-chip staging are refused with
    SONIQ_ERR_UNSUPPORTED before anything runs;
  * a barrier wait that runs out (armed by a test hook on the host, no GPU
    fault) is reported by soniq_sync_status, which resets the shared barrier,
    so the next call is exact again.

This file is collected last, so that a run stopping at its first failure has
run every other test before it."""
import dataclasses

import numpy as np
import pytest

import oracle
from paper_2311_14114_gb300 import workloads as wl

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def sq():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2311_14114_gb300 import build, soniq
    build.build()
    soniq.lib()
    return soniq


def _dev(x):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _oracle_bytes(d, rows, pad):
    A32 = rows.astype(np.float32)
    s = oracle.act_scales(A32, d["perm"], d["count"])
    U = oracle.act_codes(A32, d["perm"], d["count"], d["bits"], s)
    return s, oracle.pack_act_rows(U, d["count"], d["bits"], pad)


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
def test_oneshot_matches_the_oracle(sq):
    d = wl.random_linear(31, M=1000, K=700, N=8, bits_lo=3, bits_hi=8, frac_hi=0.3, n_outliers=3)
    lay = sq.Layout(d["perm"], d["count"], d["bits"], pad_unit=32)
    for _ in range(2):
        Ap, s_a = sq.quantize_act_oneshot(lay, _dev(d["A"]))
        assert sq.sync_status() == 0
        s_ref, Ap_ref = _oracle_bytes(d, d["A"], 32)
        assert np.array_equal(s_a.cpu().numpy(), s_ref)
        assert np.array_equal(Ap.cpu().numpy(), Ap_ref)


@pytest.mark.gpu
def test_oneshot_refuses_inputs_that_do_not_fit(sq):
    d = wl.random_linear(3, M=4096, K=4096, N=8, bits_lo=2, bits_hi=8, frac_hi=0.25)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    with pytest.raises(sq.SoniqError) as ei:
        sq.quantize_act_oneshot(lay, _dev(d["A"]))
    assert ei.value.status == sq.SONIQ_ERR_UNSUPPORTED


@pytest.mark.gpu
def test_oneshot_recovers_after_a_barrier_timeout(sq):
    d = wl.random_linear(32, M=3000, K=512, N=8, bits_lo=2, bits_hi=8, frac_hi=0.25, n_outliers=2)
    lay = sq.Layout(d["perm"], d["count"], d["bits"])
    A = _dev(d["A"])
    assert sq.sync_status() == 0
    sq.test_drop_barrier_arrival(True)         # one CTA skips its arrival: the others' waits run out
    sq.quantize_act_oneshot(lay, A)
    assert sq.sync_status() == sq.SONIQ_ERR_TIMEOUT
    assert sq.sync_status() == 0
    s_ref, Ap_ref = _oracle_bytes(d, d["A"], 128)
    for _ in range(2):
        Ap, s_a = sq.quantize_act_oneshot(lay, A)
        assert sq.sync_status() == 0
        assert np.array_equal(s_a.cpu().numpy(), s_ref)
        assert np.array_equal(Ap.cpu().numpy(), Ap_ref)
