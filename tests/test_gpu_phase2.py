"""Phase II forward (Algorithm 1, Phase II: quantize the fp32 master weights
and the activations with per-group scales on the fly, then evaluate the
layers with integer MACs) against the oracle, layer by layer: each layer's
packed weights, scales and packed activations bit for bit and its fp16
outputs within the output tolerance.  The oracle takes the GPU's previous
fp16 output as the layer input, so the layers are checked independently of
one-ulp differences upstream.  A master-weight update between steps must
reach the next step's codes."""
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


def _check_layers(net, X, layers, sub_k=0, rows=None):
    x = X
    for i, lay in enumerate(layers):
        W = net.W[i].cpu().numpy()
        if sub_k:
            r = oracle.linear_variant(x, W, lay["perm"], lay["count"], lay["bits"], lay["bits"], sub_k=sub_k,
                                      rows=rows)
            s_a_ref, s_w_ref, terms = r["s_a"].reshape(2, -1), r["s_w"], r["terms"]
        else:
            r = oracle.linear(x, W, lay["perm"], lay["count"], lay["bits"], lay["bits"], rows=rows)
            s_a_ref, s_w_ref = r["s_a"], r["s_w"]
            terms = oracle.epilogue_terms(r["acc"], r["s_a"], r["s_w"], lay["bits"], lay["bits"], rows=rows)
        assert np.array_equal(net.s_w[i].cpu().numpy(), s_w_ref.reshape(net.s_w[i].shape)), f"layer {i} s_w"
        assert np.array_equal(net.Wp[i].cpu().numpy(), r["Wp"]), f"layer {i} packed weights"
        assert np.array_equal(net.s_a[i].cpu().numpy(), s_a_ref.reshape(net.s_a[i].shape)), f"layer {i} s_a"
        assert np.array_equal(net.Ap[i].cpu().numpy(), r["Ap"]), f"layer {i} packed activations"
        Y = net.Y[i].cpu().numpy()
        sel = slice(None) if rows is None else rows
        assert_y_close(Y[sel].astype(np.float64), r["Y64"].astype(np.float16), terms, f"layer {i} outputs")
        x = Y


def _small():
    rng = np.random.default_rng(12)
    widths = (300, 520, 264, 130)
    bits = [(2, 8), (3, 6), (4, 8)]
    layers = []
    for (K, N), b in zip(zip(widths[:-1], widths[1:]), bits):
        perm, count, _ = wl.assignment(rng, K, 0.25, 0)
        layers.append(dict(W=(rng.standard_normal((N, K)) * 0.08).astype(np.float32), perm=perm, count=count,
                           bits=list(b)))
    X = rng.standard_normal((77, widths[0])).astype(np.float16)
    return X, layers


@pytest.mark.parametrize("sub_k", [0, 128])
def test_phase2_forward_layers_match_oracle(sq, sub_k):
    from paper_2311_14114_gb300.phase2 import FakeQuantMLP
    X, layers = _small()
    net = FakeQuantMLP(layers, M=X.shape[0], sub_k=sub_k)
    out = net.forward(torch.from_numpy(X).cuda())
    assert sq.sync_status() == 0
    assert out.data_ptr() == net.Y[-1].data_ptr()
    _check_layers(net, X, layers, sub_k=sub_k)


def test_phase2_master_weight_update_reaches_the_codes(sq):
    """Quantize on the fly: after an update of the fp32 master weights (outside
    the path, as the optimizer of Phase II), the next forward packs the new
    weights."""
    from paper_2311_14114_gb300.phase2 import FakeQuantMLP
    X, layers = _small()
    net = FakeQuantMLP(layers, M=X.shape[0])
    Xd = torch.from_numpy(X).cuda()
    net.forward(Xd)
    before = [w.clone() for w in net.Wp]
    g = torch.Generator(device="cuda").manual_seed(3)
    for W in net.W:
        W.sub_(0.01 * torch.randn(W.shape, generator=g, device="cuda"))
    net.forward(Xd)
    assert sq.sync_status() == 0
    assert all(not torch.equal(a, b) for a, b in zip(before, net.Wp))
    _check_layers(net, X, layers)


def test_phase2_mlp_full_size_sampled_rows(sq):
    """The bench's MLP block (2048 tokens, 4096 -> 11008 -> 4096, 3/6 bits):
    every packed byte and scale, outputs on sampled rows."""
    from paper_2311_14114_gb300.phase2 import FakeQuantMLP
    spec = wl.PHASE2_MLP
    d = wl.make_phase2(spec)
    net = FakeQuantMLP(d["layers"], M=spec.M)
    net.forward(torch.from_numpy(d["X"]).cuda())
    assert sq.sync_status() == 0
    _check_layers(net, d["X"], d["layers"], rows=np.arange(0, spec.M, 37))


@pytest.mark.parametrize("bits", [(2, 8), (3, 6), (4, 5)])
def test_weight_codes_at_rounding_boundaries(sq, bits):
    """Weights on and beside every half-integer boundary of w / s * 2^(n-1)
    (exact ties, and a few ulps either side): the packed codes equal the
    oracle's, which divides with IEEE rounding (Eq. (1), ties to even)."""
    rng = np.random.default_rng(bits[0])
    K, N = 512, 64
    perm, count, _ = wl.assignment(rng, K, 0.5, 0)
    W = np.zeros((N, K), np.float32)
    for n in range(N):
        s = np.float32(rng.uniform(0.01, 3.0))
        for g, (lo, cnt) in enumerate(((0, count[0]), (count[0], count[1]))):
            half = 1 << (bits[g] - 1)
            ks = rng.integers(-half, half, cnt)
            base = (ks + 0.5).astype(np.float64) * float(s) / half
            v = base.astype(np.float32)
            nudge = rng.integers(-3, 4, cnt).astype(np.int32)
            v = (v.view(np.int32) + nudge).view(np.float32)            # ties and near-ties
            cols = perm[lo:lo + cnt]
            W[n, cols] = v
        W[n, perm[0]] = s                                                # group 0 max |w| = s
        W[n, perm[count[0]]] = -s                                        # group 1 max |w| = s
    lay = sq.Layout(perm, count, list(bits))
    Wp, s_w = sq.pack_weights(lay, torch.from_numpy(W).cuda())
    assert sq.sync_status() == 0
    s_ref = oracle.weight_scales(W, perm, count)
    J = oracle.weight_codes(W, perm, count, list(bits), s_ref)
    assert np.array_equal(s_w.cpu().numpy(), s_ref)
    assert np.array_equal(Wp.cpu().numpy(), oracle.pack_weight_rows(J, count, list(bits), 128))
