"""Pins of the oracle's variant functions (signed activations by Eq. (1),
one-bit +-1 groups whose dot products are XNOR / POPCOUNT, and scale
sub-groups along K), each against a statement that does not reuse the
function's own formula: the Eq. (1) argmin over the level set, the popcount
identity of +-1 vectors, the reduction to the default path when a group has
one run, numpy maxima per run, and the fp64 matmul of dequantized values."""
import numpy as np
import pytest

import oracle
from paper_2311_14114_gb300 import workloads as wl


def _argmin_eq1(x: float, s: float, n: int) -> int:
    """Nearest level j / 2^(n-1), j in [-2^(n-1), 2^(n-1) - 1], to x / s (fp32
    quotient), ties to the even j; by enumeration of the level set."""
    if not s > 0:
        return 0
    q = np.float32(np.float32(x) / np.float32(s))
    best, bj = None, None
    for j in range(-(1 << (n - 1)), 1 << (n - 1)):
        d = abs(float(q) - j / float(1 << (n - 1)))
        if best is None or d < best - 1e-15 or (abs(d - best) <= 1e-15 and j % 2 == 0):
            best, bj = d, j
    return bj


@pytest.mark.parametrize("n", [2, 3, 4, 6, 8])
def test_signed_activation_code_is_eq1_argmin(n):
    rng = np.random.default_rng(n)
    s = np.float32(1.7)
    xs = list(rng.normal(0, 1.2, 300).astype(np.float32))
    half = 1 << (n - 1)
    xs += [np.float32(s * (k + 0.5) / half) for k in range(-half, half)]      # exact ties
    xs += [np.float32(5.0), np.float32(-5.0), np.float32(0.0), np.float32(-0.0)]
    C = oracle.codes_variant(np.array(xs, np.float32)[None, :], np.arange(len(xs), dtype=np.int32),
                             [len(xs), 0], [n, 1], [1, 0], 0, np.full((1, 2, 1), s, np.float32), False)[0]
    for x, c in zip(xs, C):
        assert c == _argmin_eq1(float(x), float(s), n), (x, c)


def test_pm1_code_is_the_sign():
    xs = np.array([-2.0, -1e-30, -0.0, 0.0, 1e-30, 3.0], np.float32)
    assert [oracle.pm1_code(x) for x in xs] == [-1, -1, 1, 1, 1, 1]


def test_pm1_dot_product_is_xnor_popcount():
    """Over m channels, sum u j of +-1 codes = m - 2 * popcount(bits(u) XOR bits(j))
    with bit = (code + 1) / 2, the stored pattern."""
    rng = np.random.default_rng(3)
    M, N, K = 5, 7, 333
    A = rng.normal(size=(M, K)).astype(np.float32)
    W = rng.normal(size=(N, K)).astype(np.float32)
    perm = rng.permutation(K).astype(np.int32)
    count = [K, 0]
    r = oracle.linear_variant(A, W, perm, count, [1, 1], [1, 1], kind=(2, 0))
    bu = oracle.code_patterns(r["U"], count, [1, 1], [2, 0]).astype(np.uint8)
    bj = oracle.code_patterns(r["J"], count, [1, 1], [2, 0]).astype(np.uint8)
    pop = (bu[:, None, :] ^ bj[None, :, :]).astype(np.int64).sum(axis=2)
    assert np.array_equal(r["acc"][0, 0], K - 2 * pop)
    # the bits are the signs of the inputs in packed order
    assert np.array_equal(bu.astype(bool), A[:, perm] >= 0)


def test_one_run_reduces_to_the_default_path():
    d = wl.random_linear(5, M=9, K=400, N=33, bits_lo=3, bits_hi=7, frac_hi=0.3, n_outliers=2)
    a = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"])
    for sub_k in (0, 4096):
        b = oracle.linear_variant(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], kind=(0, 0),
                                  sub_k=sub_k)
        assert np.array_equal(b["s_a"].reshape(2), a["s_a"])
        assert np.array_equal(b["s_w"].reshape(-1, 2), a["s_w"])
        assert np.array_equal(b["U"], a["U"].astype(np.int32))
        assert np.array_equal(b["J"], a["J"].astype(np.int32))
        assert np.array_equal(b["Ap"], a["Ap"])
        assert np.array_equal(b["Wp"], a["Wp"])
        assert np.array_equal(b["acc"][:, 0], a["acc"])
        assert np.array_equal(b["Y64"], a["Y64"])


@pytest.mark.parametrize("sub_k", [128, 256])
def test_run_scales_are_numpy_maxima(sub_k):
    d = wl.random_linear(6, M=6, K=700, N=10, bits_lo=4, bits_hi=8, frac_hi=0.4)
    perm, (c0, c1) = d["perm"], d["count"]
    for X, per_row in ((d["A"], False), (d["A"], True), (d["W"], True)):
        s = oracle.sub_scales(X, perm, d["count"], sub_k, per_row)
        Xp = np.abs(np.asarray(X, np.float32)[:, perm])
        for g, (lo, cnt) in enumerate(((0, c0), (c0, c1))):
            for b in range(s.shape[2]):
                cols = Xp[:, lo + b * sub_k: lo + min(cnt, (b + 1) * sub_k)]
                if cols.shape[1] == 0:
                    assert (s[:, g, b] == 0).all()
                    continue
                ref = cols.max(axis=1) if per_row else np.array([cols.max()])
                assert np.array_equal(s[:, g, b], ref.astype(np.float32))


@pytest.mark.parametrize("kind,bits,sub_k", [((0, 0), (4, 8), 128), ((1, 1), (4, 8), 0), ((1, 1), (3, 6), 128),
                                             ((2, 1), (1, 8), 256), ((2, 2), (1, 1), 0)])
def test_epilogue_is_the_dequantized_matmul(kind, bits, sub_k):
    """Y = (A_hat)(W_hat)^T in fp64, each code decoded with its own run's scale:
    u s_a / La and j s_w / Lw, La = 2^n - 1, 2^(n-1) or 1 by kind."""
    d = wl.random_linear(7, M=7, K=520, N=11, bits_lo=bits[0], bits_hi=bits[1], frac_hi=0.3)
    r = oracle.linear_variant(d["A"], d["W"], d["perm"], d["count"], list(bits), list(bits), kind=kind,
                              sub_k=sub_k)
    K = d["A"].shape[1]
    c0 = d["count"][0]
    def dec(C, s, is_w):
        out = np.zeros(C.shape, np.float64)
        for p in range(K):
            g = 0 if p < c0 else 1
            j = p if g == 0 else p - c0
            b = j // sub_k if sub_k else 0
            n = bits[g]
            if kind[g] == 2:
                L = 1.0
            elif is_w or kind[g] == 1:
                L = float(1 << (n - 1))
            else:
                L = float((1 << n) - 1)
            sc = s[:, g, b] if s.shape[0] == C.shape[0] else s[0, g, b]
            out[:, p] = C[:, p] * sc.astype(np.float64) / L
        return out
    Ah = dec(r["U"], r["s_a"], False)
    Wh = dec(r["J"], r["s_w"], True)
    Y = Ah @ Wh.T
    assert np.allclose(r["Y64"], Y, rtol=1e-12, atol=1e-12 * np.abs(Y).max())


def test_signed_accumulators_are_an_integer_matmul():
    d = wl.random_linear(8, M=12, K=300, N=20, bits_lo=5, bits_hi=8, frac_hi=0.5)
    r = oracle.linear_variant(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], kind=(1, 1))
    c0 = d["count"][0]
    U, J = r["U"].astype(np.int64), r["J"].astype(np.int64)
    assert np.array_equal(r["acc"][0, 0], U[:, :c0] @ J[:, :c0].T)
    assert np.array_equal(r["acc"][1, 0], U[:, c0:] @ J[:, c0:].T)
    assert U.min() >= -(1 << (d["bits"][1] - 1)) and (U < 0).any()
