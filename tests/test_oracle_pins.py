"""Pins for the CPU oracle: each test ties an oracle function to something the
paper or mathematics fixes independently of the oracle's own code -- the
paper's formulas enumerated by brute force, exact rational arithmetic, error
bounds, hand-derived fixtures, library routines (numpy int64 matmul, torch
fp64 conv2d) and invariances the method must have."""
import itertools
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2311_14114_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    out = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                out.append(line)
    return out


# ---------------------------------------------------------------------------
# Eq. (1): level grid and the argmin.
# ---------------------------------------------------------------------------

def eq1_value(bits):
    """q(b) = -b_{n-1} + sum_{i=0}^{n-2} b_i 2^{-(i+1)}, exactly as printed (Eq. 1)."""
    n = len(bits)
    q = Fraction(-bits[n - 1])
    for i in range(n - 1):
        q += Fraction(bits[i], 2 ** (i + 1))
    return q


@pytest.mark.parametrize("n", range(1, 9))
def test_eq1_level_grid_is_twos_complement_fractions(n):
    vals = sorted(eq1_value(b) for b in itertools.product((0, 1), repeat=n))
    expect = [Fraction(j, 2 ** (n - 1)) for j in range(-2 ** (n - 1), 2 ** (n - 1))]
    assert vals == expect


def eq1_argmin(wp: Fraction, n: int) -> int:
    """Brute-force argmin of |w' - q(b)| over all b in {0,1}^n; ties -> even j."""
    best = None
    for b in itertools.product((0, 1), repeat=n):
        q = eq1_value(b)
        j = int(q * 2 ** (n - 1))
        key = (abs(wp - q), j % 2)
        if best is None or key < best[0]:
            best = (key, j)
    return best[1]


@pytest.mark.parametrize("n", range(1, 9))
def test_weight_code_equals_eq1_bruteforce(n):
    rng = np.random.default_rng(100 + n)
    h = 2 ** (n - 1)
    # random w' in [-1, 1] plus every tie point and every level
    wps = list(rng.uniform(-1, 1, 300).astype(np.float32))
    wps += [np.float32((2 * j + 1) / (2 * h)) for j in range(-h, h)]
    wps += [np.float32(j / h) for j in range(-h, h)] + [np.float32(1.0), np.float32(-1.0)]
    for wp in wps:
        got = oracle.weight_code(float(wp), 1.0, n)
        assert got == eq1_argmin(Fraction(float(wp)), n), (n, float(wp))
    # a non-trivial scale: w' is the fp32 quotient (both sides take the code
    # decision in fp32)
    s = np.float32(0.0731)
    for w in rng.uniform(-0.0731, 0.0731, 200).astype(np.float32):
        wp = np.float32(w / s)
        assert oracle.weight_code(float(w), float(s), n) == eq1_argmin(Fraction(float(wp)), n)


@pytest.mark.parametrize("n", range(1, 9))
def test_stored_pattern_is_standard_twos_complement(n):
    """Eq. (1) labels the fraction bits from the top (b_0 weighs 1/2); stored
    as an ordinary n-bit two's-complement integer j the value is the same."""
    for j in range(-2 ** (n - 1), 2 ** (n - 1)):
        p = j & ((1 << n) - 1)
        beta = [(p >> k) & 1 for k in range(n)]
        b = [beta[n - 2 - i] for i in range(n - 1)] + [beta[n - 1]]
        assert eq1_value(b) == Fraction(j, 2 ** (n - 1))


def test_golden_weight_codes():
    for row in _rows("weight_codes.txt"):
        n, w, s, j = row.split()
        assert oracle.weight_code(float(w), float(s), int(n)) == int(j), row


# ---------------------------------------------------------------------------
# Activation quantizer.
# ---------------------------------------------------------------------------

def test_golden_act_codes():
    for row in _rows("act_codes.txt"):
        n, a, s, u = row.split()
        assert oracle.act_code(float(a), float(s), int(n)) == int(u), row


def _round_half_even(x: Fraction) -> int:
    f = x.numerator // x.denominator
    r = x - f
    if r > Fraction(1, 2) or (r == Fraction(1, 2) and f % 2 == 1):
        return f + 1
    return f


@pytest.mark.parametrize("n", range(1, 9))
def test_act_code_matches_exact_rational_rounding(n):
    """Away from ties the fp32 code equals exact rational rounding of a*(2^n-1)/s."""
    rng = np.random.default_rng(200 + n)
    L = 2 ** n - 1
    a = rng.uniform(-0.5, 1.2, 2000).astype(np.float16).astype(np.float32)
    s = np.float32(np.float16(0.97))
    for av in a:
        exact = Fraction(float(av)) * L / Fraction(float(s))
        want = min(max(_round_half_even(exact), 0), L)
        got = oracle.act_code(float(av), float(s), n)
        frac = exact - (exact.numerator // exact.denominator)
        near_tie = abs(frac - Fraction(1, 2)) < Fraction(1, 1 << 18) * max(1, L)
        if near_tie:
            assert abs(got - want) <= 1
        else:
            assert got == want, (n, float(av))


@pytest.mark.parametrize("n", range(1, 9))
def test_round_trip_error_bounds(n):
    """Quantization as bounded noise (Sec. 2.3): |decode(code(x)) - x| <= Delta/2."""
    rng = np.random.default_rng(300 + n)
    s = np.float32(2.5)
    L = 2 ** n - 1
    a = rng.uniform(-s, s, 4000).astype(np.float32)
    for av in a[:1000]:
        u = oracle.act_code(float(av), float(s), n)
        ahat = float(s) * u / L
        if av <= 0:
            assert u == 0
        else:
            assert abs(ahat - float(av)) <= float(s) / (2 * L) * (1 + 1e-6)
    h = 2 ** (n - 1)
    for wv in a[1000:2000]:
        j = oracle.weight_code(float(wv), float(s), n)
        what = float(s) * j / h
        wp = float(wv) / float(s)
        bound = float(s) / (2 * h) if wp <= (h - 1) / h else float(s) / h
        assert abs(what - float(wv)) <= bound * (1 + 1e-6)


# ---------------------------------------------------------------------------
# Scales.
# ---------------------------------------------------------------------------

def test_scales_equal_numpy_max_abs():
    d = wl.random_linear(7, M=37, K=300, N=29, bits_lo=2, bits_hi=8, frac_hi=0.3, n_outliers=3)
    A = d["A"].astype(np.float32)
    perm, count = d["perm"], d["count"]
    g0, g1 = perm[:count[0]], perm[count[0]:]
    s = oracle.act_scales(A, perm, count)
    assert s[0] == np.abs(A[:, g0]).max() and s[1] == np.abs(A[:, g1]).max()
    sr = oracle.act_scales(A, perm, count, per_row=True)
    assert (sr[:, 0] == np.abs(A[:, g0]).max(1)).all() and (sr[:, 1] == np.abs(A[:, g1]).max(1)).all()
    sw = oracle.weight_scales(d["W"], perm, count)
    assert (sw[:, 0] == np.abs(d["W"][:, g0]).max(1)).all()
    assert (sw[:, 1] == np.abs(d["W"][:, g1]).max(1)).all()
    swt = oracle.weight_scales(d["W"], perm, count, per_row=False)
    assert (swt[:, 1] == np.abs(d["W"][:, g1]).max()).all()


@pytest.mark.parametrize("n", range(1, 9))
def test_non_finite_inputs_follow_the_clip(n):
    """Sec. 3 steps 2-3 clip the rounded level to the code range: +inf lands on
    the top code, -inf on the bottom one, whatever the (finite, positive)
    scale; a NaN quotient (a NaN input, or inf / inf under an infinite scale)
    lies on neither side of the clip and is read as code 0."""
    top_a, lo_w, top_w = 2 ** n - 1, -(2 ** (n - 1)), 2 ** (n - 1) - 1
    nan, inf = float("nan"), float("inf")
    for s in (1e-30, 0.37, 1.0, 3e4, 1e30):
        assert oracle.act_code(inf, s, n) == top_a and oracle.act_code(-inf, s, n) == 0
        assert oracle.act_code(nan, s, n) == 0
        assert oracle.weight_code(inf, s, n) == top_w and oracle.weight_code(-inf, s, n) == lo_w
        assert oracle.weight_code(nan, s, n) == 0
    # an infinite scale (a group holding an infinity): finite inputs give 0, inf / inf is NaN
    for x in (0.0, 1.0, -65504.0, 65504.0, inf, -inf, nan):
        assert oracle.act_code(x, inf, n) == 0 and oracle.weight_code(x, inf, n) == 0


def test_scales_drop_nan_and_keep_inf():
    """max |a| as numpy's nanmax: NaN never becomes a scale, an infinity does."""
    d = wl.random_linear(8, M=6, K=96, N=5, bits_lo=2, bits_hi=8, frac_hi=0.25)
    A, W, perm, count = d["A"].astype(np.float32), d["W"].copy(), d["perm"], d["count"]
    g0, g1 = perm[:count[0]], perm[count[0]:]
    A[1, g0[3]] = np.nan
    A[2, g1[0]] = -np.inf
    W[0, g0[1]] = np.nan
    W[3, g1[2]] = np.inf
    sr = oracle.act_scales(A, perm, count, per_row=True)
    assert (sr[:, 0] == np.nanmax(np.abs(A[:, g0]), 1)).all()
    assert (sr[:, 1] == np.nanmax(np.abs(A[:, g1]), 1)).all()
    assert sr[2, 1] == np.inf and np.isfinite(sr[1, 0])
    s = oracle.act_scales(A, perm, count)
    assert s[0] == np.nanmax(np.abs(A[:, g0])) and s[1] == np.inf
    sw = oracle.weight_scales(W, perm, count)
    assert (sw[:, 0] == np.nanmax(np.abs(W[:, g0]), 1)).all() and sw[3, 1] == np.inf


# ---------------------------------------------------------------------------
# Packing.
# ---------------------------------------------------------------------------

def test_golden_pack_blocks():
    for row in _rows("pack_blocks.txt"):
        n, codes, words = [x.strip() for x in row.split("|")]
        n = int(n)
        c = np.zeros(32, dtype=np.uint32)
        for item in codes.split(","):
            i, v = item.split(":")
            c[int(i)] = int(v)
        want = np.array([int(w, 16) for w in words.split()], dtype=np.uint32)
        got = oracle.pack_block(c, n)
        assert (got == want).all(), (row, [hex(x) for x in got])
        assert (oracle.unpack_block(got, n) == c).all()


@pytest.mark.parametrize("n", range(1, 9))
def test_pack_round_trip_and_density(n):
    rng = np.random.default_rng(400 + n)
    for _ in range(50):
        c = rng.integers(0, 2 ** n, 32).astype(np.uint32)
        w = oracle.pack_block(c, n)
        assert w.shape == (n,)          # 32 codes in exactly n words: no waste
        assert (oracle.unpack_block(w, n) == c).all()
    # every bit of the block is used by exactly one code bit
    seen = np.zeros(n, dtype=np.uint32)
    for i in range(32):
        for bit in range(n):
            c = np.zeros(32, dtype=np.uint32)
            c[i] = 1 << bit
            w = oracle.pack_block(c, n)
            assert sum(bin(int(x)).count("1") for x in w) == 1
            assert not (seen & w).any()
            seen |= w
    assert (seen == 0xFFFFFFFF).all()


def test_row_sizes_hand_computed():
    # 4096 channels, 3482 at 3 bits and 614 at 6 bits, 128-code padding:
    # 3584*3/8 + 640*6/8 = 1344 + 480
    assert oracle.row_bytes([3482, 614], [3, 6], 128) == 1824
    # ResNet conv: 179 + 77 channels padded to 32 per pixel -> 192*4/8 + 96*8/8
    assert oracle.row_bytes([179, 77], [4, 8], 32) == 192
    # conv weights, 9 taps: roundup(9*192,128)=1792 codes at 4 bits,
    # roundup(9*96,128)=896 codes at 8 bits
    assert oracle.row_bytes([179, 77], [4, 8], 32, taps=9, is_weight=True) == 896 + 896


def _unpack_rows(packed, count, bits, pad_unit, taps=1, is_weight=False):
    """Independent decode of packed rows back to a code matrix (for invariance tests)."""
    out = []
    for row in packed:
        words = row.view(np.uint32)
        pos, codes = 0, []
        for g in range(2):
            ncodes = (oracle.weight_group_codes(count[g], pad_unit, taps) if is_weight
                      else oracle.act_group_codes(count[g], pad_unit))
            seg = []
            for blk in range(ncodes // 32):
                seg.extend(oracle.unpack_block(words[pos:pos + bits[g]], bits[g]))
                pos += bits[g]
            codes.append(np.array(seg, dtype=np.int64))
        out.append(codes)
    return out


def test_padding_does_not_change_codes():
    """Fig. 2 caption: padding each block to the vector width leaves results unchanged."""
    d = wl.random_linear(11, M=5, K=200, N=3, bits_lo=3, bits_hi=7, frac_hi=0.4)
    r = {pad: oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"],
                            pad_unit=pad) for pad in (32, 128)}
    assert (r[32]["acc"] == r[128]["acc"]).all()
    a32 = _unpack_rows(r[32]["Ap"], d["count"], d["bits"], 32)
    a128 = _unpack_rows(r[128]["Ap"], d["count"], d["bits"], 128)
    for x, y in zip(a32, a128):
        for g in range(2):
            c = d["count"][g]
            assert (x[g][:c] == y[g][:c]).all() and not x[g][c:].any() and not y[g][c:].any()


def test_packed_rows_hold_the_codes():
    d = wl.random_linear(12, M=4, K=300, N=6, bits_lo=1, bits_hi=5, frac_hi=0.2)
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], pad_unit=128)
    c0, c1 = d["count"]
    for m, codes in enumerate(_unpack_rows(r["Ap"], d["count"], d["bits"], 128)):
        assert (codes[0][:c0] == r["U"][m, :c0]).all()
        assert (codes[1][:c1] == r["U"][m, c0:]).all()
    for n, codes in enumerate(_unpack_rows(r["Wp"], d["count"], d["bits"], 128, is_weight=True)):
        for g, (lo, hi) in enumerate(((0, c0), (c0, c0 + c1))):
            j = codes[g][:hi - lo]
            j = np.where(j >= 2 ** (d["bits"][g] - 1), j - 2 ** d["bits"][g], j)
            assert (j == r["J"][n, lo:hi]).all()


# ---------------------------------------------------------------------------
# Accumulators and epilogue.
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("bits", [(8, 8), (2, 8), (1, 4), (3, 6), (4, 4)])
def test_accumulators_equal_int64_matmul(bits):
    """All-8-bit channels are a plain u8 x s8 GEMM (Sec. 4.2); any widths reduce
    to an int64 matmul of the code matrices per group."""
    d = wl.random_linear(20 + bits[0], M=23, K=333, N=19, bits_lo=bits[0], bits_hi=bits[1],
                         frac_hi=0.35, n_outliers=2)
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"])
    U, J = r["U"].astype(np.int64), r["J"].astype(np.int64)
    c0 = d["count"][0]
    assert (r["acc"][0] == U[:, :c0] @ J[:, :c0].T).all()
    assert (r["acc"][1] == U[:, c0:] @ J[:, c0:].T).all()
    assert np.abs(r["acc"]).max() < 2 ** 31


@pytest.mark.parametrize("act_mode", ["tensor", "row"])
def test_epilogue_equals_dequantized_matmul(act_mode):
    """Factoring identity: sum_g alpha_g Acc_g equals the fp64 product of the
    decoded activations s*b/(2^n-1) and weights s*q(b) (Sec. 3 decode rules)."""
    d = wl.random_linear(31, M=17, K=260, N=13, bits_lo=2, bits_hi=8, frac_hi=0.25, n_outliers=3)
    r = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], act_mode=act_mode)
    c0 = d["count"][0]
    grp = np.r_[np.zeros(c0, int), np.ones(d["count"][1], int)]
    La = np.array([2.0 ** b - 1 for b in d["bits"]])[grp]
    Lw = np.array([2.0 ** (b - 1) for b in d["bits"]])[grp]
    sa = r["s_a"][:, grp] if act_mode == "row" else r["s_a"][grp][None, :]
    Ahat = sa.astype(np.float64) * r["U"] / La
    What = r["s_w"][:, grp].astype(np.float64) * r["J"] / Lw
    Yref = Ahat @ What.T
    assert np.allclose(r["Y64"], Yref, rtol=1e-12, atol=1e-12 * np.abs(Yref).max())


def test_conv_equals_torch_conv2d_of_decoded_tensors():
    """im2col accumulation vs torch's fp64 conv2d of the decoded tensors in the
    original channel order (checks tap order, padding and the permutation)."""
    torch = pytest.importorskip("torch")
    spec = wl.ConvSpec("t", batch=2, H=5, W=6, C=40, C_out=7, R=3, S=3, stride=(1, 1), pad=(1, 1),
                       bits_lo=3, bits_hi=8, frac_hi=0.3, seed=5)
    for stride, pad in (((1, 1), (1, 1)), ((2, 1), (0, 1))):
        d = wl.make_conv(spec)
        r = oracle.conv2d(d["X"], d["W"], d["perm"], d["count"], d["bits"], d["bits"], 3, 3,
                          stride=stride, pad=pad)
        perm, c0 = d["perm"], d["count"][0]
        inv = np.argsort(perm)
        grp = (inv >= c0).astype(int)     # group of each original channel
        La = np.array([2.0 ** b - 1 for b in d["bits"]])[grp]
        Lw = np.array([2.0 ** (b - 1) for b in d["bits"]])[grp]
        Xhat = r["s_a"][grp].astype(np.float64) * r["U"][:, inv] / La             # [pix][C] original order
        Xhat = Xhat.reshape(spec.batch, spec.H, spec.W, spec.C).transpose(0, 3, 1, 2)
        What = r["s_w"][:, grp][:, None, :].astype(np.float64) * r["J"][:, :, inv] / Lw   # [Cout][RS][C]
        What = What.reshape(spec.C_out, 3, 3, spec.C).transpose(0, 3, 1, 2)
        Yt = torch.nn.functional.conv2d(torch.from_numpy(np.ascontiguousarray(Xhat)),
                                        torch.from_numpy(np.ascontiguousarray(What)),
                                        stride=stride, padding=pad)
        Yt = Yt.permute(0, 2, 3, 1).reshape(-1, spec.C_out).numpy()
        assert np.allclose(r["Y64"], Yt, rtol=1e-11, atol=1e-11 * np.abs(Yt).max())


def test_permutation_invariance():
    """Relabelling the original channels (and the permutation with them) leaves
    the output unchanged: only the packed order matters."""
    d = wl.random_linear(41, M=9, K=150, N=8, bits_lo=2, bits_hi=6, frac_hi=0.3, n_outliers=2)
    r1 = oracle.linear(d["A"], d["W"], d["perm"], d["count"], d["bits"], d["bits"])
    rng = np.random.default_rng(0)
    pi = rng.permutation(150)                    # new channel c' = pi[c]
    A2 = np.empty_like(d["A"]); A2[:, pi] = d["A"]
    W2 = np.empty_like(d["W"]); W2[:, pi] = d["W"]
    perm2 = pi[d["perm"]].astype(np.int32)
    r2 = oracle.linear(A2, W2, perm2, d["count"], d["bits"], d["bits"])
    assert (r1["acc"] == r2["acc"]).all() and (r1["Y64"] == r2["Y64"]).all()


def test_zero_group_gives_zero_scale_codes_and_contribution():
    d = wl.random_linear(51, M=6, K=96, N=5, bits_lo=2, bits_hi=8, frac_hi=0.25)
    A = d["A"].copy()
    A[:, d["perm"][d["count"][0]:]] = 0      # high group all zeros
    r = oracle.linear(A, d["W"], d["perm"], d["count"], d["bits"], d["bits"])
    assert r["s_a"][1] == 0 and not r["U"][:, d["count"][0]:].any()
    assert not r["acc"][1].any() and np.isfinite(r["Y64"]).all()


def test_closed_form_constant_inputs():
    """A = s everywhere gives u = 2^n - 1; constant weight rows w = c give
    j = round(c/max|w| * 2^(n-1)) clamped; Acc_g = count_g * u * j."""
    K, M, N = 160, 3, 4
    perm = np.arange(K, dtype=np.int32)
    count = [120, 40]
    bits = [3, 8]
    A = np.full((M, K), 1.5, dtype=np.float16)
    W = np.zeros((N, K), dtype=np.float32)
    W[:, :120] = np.array([0.5, -0.5, 0.25, -1.0])[:, None]
    W[:, 120:] = np.array([0.2, 0.3, -0.7, 0.01])[:, None]
    r = oracle.linear(A, W, perm, count, bits, bits)
    assert (r["U"][:, :120] == 7).all() and (r["U"][:, 120:] == 255).all()
    # each row is constant within a group, so w' = +-1 -> j = 3 or -4 (3-bit), 127 or -128 (8-bit)
    j0 = np.array([3, -4, 3, -4])
    j1 = np.array([127, 127, -128, 127])
    assert (r["acc"][0] == 120 * 7 * j0[None, :]).all()
    assert (r["acc"][1] == 40 * 255 * j1[None, :]).all()


def _fp32(x):
    return float(np.float32(x))


def test_tiny_end_to_end_bruteforce():
    """Every bit pair on tiny shapes, recomputed from the definitions with exact
    rationals (fp32 quotient for the code decision), against the oracle."""
    rng = np.random.default_rng(61)
    for lo, hi in itertools.product(range(1, 9), repeat=2):
        M, N, K = 2, 3, 6
        perm = rng.permutation(K).astype(np.int32)
        count = [4, 2]
        A = rng.standard_normal((M, K)).astype(np.float16)
        W = (rng.standard_normal((N, K)) * 0.1).astype(np.float32)
        r = oracle.linear(A, W, perm, count, [lo, hi], [lo, hi])
        bits = [lo, hi]
        groups = [perm[:4], perm[4:]]
        Y = np.zeros((M, N))
        for g in range(2):
            n = bits[g]
            sa = max(abs(float(A[m, c])) for m in range(M) for c in groups[g])
            for m in range(M):
                for o in range(N):
                    sw = max(abs(float(W[o, c])) for c in groups[g])
                    acc = 0
                    for c in groups[g]:
                        q = _fp32(np.float32(float(A[m, c])) / np.float32(sa))
                        u = min(max(_round_half_even(Fraction(_fp32(np.float32(q) * np.float32(2 ** n - 1)))), 0), 2 ** n - 1)
                        wp = Fraction(_fp32(np.float32(W[o, c]) / np.float32(sw)))
                        j = eq1_argmin(wp, n)
                        acc += u * j
                    assert acc == r["acc"][g, m, o]
                    Y[m, o] += sa * sw * acc / ((2 ** n - 1) * 2 ** (n - 1))
        assert np.allclose(r["Y64"], Y, rtol=1e-13, atol=1e-15)
