"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test ties one oracle function to something other than itself: a value
the paper prints (fixtures under tests/golden/, each with its citation), a
second formulation the paper states is equivalent, a textbook result, an
invariant, or brute force on tiny inputs.  CPU only.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle as o
from conftest import oracle_step_function, read_golden, step_function_codes

ALL_FORMATS = [(b, k) for b in range(2, 9) for k in range(0, b)]
SMALL_FORMATS = [(b, k) for b in range(2, 7) for k in range(0, b)]


# --------------------------------------------------------------- Table 1 ---

@pytest.mark.parametrize("row", read_golden("table1_alpha_dda.txt"))
def test_table1_alpha_star_and_dda(row):
    b, k = int(row[0]), int(row[1])
    dda, astar = float(row[2]), float(row[3])
    a, d_half = o.alpha_star(b, k)
    assert abs(a - astar) <= 5e-5 + 1e-12, (b, k, a)
    # Table 1's DDA is the squared error over both halves of N(0,1).
    assert abs(2.0 * d_half - dda) <= 5e-5 + 1e-12, (b, k, 2 * d_half)


def test_lloyd_max_three_level_gaussian():
    g = {r[0]: float(r[1]) for r in read_golden("lloyd_max_gaussian_3level.txt")}
    a, d_half = o.alpha_star(2, 0)
    assert abs(a - g["output"]) < 5e-4
    assert abs(a / 2 - g["threshold"]) < 5e-4       # midpoint of {0, alpha}
    assert abs(2 * d_half - g["mse"]) < 5e-4
    # The optimum satisfies the centroid condition: the output level is the
    # mean of N(0,1) on [threshold, inf) -> phi(t) / Q(t).
    t = a / 2
    phi = math.exp(-t * t / 2) / math.sqrt(2 * math.pi)
    Q = 0.5 * math.erfc(t / math.sqrt(2))
    assert abs(a - phi / Q) < 1e-6


@pytest.mark.parametrize("b", [3, 4, 5, 6])
def test_alpha_star_scale_identity(b):
    # ESB(b, b-1) is ESB(b, b-2) scaled by 1/2, so its optimal alpha doubles.
    s1 = o.set_nonneg(b, b - 1)
    s2 = o.set_nonneg(b, b - 2)
    assert np.array_equal(s1 * 2, s2)
    a1, d1 = o.alpha_star(b, b - 1)
    a2, d2 = o.alpha_star(b, b - 2)
    assert abs(a1 - 2 * a2) <= 1e-7 * a1
    assert abs(d1 - d2) <= 1e-9


def test_D_against_monte_carlo():
    # D(alpha) is the half-line squared error of nearest-element projection;
    # compare the closed form with a large sample of |N(0,1)|.
    rng = np.random.default_rng(7)
    t = np.abs(rng.standard_normal(2_000_000))
    for (b, k, alpha) in [(4, 2, 1.4), (4, 1, 0.5), (5, 2, 0.3), (3, 0, 0.8)]:
        s = o.set_nonneg(b, k) * alpha
        mids = 0.5 * (s[1:] + s[:-1])
        idx = np.searchsorted(mids, t, side="right")
        mse_half = np.mean((t - s[idx]) ** 2) * 0.5   # density of the half is phi, mass 1/2
        assert abs(mse_half - o.D(alpha, b, k)) < 3e-3 * max(o.D(alpha, b, k), 1e-3) + 2e-5


# ------------------------------------------------------------- value set ---

@pytest.mark.parametrize("b,k", ALL_FORMATS)
def test_set_size_extremes_symmetry(b, k):
    s = o.set_full(b, k)
    assert len(s) == 2 ** b - 1
    assert len(np.unique(s)) == len(s)
    assert np.array_equal(np.sort(s), s)
    assert np.array_equal(s, -s[::-1])
    assert 0.0 in s
    N = 2 ** (b - k - 1) - 1
    C = (2 ** (k + 1) - 1) * 2.0 ** (N - 1 - k) if N >= 1 else (2 ** k - 1) / 2.0 ** k
    assert s[-1] == C == o.C_of(b, k)


def test_intro_two_significant_bit_set():
    g = {r[0]: [int(v) for v in r[1:]] for r in read_golden("two_significant_bit_set_b5.txt")}
    pos = set(g["base"])
    for e in g["shifts"]:
        pos |= {v << e for v in g["shift_base"]}
    full = sorted(pos | {-v for v in pos})
    assert len(full) == g["count"][0] == 2 ** g["bits"][0] - 1
    assert sorted(full)[-len(g["printed_tail"]):] == g["printed_tail"]
    # Two significant bits in five bits is ESB(5, 1); its integer images.
    b, k = g["bits"][0], g["significant"][0] - 1
    imgs = (o.set_full(b, k) * 2 ** k).astype(np.int64).tolist()
    assert imgs == full


@pytest.mark.parametrize("b", range(2, 9))
def test_linear_special_case(b):
    # k = b - 2 is linear quantization Q_l: {0, +-1, ..., +-(2^(b-1)-1)} * alpha'.
    if b < 2:
        return
    k = b - 2
    imgs = o.set_full(b, k) * 2 ** k
    assert np.array_equal(imgs, np.arange(-(2 ** (b - 1) - 1), 2 ** (b - 1)))


@pytest.mark.parametrize("b", range(2, 8))
def test_pot_special_case(b):
    # k = 0 is the power-of-two set with 2^b - 1 elements.
    n = 2 ** (b - 1) - 1
    pos = [0.0] + [2.0 ** j for j in range(n)]
    exp = sorted(set(pos) | {-v for v in pos})
    assert o.set_full(b, 0).tolist() == exp


def test_ternary_special_case():
    assert o.set_full(2, 0).tolist() == [-1.0, 0.0, 1.0]


def test_fig10_one_sign_two_exponent_one_fraction():
    # Fig. 10: ESB with 1 sign, 2 exponent and 1 fraction bit = ESB(4, 1).
    # Decoding every code with the format equation gives the set.
    vals = sorted({abs(o.decode(c, 4, 1)) for c in range(16)})
    assert vals == [0, 0.5, 1, 1.5, 2, 3, 4, 6]
    assert np.array_equal(o.set_nonneg(4, 1), np.array(vals))


@pytest.mark.parametrize("b,k", ALL_FORMATS)
def test_format_decode_equals_set(b, k):
    # Sec. IV-A format equation versus Sec. III-B set construction.
    vals = [o.decode(c, b, k) for c in range(2 ** b)]
    s = o.set_full(b, k)
    assert sorted(set(vals)) == s.tolist()
    # every non-zero element has exactly one code; zero has two bit patterns
    # (sign 0 and sign 1), and encode always returns the sign-0 one.
    assert len(vals) == len(s) + 1
    z = o.zero_code(b, k)
    assert o.decode(z, b, k) == 0.0 and (z >> (b - 1)) == 0
    for c in range(2 ** b):
        q = o.decode(c, b, k)
        assert o.encode(q, b, k) == (z if q == 0 else c)


@pytest.mark.parametrize("b,k", [(b, k) for b in range(2, 7) for k in range(0, b)])
def test_multiplication_identity(b, k):
    # Eq. esb_multiplication: q_i q_j = (-1)^(s_i ^ s_j) (f << e), with
    # f = (z_i + 0.f_i)(z_j + 0.f_j), e = e_i z_i + e_j z_j, z = [e != 2^(b-k-1)-1].
    N = 2 ** (b - k - 1) - 1
    ew = b - k - 1

    def fields(c):
        s = (c >> (b - 1)) & 1
        e = (c >> k) & ((1 << ew) - 1) if ew > 0 else 0
        f = c & ((1 << k) - 1)
        return s, e, f

    codes = list(range(2 ** b))
    for ci in codes:
        si, ei, fi = fields(ci)
        zi = 1 if ei != N else 0
        for cj in codes:
            sj, ej, fj = fields(cj)
            zj = 1 if ej != N else 0
            f = (Fraction(zi) + Fraction(fi, 2 ** k)) * (Fraction(zj) + Fraction(fj, 2 ** k))
            e = ei * zi + ej * zj
            rhs = (-1) ** (si ^ sj) * f * 2 ** e
            lhs = Fraction(o.decode(ci, b, k)) * Fraction(o.decode(cj, b, k))
            assert lhs == rhs


# ------------------------------------------------------------ projection ---

def test_worked_projection_example():
    g = {r[0]: float(r[1]) for r in read_golden("projection_example_b5k2.txt")}
    b, k = int(g["b"]), int(g["k"])
    alpha = np.float32(g["x"] / g["scaled"])
    q = o.project_value(g["x"], float(alpha), b, k)
    assert q == g["projected"]
    assert abs(float(alpha) * q - g["rescaled"]) < 0.01


def _midpoint_probe_values(b, k):
    s = o.set_nonneg(b, k)
    mids = 0.5 * (s[1:] + s[:-1])
    pts = np.concatenate([s, mids, [o.C_of(b, k) * 1.5, 1e30]]).astype(np.float32)
    out = [pts]
    for step in (1, 2, 3):
        out.append(np.nextafter(pts, np.float32(np.inf)))
        out.append(np.nextafter(pts, np.float32(-np.inf)))
        pts = out[-1]
    v = np.concatenate(out)
    return np.concatenate([v, -v, [0.0, -0.0, np.inf, -np.inf, np.nan]]).astype(np.float32)


@pytest.mark.parametrize("b,k", SMALL_FORMATS)
@pytest.mark.parametrize("signed", [True, False])
@pytest.mark.parametrize("rounding", [0, 1])
def test_lookup_equals_shift_and_round(b, k, signed, rounding):
    # Eq. thresholing_func and Eq. fast_projection give the same projection.
    C = o.C_of(b, k)
    x = [_midpoint_probe_values(b, k)]
    # a strided sweep over every fp32 bit pattern in [0, 1.25 C]
    hi = np.float32(1.25 * C).view(np.uint32)
    x.append(np.arange(0, int(hi), 4099, dtype=np.uint32).view(np.float32))
    x.append(np.random.default_rng(b * 10 + k).standard_normal(20000).astype(np.float32) * C)
    x = np.concatenate(x)
    x = np.concatenate([x, -x])
    for alpha in (1.0, 0.7310585, 3.0):
        a = o.project_values(x, alpha, b, k, signed, rounding)
        s = o.project_values_shift(x, alpha, b, k, signed, rounding)
        assert np.array_equal(a, s), (alpha, x[a != s][:5])


@pytest.mark.parametrize("b,k", [(b, k) for b in range(2, 6) for k in range(0, b)])
def test_projection_brute_force_nearest(b, k):
    rng = np.random.default_rng(100 + 10 * b + k)
    s = o.set_full(b, k)
    x = np.concatenate([rng.standard_normal(3000) * o.C_of(b, k),
                        (0.5 * (s[1:] + s[:-1]))]).astype(np.float32)
    alpha = np.float32(0.8125)        # exact dyadic: v = x / alpha is exact enough to hit ties
    x = np.concatenate([x, (x * alpha).astype(np.float32)])
    got = o.project_values(x, float(alpha), b, k)
    v = x / alpha                      # numpy float32 division is IEEE single
    for xi, vi, gi in zip(x, v.astype(np.float64), got):
        d = np.abs(s - vi)
        best = d.min()
        cands = s[d == best]
        exp = cands[np.argmax(np.abs(cands))]   # tie -> larger magnitude
        assert gi == exp, (xi, vi, gi, exp)


@pytest.mark.parametrize("b,k", SMALL_FORMATS)
def test_projection_invariants(b, k):
    s = o.set_full(b, k)
    C = o.C_of(b, k)
    for alpha in (1.0, 0.37, 1.9):
        # idempotence: every set element (scaled by alpha) projects onto itself
        xs = (s * alpha).astype(np.float32)
        assert np.array_equal(o.project_values(xs, alpha, b, k), s)
    rng = np.random.default_rng(b * 7 + k)
    x = np.sort(rng.standard_normal(5000).astype(np.float32) * np.float32(C))
    q = o.project_values(x, 0.9, b, k)
    assert np.all(np.diff(q) >= 0)                                  # monotone
    assert np.array_equal(o.project_values(-x, 0.9, b, k), -q)      # symmetric
    assert set(np.unique(q)).issubset(set(s))
    qu = o.project_values(x, 0.9, b, k, signed=False)
    assert np.all(qu >= 0) and np.array_equal(qu[x > 0], q[x > 0])
    sp = np.array([np.inf, -np.inf, np.nan, 1e38, -1e38, 0.0, -0.0], dtype=np.float32)
    assert o.project_values(sp, 1.0, b, k).tolist() == [C, -C, 0.0, C, -C, 0.0, 0.0]


def test_tie_rules_differ_only_on_ties():
    b, k = 4, 2
    s = o.set_nonneg(b, k)
    mids = (0.5 * (s[1:] + s[:-1])).astype(np.float32)
    away = o.project_values(mids, 1.0, b, k, rounding=0)
    even = o.project_values(mids, 1.0, b, k, rounding=1)
    assert np.array_equal(away, s[1:])
    imgs = (even * 4).astype(int)
    assert np.all(imgs % 2 == 0)
    x = np.nextafter(mids, np.float32(0))
    assert np.array_equal(o.project_values(x, 1.0, b, k, rounding=0),
                          o.project_values(x, 1.0, b, k, rounding=1))


def test_pack_layout():
    # Packing: floor(32/b) codes per word, code j in bits [b*j, b*j+b);
    # unused slots hold the zero code; unused high bits are zero.
    b, k = 4, 2
    z = o.zero_code(b, k)
    assert z == 0b0100
    w = o.pack(np.array([[1, 2, 3]], dtype=np.uint32), b, k)
    assert w.tolist() == [[0x44444321]]
    b, k = 3, 1
    z = o.zero_code(b, k)                 # sign 0, e = N = 1, f = 0
    assert z == 0b010
    w = o.pack(np.array([[7, 1]], dtype=np.uint32), b, k)
    assert w[0, 0] == (7 | 1 << 3 | sum(z << (3 * j) for j in range(2, 10)))
    rng = np.random.default_rng(3)
    for b in range(2, 9):
        codes = rng.integers(0, 2 ** b, size=(5, 37), dtype=np.uint32)
        assert np.array_equal(o.unpack(o.pack(codes, b, 0, ld_words=12), 37, b), codes)


# ----------------------------------------------------------- calibration ---

def test_calibration_closed_forms():
    astar = o.alpha_star(4, 2)[0]
    a, st = o.calibrate(np.array([1, 2, 3, 4], np.float32), 4, 2)
    assert st[0] == 2.5 and abs(st[1] - math.sqrt(1.25)) < 1e-15 and st[2] == 4
    assert a == np.float32(astar * (math.sqrt(1.25) + 1e-7))
    a, st = o.calibrate(np.full(1000, 3.25, np.float32), 4, 2)
    assert st[1] == 0.0 and a == np.float32(astar * 1e-7)
    x = np.array([-2.5, 2.5] * 50, np.float32)
    a, st = o.calibrate(x, 4, 2)
    assert st[0] == 0.0 and st[1] == 2.5
    a, st = o.calibrate(np.array([3.0, 4.0], np.float32), 4, 2, signed=False)
    assert abs(st[1] - math.sqrt(12.5)) < 1e-15
    # large offset: two-pass moments are unaffected by the mean
    rng = np.random.default_rng(0)
    y = rng.standard_normal(10000).astype(np.float32)
    _, s0 = o.calibrate(y, 4, 2)
    _, s1 = o.calibrate((y.astype(np.float64) + 1024.0).astype(np.float32), 4, 2)
    assert abs(s1[1] - s0[1]) < 1e-4


# ----------------------------------------------------------- contraction ---

def _image_table(b, k):
    return np.array([o.image(c, b, k) for c in range(2 ** b)], dtype=np.int64)


@pytest.mark.parametrize("fa,fb", [((4, 2), (4, 2)), ((3, 1), (6, 3)), ((5, 2), (5, 1))])
def test_gemm_brute_force(fa, fb):
    rng = np.random.default_rng(11)
    M, N, K = 7, 5, 29
    ca = rng.integers(0, 2 ** fa[0], size=(M, K), dtype=np.uint32)
    cb = rng.integers(0, 2 ** fb[0], size=(N, K), dtype=np.uint32)
    A = o.pack(ca, fa[0], fa[1], ld_words=o.words_for(K, fa[0]) + 1)
    B = o.pack(cb, fb[0], fb[1])
    got = o.gemm_i64(A, fa, B, fb, M, N, K)
    exp = _image_table(*fa)[ca] @ _image_table(*fb)[cb].T
    assert np.array_equal(got, exp)
    assert o.gemm_entry(A, fa, B, fb, K, 3, 4) == exp[3, 4]


@pytest.mark.parametrize("fa,fb", [((6, 1), (6, 1)), ((5, 0), (4, 2)), ((6, 0), (3, 1))])
def test_gemm_large_images_brute_force(fa, fb):
    # power-of-two-like sets with images up to 2^30: Python integers as truth
    rng = np.random.default_rng(7)
    M, N, K = 5, 4, 9
    ca = rng.integers(0, 2 ** fa[0], size=(M, K), dtype=np.uint32)
    cb = rng.integers(0, 2 ** fb[0], size=(N, K), dtype=np.uint32)
    A = o.pack(ca, *fa, ld_words=4)
    B = o.pack(cb, *fb, ld_words=4)
    got = o.gemm_i64(A, fa, B, fb, M, N, K)
    ta = [o.image(c, *fa) for c in range(2 ** fa[0])]
    tb = [o.image(c, *fb) for c in range(2 ** fb[0])]
    for m in range(M):
        for n in range(N):
            assert int(got[m, n]) == sum(ta[int(ca[m, j])] * tb[int(cb[n, j])] for j in range(K))


def test_conv_and_depthwise_brute_force():
    rng = np.random.default_rng(5)
    fx, fw = (4, 2), (4, 1)
    Nb, H, Wd, C, Cout, R, S = 2, 6, 5, 11, 3, 3, 3
    for stride, pad in [(1, 1), (2, 1), (1, 0), (2, 0)]:
        cx = rng.integers(0, 16, size=(Nb, H, Wd, C), dtype=np.uint32)
        cw = rng.integers(0, 16, size=(Cout, R, S, C), dtype=np.uint32)
        X = o.pack(cx.reshape(-1, C), *fx, ld_words=4).reshape(Nb, H, Wd, 4)
        W = o.pack(cw.reshape(-1, C), *fw, ld_words=4).reshape(Cout, R, S, 4)
        got = o.conv2d_i64(X, fx, W, fw, Nb, H, Wd, C, Cout, R, S, stride, pad)
        ix = np.pad(_image_table(*fx)[cx], ((0, 0), (pad, pad), (pad, pad), (0, 0)))
        iw = _image_table(*fw)[cw]
        P, Q = got.shape[1], got.shape[2]
        exp = np.zeros_like(got)
        for r in range(R):
            for s_ in range(S):
                patch = ix[:, r:r + stride * P:stride, s_:s_ + stride * Q:stride, :]
                exp += np.einsum("npqc,oc->npqo", patch, iw[:, r, s_, :])
        assert np.array_equal(got, exp)
        # the row-restricted form (the CPU baseline's bounded samples): every
        # window of output rows, first and last rows included
        for p0 in range(P):
            for p1 in range(p0 + 1, P + 1):
                part = o.conv2d_rows_i64(X, fx, W, fw, Nb, H, Wd, C, Cout, R, S, stride, pad, p0, p1)
                assert np.array_equal(part, exp[:, p0:p1]), (stride, pad, p0, p1)
        # depthwise with one filter per channel
        cwd = rng.integers(0, 16, size=(R, S, C), dtype=np.uint32)
        Wd_ = o.pack(cwd.reshape(-1, C), *fw, ld_words=4).reshape(R, S, 4)
        gotd = o.dwconv_i64(X, fx, Wd_, fw, Nb, H, Wd, C, R, S, stride, pad)
        iwd = _image_table(*fw)[cwd]
        expd = np.zeros_like(gotd)
        for r in range(R):
            for s_ in range(S):
                expd += ix[:, r:r + stride * P:stride, s_:s_ + stride * Q:stride, :] * iwd[r, s_]
        assert np.array_equal(gotd, expd)


def test_pooling_brute_force():
    rng = np.random.default_rng(9)
    b, k = 4, 2
    Nb, H, Wd, C = 2, 7, 6, 9
    cx = rng.integers(0, 16, size=(Nb, H, Wd, C), dtype=np.uint32)
    X = o.pack(cx.reshape(-1, C), b, k, ld_words=4).reshape(Nb, H, Wd, 4)
    vals = np.vectorize(lambda c: o.decode(int(c), b, k))(cx)
    Y = o.maxpool_codes(X, b, k, Nb, H, Wd, C, 3, 2, 1)
    P, Q = Y.shape[1], Y.shape[2]
    assert (P, Q) == (math.ceil(H / 2), math.ceil(Wd / 2))   # Sec. IV-B: ceil(h/s)
    yv = np.vectorize(lambda c: o.decode(int(c), b, k))(o.unpack(Y.reshape(-1, 4), C, b)).reshape(Nb, P, Q, C)
    padded = np.pad(vals, ((0, 0), (1, 1), (1, 1), (0, 0)), constant_values=-np.inf)
    for p in range(P):
        for q in range(Q):
            win = padded[:, 2 * p:2 * p + 3, 2 * q:2 * q + 3, :]
            assert np.array_equal(yv[:, p, q, :], win.max(axis=(1, 2)))
    sums = o.avgpool_sum_i64(X, b, k, Nb, H * Wd, C)
    assert np.array_equal(sums, _image_table(b, k)[cx].sum(axis=(1, 2)))


# --------------------------------------------------------------- epilogue ---

def _fma32_exact(s, a, c):
    """Correctly rounded float32 of s*a + c (exact rational, then RN-even)."""
    exact = Fraction(float(s)) * Fraction(float(a)) + Fraction(float(c))
    f = np.float32(float(exact))
    lo, hi = np.nextafter(f, np.float32(-np.inf)), np.nextafter(f, np.float32(np.inf))
    best = min((lo, f, hi), key=lambda t: (abs(Fraction(float(t)) - exact),
                                           int(np.float32(t).view(np.uint32)) & 1))
    return np.float32(best)


def test_epilogue_op_order():
    rng = np.random.default_rng(2)
    fo = (4, 2, False)
    acc = rng.integers(-3000, 3000, size=(6, 8)).astype(np.int64)
    scale = rng.uniform(1e-4, 1e-2, 8).astype(np.float32)
    bias = rng.uniform(-0.5, 0.5, 8).astype(np.float32)
    res = rng.integers(-7, 8, size=(6, 8)).astype(np.int64)
    y, codes = o.epilogue(acc, scale, bias, 1, 0.41, fo, res_images=res, res_scale=0.0625)
    for m in range(6):
        for n in range(8):
            t = _fma32_exact(scale[n], np.float32(acc[m, n]), bias[n])
            t = _fma32_exact(np.float32(0.0625), np.float32(res[m, n]), t)
            t = max(t, np.float32(0.0))
            assert y[m, n] == t
            assert codes[m, n] == o.encode(o.project_value(float(t), 0.41, *fo), 4, 2, False)
    y6, _ = o.epilogue(acc * 100, scale, bias, 2, 0.41, fo)
    assert y6.max() <= 6.0 and y6.min() >= 0.0


@pytest.mark.parametrize("b,k", [(4, 2), (5, 1), (6, 3), (3, 0), (2, 0)])
def test_dD_is_the_derivative_of_D(b, k):
    # D'(alpha) (used to locate alpha*) against central differences of D.
    for a in (0.05, 0.3, 1.0, 1.7):
        h = a * 1e-5
        fd = (o.D(a + h, b, k) - o.D(a - h, b, k)) / (2 * h)
        assert abs(fd - o.dD(a, b, k)) < 1e-6 * max(1.0, abs(fd)), (a, fd, o.dD(a, b, k))
    a_star, _ = o.alpha_star(b, k)
    assert abs(o.dD(a_star, b, k)) < 1e-12
    assert o.dD(a_star * 0.99, b, k) < 0 < o.dD(a_star * 1.01, b, k)


STEP_CASES = [(2, 0, True, 0, 1.0), (3, 1, True, 0, 3.0), (4, 2, True, 0, 0.7310585), (4, 2, False, 1, 1.0),
              (5, 2, False, 0, 0.7310585), (6, 3, True, 1, 0.7310585), (8, 4, True, 0, 0.37), (8, 7, True, 0, 1.0)]


@pytest.mark.parametrize("b,k,signed,rounding,alpha", STEP_CASES)
def test_projection_is_the_step_function_of_its_breakpoints(b, k, signed, rounding, alpha):
    # The oracle's projection of any fp32 is fixed by the L-1 breakpoints
    # found from it by bisection (monotone in |x|, symmetric or clamped for
    # x < 0, NaN alone): checked on random bit patterns, every breakpoint and
    # its neighbours, and the special values.  The GPU test that projects
    # every one of the 2^32 patterns compares against this step function.
    import torch
    step = oracle_step_function(alpha, b, k, signed, rounding)
    T = step[0]
    rng = np.random.default_rng(b * 100 + k)
    bits = np.concatenate([rng.integers(0, 1 << 32, 1 << 17, dtype=np.int64),
                           T, T - 1, T + 1, T | (1 << 31), (T - 1) | (1 << 31),
                           [0, 1 << 31, 0x7F800000, 0xFF800000, 0x7F800001, 0x7FC00000, 0xFFC00000, 1, 0x80000001,
                            0x7F7FFFFF, 0xFF7FFFFF]]).astype(np.int64)
    x = bits.astype(np.uint32).view(np.float32)
    exp = o.project_codes(x, alpha, b, k, signed, rounding).astype(np.int64)
    got = step_function_codes(torch.from_numpy(bits), step).numpy()
    bad = np.nonzero(got != exp)[0]
    assert bad.size == 0, [(hex(int(bits[i])), int(exp[i]), int(got[i])) for i in bad[:5]]


@pytest.mark.parametrize("b,k", ALL_FORMATS)
def test_code_rank_is_the_rotated_exponent_field(b, k):
    # Sec. IV-A's code (e, f) with e = N for the values below one: ordering
    # the non-negative codes by value is ordering them by (code + 2^k) mod
    # 2^(b-1), so comparisons of codes (max pooling) need no decode.
    L = 1 << (b - 1)
    order = sorted(range(L), key=lambda c: o.decode(c, b, k))
    assert [(c + (1 << k)) % L for c in order] == list(range(L))


# ------------------------------------------- DDA for other data densities ---

def test_laplace_ternary_closed_form():
    # ternary set {0, +-alpha}: alpha* satisfies the centroid condition
    # alpha = E[t | t > alpha / 2]; the Laplace tail is memoryless, so
    # E[t | t > c] = c + 1/lam and alpha* = 2 / lam = sqrt 2 (unit variance);
    # the squared error is then 1 - alpha*^2 P(|t| > alpha*/2) = 1 - 2/e
    a, dda = o.alpha_star_laplace(2, 0)
    assert abs(a - math.sqrt(2.0)) <= 1e-7
    assert abs(dda - (1.0 - 2.0 / math.e)) <= 1e-9


@pytest.mark.parametrize("b,k", [(3, 1), (4, 2), (4, 1)])
def test_laplace_D_against_monte_carlo(b, k):
    rng = np.random.default_rng(b * 10 + k)
    t = np.abs(rng.laplace(0.0, 1.0 / math.sqrt(2.0), 2_000_000))    # unit variance
    s = o.set_nonneg(b, k)
    for alpha in (0.3, 1.0, 2.0):
        v = t / alpha
        idx = np.clip(np.searchsorted(0.5 * (s[1:] + s[:-1]), v, side="right"), 0, len(s) - 1)
        err = (t - alpha * s[idx]) ** 2
        mc = 0.5 * err.mean()                     # D covers the half-line: half the mass
        assert abs(o.D_laplace(alpha, b, k) - mc) <= 4 * 0.5 * err.std() / math.sqrt(t.size)


@pytest.mark.parametrize("b", [3, 4])
def test_laplace_alpha_star_scale_identity(b):
    # the (b, b-1) set is the (b, b-2) set halved, for any density
    a1, d1 = o.alpha_star_laplace(b, b - 1)
    a2, d2 = o.alpha_star_laplace(b, b - 2)
    assert abs(a1 - 2.0 * a2) <= 1e-7 * a1
    assert abs(d1 - d2) <= 1e-12


def test_laplace_D_limits():
    # every value projects to (nearly) 0 as alpha -> 0 (the clip) and as
    # alpha -> infinity: D -> E[t^2] / 2 = 1/2
    assert abs(o.D_laplace(1e-9, 4, 2) - 0.5) < 1e-6
    assert abs(o.D_laplace(1e3, 4, 2) - 0.5) < 1e-6       # one wide Simpson cell


def test_histogram_bins_follow_their_fp32_definition():
    rng = np.random.default_rng(3)
    x = np.concatenate([rng.normal(2.0, 3.0, 100000).astype(np.float32), np.float32([np.nan, np.inf, -np.inf, 2.0])])
    mean, spread, nb, tmax = 2.0000001, 2.9999, 1000, 8.0
    got = o.histogram_abs(x, True, mean, spread, nb, tmax)
    scale = np.float32(nb) / (np.float32(tmax) * np.float32(spread))
    xv = x[~np.isnan(x)]
    u = np.abs(xv - np.float32(mean)) * scale
    bins = np.where(u < nb, np.floor(u), nb - 1).astype(np.int64)
    assert np.array_equal(got, np.bincount(bins, minlength=nb).astype(np.uint64))


def test_histogram_D_of_one_bin_is_the_plain_integral():
    # all mass in one bin [e0, e1): D = (1/2) (1/w) int (t - alpha q(t))^2 dt
    nb, tmax, b, k = 64, 4.0, 4, 2
    counts = np.zeros(nb, np.uint64)
    counts[13] = 1000
    w = tmax / nb
    t = 13 * w + (np.arange(2_000_000) + 0.5) * (w / 2_000_000)     # midpoint rule
    s = o.set_nonneg(b, k)
    for alpha in (0.1, 0.37, 1.3):
        idx = np.clip(np.searchsorted(0.5 * (s[1:] + s[:-1]), t / alpha, side="right"), 0, len(s) - 1)
        ref = 0.5 * np.mean((t - alpha * s[idx]) ** 2)
        assert abs(o.D_hist(alpha, counts, tmax, b, k) - ref) <= 1e-9 * max(ref, 1e-12) + 1e-15


def test_histogram_alpha_star_of_gaussian_data_is_table_1():
    # a histogram of 2^23 N(0,1) values recovers the alpha* of Table 1 (D is
    # flat near its minimum, so a sample moves alpha* by about a percent)
    x = np.random.default_rng(4).normal(size=1 << 23).astype(np.float32)
    _, st = o.calibrate(x, 4, 2, True)
    c = o.histogram_abs(x, True, st[0], st[1], 8192, 16.0)
    for (b, k), ref in [((4, 2), 1.4136), ((5, 2), 0.4828), ((3, 1), 1.3015)]:
        a, _ = o.alpha_star_hist(c, 16.0, b, k)
        assert abs(a - ref) <= 0.02 * ref


# ----------------------------------------- quantisation-aware training ---

def test_dn_backward_is_the_derivative_of_dn():
    # central finite differences of L(x) = sum_i w_i x_hat_i(x), x_hat = DN(x)
    # in fp64 (mean and sigma recomputed from the perturbed x)
    rng = np.random.default_rng(12)
    x = rng.normal(1.5, 2.0, 40)
    w = rng.normal(size=40)

    def loss(v):
        mu = v.mean()
        sig = np.sqrt(((v - mu) ** 2).mean())
        return float(np.dot(w, (v - mu) / (sig + 1e-7)))

    mu = x.mean()
    sig = np.sqrt(((x - mu) ** 2).mean())
    got = o.dn_backward(w.astype(np.float32), x.astype(np.float32), mu, sig).astype(np.float64)
    h = 1e-6
    for j in range(40):
        e = np.zeros(40)
        e[j] = h
        fd = (loss(x + e) - loss(x - e)) / (2 * h)
        # the oracle sees x and g rounded to fp32
        assert abs(got[j] - fd) <= 1e-4 * max(1.0, abs(fd))


def test_dn_backward_kills_shift_and_scale_directions():
    # DN(x + a) = DN(x) and DN(c x) ~ DN(x): the gradient is orthogonal to
    # the constant vector and (for eps -> 0) to x - mu
    rng = np.random.default_rng(13)
    x = rng.normal(0.3, 1.7, 500).astype(np.float32)
    g = rng.normal(size=500).astype(np.float32)
    xd = x.astype(np.float64)
    mu = xd.mean()
    sig = np.sqrt(((xd - mu) ** 2).mean())
    gx = o.dn_backward(g, x, mu, sig).astype(np.float64)
    assert abs(gx.sum()) <= 1e-4 * np.abs(gx).sum()
    assert abs(np.dot(gx, xd - mu)) <= 1e-4 * np.abs(gx).sum() * sig


def test_ema_closed_form():
    # T updates with constant batch statistics b: r_T = b + (1 - gamma)^T (r_0 - b)
    r = np.array([2.0, 0.5])
    b = np.array([-1.0, 3.0])
    g = 0.1
    for _ in range(50):
        r = o.ema(b, r, g)
    exp = b + (1 - g) ** 50 * (np.array([2.0, 0.5]) - b)
    assert np.allclose(r, exp, rtol=1e-13, atol=1e-13)


def test_dn_project_is_dn_then_projection():
    rng = np.random.default_rng(14)
    x = rng.normal(0.7, 2.5, 3000).astype(np.float32)
    mu, sig = float(x.astype(np.float64).mean()), float(x.astype(np.float64).std())
    a = float(np.float32(o.alpha_star(4, 2)[0]))
    codes, xq = o.dn_project(x, mu, sig, a, 4, 2, True)
    xh = (x - np.float32(mu)) / np.float32(sig + 1e-7)           # float32 ops
    assert np.array_equal(codes, o.project_codes(xh, a, 4, 2, True))
    q = o.project_values(xh, a, 4, 2, True)
    assert np.array_equal(xq, (np.float32(a) * q.astype(np.float32)))
