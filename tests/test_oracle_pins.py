"""Pins of the CPU oracle against what the paper and the mathematics fix.

Nothing here re-types the oracle's formulas: each check uses an independent
characterisation (exact rational arithmetic, a library rounding routine,
closed-form special cases, brute force on tiny inputs, hand-derived golden
values from ``tests/golden``).
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- helpers
def exact_bf16_rne(x: Fraction):
    """RNE of a rational to BF16 (8-bit significand, FP32 exponent range), exact."""
    if x == 0:
        return Fraction(0)
    s = -1 if x < 0 else 1
    a = abs(x)
    E = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** E > a:
        E -= 1                                  # now 2^E <= a < 2^(E+1)
    E = max(E, -126)
    q = Fraction(2) ** (E - 7)
    r = round(a / q) * q                        # Fraction.__round__ ties to even
    if r >= Fraction(2) ** 128:
        return s * math.inf
    return s * r


def frac_val(bits):
    return Fraction(oracle.bf16_value(int(bits)))


def grid_round(x: Fraction, e: int) -> Fraction:
    """Round x to the nearest multiple of 2^e, ties to even (exact)."""
    q = Fraction(2) ** e
    return round(x / q) * q


# ------------------------------------------------------------ fl_BF16 pins
def test_fl_bf16_golden_values():
    n = 0
    with open(os.path.join(GOLDEN, "bf16_rounding.txt")) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            expr, hexbits, _ = [t.strip() for t in line.split("|")]
            x = float(eval(expr))  # literal arithmetic on powers of two, exact in double
            assert oracle.fl_bf16(x) == int(hexbits, 16), (expr, hex(oracle.fl_bf16(x)))
            n += 1
    assert n >= 14


def test_fl_bf16_matches_library_rne_on_normal_floats():
    """torch's float32 -> bfloat16 cast is IEEE round-to-nearest-even."""
    rng = np.random.default_rng(7)
    bits = rng.integers(0, 2**32, size=200_000, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    e = (bits >> 23) & 0xFF
    x = x[(e > 0) & (e < 0xFE)]                 # normal, far from overflow
    planes, _ = oracle.split_f32(x.reshape(1, -1))
    ref = torch.from_numpy(x.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(planes[0, 0], ref)


def test_fl_bf16_matches_exact_rational_rounding():
    """Independent exact rounding (Fractions) incl. subnormals, ties and overflow."""
    rng = np.random.default_rng(11)
    vals = []
    for _ in range(600):
        e = int(rng.integers(-140, 129))
        m = int(rng.integers(0, 2**52))
        vals.append(math.ldexp(1 + m / 2**52, e) * (1 if rng.random() < 0.5 else -1))
    for _ in range(300):                        # exact ties at random binades
        e = int(rng.integers(-133, 120))
        k = int(rng.integers(128, 256))
        vals.append(math.ldexp(k + 0.5, e - 7))
    for x in vals:
        want = exact_bf16_rne(Fraction(x))
        got = oracle.bf16_value(oracle.fl_bf16(x))
        if isinstance(want, float):
            assert math.isinf(got) and math.copysign(1, got) == math.copysign(1, want)
        else:
            assert Fraction(got) == want, (x, got, want)


def test_ceil_log2():
    for k in range(-130, 130):
        p = math.ldexp(1.0, k)
        assert oracle.ceil_log2(p) == k
        assert oracle.ceil_log2(p * (1 + 2**-52)) == k + 1
        assert oracle.ceil_log2(p * (1 - 2**-53)) == k
    assert oracle.ceil_log2(3.0) == 2 and oracle.ceil_log2(0.3) == -1


# --------------------------------------------------------- FP32 split pins
def _random_normal_floats(n, seed, emin=-100, emax=100):
    rng = np.random.default_rng(seed)
    mant = rng.integers(0, 2**23, size=n, dtype=np.uint32)
    exp = rng.integers(127 + emin, 127 + emax, size=n).astype(np.uint32)
    sign = rng.integers(0, 2, size=n).astype(np.uint32)
    return ((sign << 31) | (exp << 23) | mant).view(np.float32)


def test_split_f32_reconstructs_exactly():
    """Eq. (fp32split), Section 4.2: the three slices sum back to x exactly for
    normal inputs away from underflow (R_A = 0), each residual step shrinks by
    at least u_BF16 = 2^-8, and the split is exact slice by slice."""
    x = _random_normal_floats(300_000, 3).reshape(300, 1000)
    planes, flags = oracle.split_f32(x)
    assert flags == 0
    a = [oracle.bf16_to_f32(planes[r]).astype(np.float64) for r in range(3)]
    assert np.array_equal(a[0] + a[1] + a[2], x.astype(np.float64))
    assert np.all(np.abs(a[1]) <= np.abs(a[0]) * 2.0**-8)
    assert np.all(np.abs(a[2]) <= np.abs(a[1]) * 2.0**-8)


def test_split_f32_uniform_workload_and_flags():
    A = synth.uniform_f32(0, 0, (64, 96))
    planes, flags = oracle.split_f32(A)
    assert flags == 0
    s = sum(oracle.bf16_to_f32(planes[r]).astype(np.float64) for r in range(3))
    assert np.array_equal(s, A.astype(np.float64))
    bad = A.copy()
    bad[3, 5] = np.nan
    assert oracle.split_f32(bad)[1] & oracle.FLAG_NONFINITE
    big = A.copy()
    big[0, 0] = np.float32(3.4e38)              # rounds past the largest BF16
    assert oracle.split_f32(big)[1] & oracle.FLAG_SLICE


# --------------------------------------------------------- FP64 split pins
def _check_fp64_split_exact(X):
    """Independent exact restatement of Eq. (fp64split) in rationals.

    With sigma = 2^(v+45) and |R| <= 2^v, fl64(R + sigma) lies in the binade
    [2^(v+45), 2^(v+46)) when R >= 0 (spacing 2^(v-7)) and in
    [2^(v+44), 2^(v+45)] when R < 0 (spacing 2^(v-8)); the subtraction of sigma
    is exact (Sterbenz).  So slice r is the exact residual rounded to nearest
    (ties to even) on the grid 2^(v_r-7) for R >= 0 and 2^(v_r-8) for R < 0:
    at most 256 units, hence always 8 significant bits.  Also v_r bounds the
    residual max, and the residual after six slices is at most 2^(v_5 - 8)."""
    planes, v, flags = oracle.split_f64(X)
    assert flags == 0
    R = [[Fraction(float(t)) for t in row] for row in X]
    for r in range(6):
        m = max(abs(t) for row in R for t in row)
        if m == 0:
            assert all(v[t] == oracle.ZERO_LEVEL for t in range(r, 6))
            assert not planes[r:].any()
            return
        vr = int(v[r])
        assert Fraction(2) ** (vr - 1) < m <= Fraction(2) ** vr        # v = ceil(log2 max)
        if r:
            assert vr <= int(v[r - 1]) - 8                              # residual shrinks by 2^-8
        for i, row in enumerate(R):
            for j, t in enumerate(row):
                z = grid_round(t, vr - 7 if t >= 0 else vr - 8)
                assert frac_val(planes[r, i, j]) == z
                row[j] = t - z
    m6 = max(abs(t) for row in R for t in row)
    assert m6 <= Fraction(2) ** (int(v[5]) - 8)


def test_split_f64_uniform_exact():
    _check_fp64_split_exact(synth.uniform_f64(1, 0, (12, 17)))


def test_split_f64_scaled_class_exact():
    _check_fp64_split_exact(synth.scaled_f64(5, 0, 4.0, (9, 13)))


def test_split_f64_levels_drop_by_eight_on_uniform_data():
    _, v, flags = oracle.split_f64(synth.uniform_f64(1, 0, (128, 128)))
    assert flags == 0 and v[0] == 0
    assert list(np.diff(v)) == [-8] * 5


def test_split_f64_integer_inputs_stop_early():
    """Integers with |x| <= 100: the first slice is x itself (grid 2^0), the
    residual is zero and every later slice is zero (Section 4.3 early stop)."""
    rng = np.random.default_rng(2)
    X = rng.integers(-100, 101, size=(20, 30)).astype(np.float64)
    X[0, 0] = 100.0
    planes, v, flags = oracle.split_f64(X)
    assert flags == 0 and v[0] == 7
    assert all(t == oracle.ZERO_LEVEL for t in v[1:])
    assert np.array_equal(oracle.bf16_to_f32(planes[0]).astype(np.float64), X)
    assert not planes[1:].any()


def test_split_f64_zero_matrix_and_domain_flags():
    planes, v, flags = oracle.split_f64(np.zeros((4, 5)))
    assert flags == 0 and not planes.any() and all(t == oracle.ZERO_LEVEL for t in v)
    X = synth.uniform_f64(3, 0, (8, 8))
    for val, bit in [(np.nan, oracle.FLAG_NONFINITE), (np.inf, oracle.FLAG_NONFINITE),
                     (2.0**-127, oracle.FLAG_RANGE), (2.0**129, oracle.FLAG_RANGE)]:
        Y = X.copy()
        Y[2, 3] = val
        assert oracle.split_f64(Y)[2] & bit, val
    # a nonzero residual slice below the normal BF16 range (Section 3.1)
    Y = np.full((2, 2), 2.0**-120)
    Y[0, 0] = 2.0**-120 + 2.0**-140
    assert oracle.split_f64(Y)[2] & oracle.FLAG_SLICE
    # the top of the stated domain rounds to 2^128 in slice 0: not a BF16 value
    Y = np.array([[(2 - 2.0**-7) * 2.0**127]])
    assert oracle.split_f64(Y)[2] & oracle.FLAG_SLICE


# ---------------------------------------------------------- product sets
def _golden_sets():
    out = {}
    with open(os.path.join(GOLDEN, "product_sets.txt")) as f:
        for line in f:
            if line.startswith("#") or ":" not in line:
                continue
            k, val = line.split(":", 1)
            out[k.strip()] = val.strip()
    return out


def test_product_sets_match_paper():
    g = _golden_sets()
    counts = {int(a): int(b) for a, b in (t.split(":") for t in g["counts"].split())}
    for d, n in counts.items():
        pairs = oracle.products(64, n)
        assert len(pairs) == n == len(set(pairs))
        assert set(pairs) == {(i, j) for i in range(6) for j in range(6) if i + j < d}
        diag = [i + j for i, j in pairs]
        assert diag == sorted(diag)                          # diagonal by diagonal
        for l in range(d):
            assert [i for i, j in pairs if i + j == l] == list(range(l + 1))
    chain = [tuple(int(t) for t in p.split(",")) for p in g["fp32_chain"].split()]
    assert oracle.products(32, 6) == chain
    assert set(chain) == {(i, j) for i in range(3) for j in range(3) if i + j < 3}
    loads = 2 + sum(1 for a, b in zip(chain, chain[1:]) if (a[0] == b[0]) != (a[1] == b[1]))
    assert loads == int(g["fp32_chain_loads"])
    with pytest.raises(ValueError):
        oracle.products(64, 7)


# ------------------------------------------------------- product-sum pins
def test_fp64_chunk_partials_are_exact():
    """Section 5.2: BF16 x BF16 products are exact in FP32; with slices on the
    grid of Eq. (fp64split) every 256-long chunk partial is exact too."""
    for X, Y in [synth.gemm_inputs("f64", 24, 20, 600, 1),
                 synth.gemm_inputs("f64_scaled", 16, 16, 520, 5, phi=4.0),
                 (np.ones((8, 512)), np.ones((512, 8)))]:
        Ap, _, _ = oracle.split_f64(X)
        Bp, _, _ = oracle.split_f64(Y)
        _, bad = oracle.prodsum_f64(Ap, Bp, 21, check_exact=True)
        assert bad == 0


def _exact_slice_sum(Ap, Bp, pairs):
    """Exact sum_{(i,j) in pairs} A_i B_j in rationals (tiny sizes only)."""
    a = [[[frac_val(t) for t in row] for row in Ap[s]] for s in range(Ap.shape[0])]
    b = [[[frac_val(t) for t in row] for row in Bp[s]] for s in range(Bp.shape[0])]
    M, K, N = Ap.shape[1], Ap.shape[2], Bp.shape[2]
    out = [[Fraction(0)] * N for _ in range(M)]
    absout = [[Fraction(0)] * N for _ in range(M)]
    for (i, j) in pairs:
        for m in range(M):
            for n in range(N):
                for k in range(K):
                    p = a[i][m][k] * b[j][k][n]
                    out[m][n] += p
                    absout[m][n] += abs(p)
    return out, absout


@pytest.mark.parametrize("order", ["chunk", "product"])
@pytest.mark.parametrize("K", [8, 300])
def test_brute_force_fp64_against_exact_retained_sum(K, order):
    """8x8xK brute force: the oracle's FP64 product-sum equals the exact sum of
    the retained products up to the FP64 rounding of its additions (in either
    summation order of the exact chunk partials)."""
    A, B = synth.gemm_inputs("f64", 8, 8, K, 17)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    nch = -(-K // oracle.KCHUNK)
    for nprod in (6, 21):
        C = oracle.prodsum_f64(Ap, Bp, nprod, order=order)
        S, absS = _exact_slice_sum(Ap, Bp, oracle.products(64, nprod))
        nadd = nch * nprod
        for m in range(8):
            for n in range(8):
                err = abs(Fraction(float(C[m, n])) - S[m][n])
                assert err <= nadd * Fraction(2) ** -53 * absS[m][n] * 2


def test_brute_force_fp32_against_exact_retained_sum():
    A, B = synth.gemm_inputs("f32", 8, 8, 300, 19)
    Ap, _ = oracle.split_f32(A)
    Bp, _ = oracle.split_f32(B)
    C = oracle.prodsum_f32(Ap, Bp)
    S, absS = _exact_slice_sum(Ap, Bp, oracle.products(32, 6))
    for m in range(8):
        for n in range(8):
            err = abs(Fraction(float(C[m, n])) - S[m][n])
            assert err <= (6 * 300 + 2) * Fraction(2) ** -24 * absS[m][n]
    # and the whole path is FP32-accurate against the exact product
    hi, lo = oracle.ref_dd(A.astype(np.float64), B.astype(np.float64))
    absAB = np.abs(A.astype(np.float64)) @ np.abs(B.astype(np.float64))
    assert np.all(np.abs((C - hi) - lo) <= 1e-5 * absAB)


def test_fp32_bf16_exact_integers_give_exact_product():
    """A_1 = A_2 = 0 for small integers; products and sums stay exact integers."""
    rng = np.random.default_rng(4)
    for K in (200, 700):
        A = rng.integers(-12, 13, size=(20, K)).astype(np.float32)
        B = rng.integers(-12, 13, size=(K, 24)).astype(np.float32)
        C, flags = oracle.gemm_f32(A, B)
        assert flags == 0
        assert np.array_equal(C.astype(np.int64), A.astype(np.int64) @ B.astype(np.int64))


@pytest.mark.parametrize("order", ["chunk", "product"])
@pytest.mark.parametrize("nprod", [6, 10, 15, 21])
def test_fp64_two_slice_integers_give_exact_product(nprod, order):
    """Integers |x| <= 2^15 need two slices; with d >= 3 all of A0B0, A0B1,
    A1B0, A1B1 are retained, so the result is the exact product."""
    rng = np.random.default_rng(5)
    A = rng.integers(-2**15, 2**15 + 1, size=(16, 520)).astype(np.float64)
    B = rng.integers(-2**15, 2**15 + 1, size=(520, 12)).astype(np.float64)
    C, flags = oracle.gemm_f64(A, B, nprod, order=order)
    assert flags == 0
    assert np.array_equal(C, (A.astype(np.int64) @ B.astype(np.int64)).astype(np.float64))


@pytest.mark.parametrize("order", ["chunk", "product"])
@pytest.mark.parametrize("nprod", [6, 10, 15])
def test_fp64_omitted_products_term(nprod, order):
    """Integers up to 2^23 need three slices, all integer-valued.  Every sum is
    then exact, so C_hat = A.B - E_omit exactly, with E_omit of Eq. (omit)."""
    rng = np.random.default_rng(6)
    A = rng.integers(-2**23, 2**23, size=(6, 40)).astype(np.float64)
    B = rng.integers(-2**23, 2**23, size=(40, 5)).astype(np.float64)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    a = [oracle.bf16_to_f32(Ap[s]).astype(np.int64) for s in range(6)]
    b = [oracle.bf16_to_f32(Bp[s]).astype(np.int64) for s in range(6)]
    assert all(np.array_equal(x.astype(np.float64), oracle.bf16_to_f32(Ap[s])) for s, x in enumerate(a))
    retained = set(oracle.products(64, nprod))
    omit = sum(a[i] @ b[j] for i in range(6) for j in range(6) if (i, j) not in retained)
    C = oracle.prodsum_f64(Ap, Bp, nprod, order=order)
    exact = A.astype(np.int64) @ B.astype(np.int64)
    assert np.array_equal(C.astype(np.int64), exact - omit)
    assert np.array_equal(C, (exact - omit).astype(np.float64))


# ------------------------------------------------- reference and metrics
def test_ref_dd_against_exact():
    A, B = synth.gemm_inputs("f64_scaled", 5, 4, 33, 8, phi=2.0)
    hi, lo = oracle.ref_dd(A, B)
    for m in range(5):
        for n in range(4):
            ex = sum(Fraction(float(A[m, k])) * Fraction(float(B[k, n])) for k in range(33))
            got = Fraction(float(hi[m, n])) + Fraction(float(lo[m, n]))
            scale = sum(abs(Fraction(float(A[m, k])) * Fraction(float(B[k, n]))) for k in range(33))
            assert abs(got - ex) <= scale * Fraction(2) ** -100


def test_error_metrics_hand_example():
    C = np.array([[1.0, 2.0], [3.0, 4.0]])
    hi = np.array([[1.0, 2.0], [3.0, 5.0]])
    lo = np.zeros_like(hi)
    absAB = np.array([[1.0, 0.0], [2.0, 4.0]])
    C2 = C.copy()
    C2[0, 1] = 2.5
    e = oracle.errors(C2, hi, lo, absAB)
    assert e["e_F"] == pytest.approx(math.sqrt(0.25 + 1.0) / math.sqrt(39.0))
    assert e["e_max"] == 1.0
    assert e["e_scaled"] == 0.25                 # |4-5| / 4
    assert e["e_abs_zero_den"] == 0.5            # zero denominator reported separately


def test_accuracy_magnitudes_uniform_n256():
    """Regression band for the literal whole-matrix split on uniform inputs:
    each retained diagonal gains about 2^-8 (u_BF16); FP32 mode is FP32-level."""
    A, B = synth.gemm_inputs("f64", 256, 256, 256, 1)
    hi, lo = oracle.ref_dd(A, B)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    got = {n: oracle.errors(oracle.prodsum_f64(Ap, Bp, n), hi, lo)["e_F"] for n in (6, 10, 15, 21)}
    band = {6: 8.5e-8, 10: 3.6e-10, 15: 1.5e-12, 21: 6.4e-15}
    for n, ref in band.items():
        assert ref / 2 < got[n] < ref * 2, (n, got[n])
    for n in (6, 10, 15):
        ratio = got[n] / got[{6: 10, 10: 15, 15: 21}[n]]
        assert 2**6 < ratio < 2**10
    A32, B32 = synth.gemm_inputs("f32", 256, 256, 256, 0)
    C32, _ = oracle.gemm_f32(A32, B32)
    hi, lo = oracle.ref_dd(A32.astype(np.float64), B32.astype(np.float64))
    # one FP32 accumulator takes 6 x 256 sequential additions per chunk: a
    # random-walk estimate of the rounding error is sqrt(1536) * u32/sqrt(12)
    # relative, about 7e-7, the same order as the paper's 3e-7 against SGEMM.
    assert 1e-7 < oracle.errors(C32, hi, lo)["e_F"] < 1.2e-6


def test_fp32_kchunk_is_256():
    """B_K = 256 (Section 6.1) fixes where FP32 rounding happens: each chunk
    is accumulated on its own, then added into the output accumulator.
    Row 0: 256 ones then 256 x 2^-22.  Per-chunk: 256 + 256*2^-22 = 256 + 2^-14
    (exact); one long accumulator would round every 2^-22 away (ulp(256) = 2^-15).
    Row 1: 128 ones then 128 x 2^-22 inside the first chunk: each 2^-22 is lost
    against 128 (ulp 2^-16), giving exactly 128; a 128-long chunk would keep
    128 + 2^-15."""
    A = np.zeros((2, 512), dtype=np.float32)
    A[0, :256] = 1.0
    A[0, 256:] = 2.0**-22
    A[1, :128] = 1.0
    A[1, 128:256] = 2.0**-22
    B = np.ones((512, 1), dtype=np.float32)
    C, flags = oracle.gemm_f32(A, B)
    assert flags == 0
    assert C[0, 0] == np.float32(256 + 2.0**-14)
    assert C[1, 0] == np.float32(128.0)


def test_fp64_partials_exact_at_the_2pow24_edge():
    """Negative entries sit on the finer grid 2^(v-8): -255/256 is 255 units,
    a product is up to 2^16 units and a 256-long chunk up to 2^24 units, the
    edge of exact FP32.  Here chunk 0 sums to 16646145 units (24 bits); over
    512 terms the FP32 sum would round (odd, > 2^24), per chunk it stays exact
    and the FP64 result is the exact product."""
    K = 512
    A = np.full((1, K), -255 / 256)
    B = np.full((K, 1), -255 / 256)
    B[0, 0] = -254 / 256
    Ap, va, fa = oracle.split_f64(A)
    Bp, vb, fb = oracle.split_f64(B)
    assert fa == fb == 0 and va[0] == vb[0] == 0
    C, bad = oracle.prodsum_f64(Ap, Bp, 6, check_exact=True)
    assert bad == 0
    assert C[0, 0] == (65025 * 511 + 255 * 254) * 2.0**-16
    assert (65025 * 255 + 255 * 254) > 2**23          # chunk 0 needs all 24 bits


def test_fp64_orders_agree_within_fp64_rounding():
    """The two summation orders add the same exact chunk partials; they may
    differ only by the FP64 rounding of the additions, and the product-outer
    order rounds less often (one addition per product instead of one per
    chunk and product)."""
    A, B = synth.gemm_inputs("f64_scaled", 40, 36, 1500, 7, phi=2.0)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    hi, lo = oracle.ref_dd(A, B)
    nch = -(-1500 // oracle.KCHUNK)
    for nprod in (6, 21):
        Cc = oracle.prodsum_f64(Ap, Bp, nprod, order="chunk")
        Cp = oracle.prodsum_f64(Ap, Bp, nprod, order="product")
        a = [oracle.bf16_to_f32(Ap[s]).astype(np.float64) for s in range(6)]
        b = [oracle.bf16_to_f32(Bp[s]).astype(np.float64) for s in range(6)]
        absP = sum(np.abs(a[i]) @ np.abs(b[j]) for i, j in oracle.products(64, nprod))
        assert np.all(np.abs(Cc - Cp) <= 2 * nprod * nch * 2.0**-53 * absP)
        ec, ep = oracle.errors(Cc, hi, lo), oracle.errors(Cp, hi, lo)
        assert ep["e_F"] <= 1.01 * ec["e_F"] + 1e-300


# ----------------------------------------------------- general GEMM (gemm_ex)
def _exact_ex(A_eff, B_eff, alpha, beta, C):
    """alpha op(A) op(B) + beta C in exact rational arithmetic."""
    from fractions import Fraction
    M, K = A_eff.shape
    N = B_eff.shape[1]
    out = np.empty((M, N), dtype=object)
    for i in range(M):
        for j in range(N):
            p = sum(Fraction(float(A_eff[i, k])) * Fraction(float(B_eff[k, j])) for k in range(K))
            out[i, j] = Fraction(alpha) * p + (Fraction(beta) * Fraction(float(C[i, j])) if beta != 0 else 0)
    return out


@pytest.mark.parametrize("dtype,nprod", [(np.float32, None), (np.float64, 6)])
@pytest.mark.parametrize("opA,opB", [(0, 0), (0, 1), (1, 0), (1, 1)])
def test_gemm_ex_exact_on_small_integers(dtype, nprod, opA, opB):
    """Small integers are BF16-exact (one slice), so the emulated product is
    A B exactly (K <= 256 keeps FP32 sums exact); with alpha, beta powers of
    two the epilogue is exact too.  The oracle must then return
    alpha op(A) op(B) + beta C exactly, for each placement of the operands."""
    rng = np.random.default_rng(17 + 2 * opA + opB)
    M, N, K = 7, 5, 40
    A_eff = rng.integers(-16, 17, size=(M, K)).astype(dtype)
    B_eff = rng.integers(-16, 17, size=(K, N)).astype(dtype)
    C = rng.integers(-100, 101, size=(M, N)).astype(dtype)
    A = np.ascontiguousarray(A_eff.T) if opA else A_eff
    B = np.ascontiguousarray(B_eff.T) if opB else B_eff
    for alpha, beta in [(1.0, 0.0), (0.5, -2.0), (-4.0, 0.25), (2.0, 0.0)]:
        got, flags = oracle.gemm_ex(opA, opB, alpha, A, B, beta, C, nprod=nprod)
        assert flags == 0 and got.dtype == dtype
        want = _exact_ex(A_eff, B_eff, alpha, beta, C)
        assert all(got[i, j] == float(want[i, j]) for i in range(M) for j in range(N)), (alpha, beta)


def test_gemm_ex_beta_zero_does_not_read_c():
    A, B = synth.gemm_inputs("f64", 9, 6, 30, 5)
    C = np.full((9, 6), np.nan)
    got, _ = oracle.gemm_ex(0, 0, 3.0, A, B, 0.0, C, nprod=10)
    P, _ = oracle.gemm_f64(A, B, 10)
    assert np.array_equal(got, 3.0 * P)


# --------------------------------------- per-row / per-column levels (NEXT-2)
def test_split_rows_commutes_with_power_of_two_row_scaling():
    """With one set of levels per row, scaling a row by 2^e scales every slice
    of that row by 2^e and shifts its levels by e, exactly.  A split that
    shared levels across rows would round the small rows on the large rows'
    grid and fail this."""
    rng = np.random.default_rng(31)
    U = synth.uniform_f64(31, 0, (12, 40))
    e = rng.integers(-60, 60, size=12)
    X = U * np.ldexp(1.0, e)[:, None]
    P, v, f = oracle.split_f64_rows(X)
    Pu, vu, fu = oracle.split_f64_rows(U)
    assert f == fu == 0
    vals = (P.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    vals_u = (Pu.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert np.array_equal(vals, vals_u * np.ldexp(1.0, e)[None, :, None])
    assert np.array_equal(v, vu + e[:, None])


def test_split_rows_levels_are_the_row_maxima():
    """v[i, r] = ceil(log2 max_j |A^(r)_ij|) row by row, and a row that is
    exact after r slices stops there (zero levels), independently of other rows."""
    X = synth.uniform_f64(32, 0, (5, 30))
    X[2] = np.round(X[2] * 64)                      # integers: one slice
    P, v, _ = oracle.split_f64_rows(X)
    for i in range(5):
        R = X[i].copy()
        for r in range(6):
            m = np.max(np.abs(R))
            if m == 0:
                assert v[i, r] == oracle.ZERO_LEVEL
                continue
            assert 2.0 ** (v[i, r] - 1) < m <= 2.0 ** v[i, r]
            R = R - (P[r, i].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    assert v[2, 1] == oracle.ZERO_LEVEL


def test_gemm_rowcol_commutes_with_row_and_column_scaling():
    """Per-row levels for A and per-column levels for B make the emulated
    product of D_A U and V D_B (D diagonal powers of two) equal to
    D_A (U V) D_B exactly, with every chunk partial exact in its own unit; one
    level per matrix instead rounds the small rows and columns on the large
    ones' grid and loses them (far larger scaled error, same product count)."""
    M, N, K = 24, 20, 300
    U, V = synth.gemm_inputs("f64", M, N, K, 4)
    rng = np.random.default_rng(33)
    # ea + eb >= -30 keeps every product unit 2^(vA_5 + vB_5 - 16) a normal FP32 number
    ea, eb = rng.integers(-15, 41, size=M), rng.integers(-15, 41, size=N)
    A, B = U * np.ldexp(1.0, ea)[:, None], V * np.ldexp(1.0, eb)[None, :]
    Ap, _, _ = oracle.split_f64_rows(A)
    Bt, _, _ = oracle.split_f64_rows(np.ascontiguousarray(B.T))
    _, bad = oracle.prodsum_f64(Ap, np.ascontiguousarray(Bt.transpose(0, 2, 1)), 21, check_exact=True)
    assert bad == 0
    for nprod in (6, 10, 21):
        C1, f1 = oracle.gemm_f64_rowcol(A, B, nprod)
        C0, f0 = oracle.gemm_f64_rowcol(U, V, nprod)
        assert f1 == f0 == 0
        assert np.array_equal(C1, C0 * np.ldexp(1.0, ea)[:, None] * np.ldexp(1.0, eb)[None, :])
    hi, lo = oracle.ref_dd(A, B)
    absab = np.abs(A) @ np.abs(B)
    e_rc = oracle.errors(oracle.gemm_f64_rowcol(A, B, 10)[0], hi, lo, absab)["e_scaled"]
    e_gl = oracle.errors(oracle.gemm_f64(A, B, 10)[0], hi, lo, absab)["e_scaled"]
    assert e_rc < 1e-3 * e_gl, (e_rc, e_gl)
