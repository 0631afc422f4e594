"""The arithmetic of the FP64 product-sum's carry (the drain's overflow path)
checked in IEEE FP32 on the CPU, independent of the kernel: values that are
integer multiples of a unit u with |x| <= 2^24 u (a running sum below the
exact bound, or one chunk partial) split by the add-subtract projection with
the constant 1.5 * 2^35 u into a multiple of 2^12 u and a remainder of at
most 2^11 u, both exact; a coarse sum that takes the two coarse parts of a
running sum and a partial per carry stays exact for 2^11 carries (below
2^36 u).  Also the product-sums' short FP32 -> FP64 widening for zero and
normal values, restated on the bit patterns and checked against numpy's
conversion."""
import numpy as np

F = np.float32


def _split(x, u):
    cm = F(1.5 * 2.0**35) * u
    h = (x + cm) - cm
    return h, x - h


def test_split_is_exact_and_on_the_grid():
    rng = np.random.default_rng(1)
    for e in (-120, -30, 0, 40, 80):
        u = F(2.0**e)
        n = rng.integers(-2**24, 2**24 + 1, size=200000)
        n = np.concatenate([n, [0, 1, -1, 2**11, -2**11, 2**11 + 1, 2**24, -2**24, 3 * 2**11, 2**24 - 1]])
        x = n.astype(np.float64) * float(u)
        assert np.array_equal(x.astype(F).astype(np.float64), x)      # the inputs are exact FP32 values
        xf = x.astype(F)
        h, l = _split(xf, u)
        hi_units = h.astype(np.float64) / float(u)
        lo_units = l.astype(np.float64) / float(u)
        assert np.array_equal(hi_units + lo_units, n.astype(np.float64))            # exact split
        assert np.all(np.mod(hi_units, 2**12) == 0)                                  # coarse part on 2^12 u
        assert np.all(np.abs(lo_units) <= 2**11)                                     # remainder <= 2^11 u


def test_coarse_sum_stays_exact_for_2048_carries():
    rng = np.random.default_rng(2)
    u = F(2.0**-40)
    n = rng.integers(2**23, 2**24 + 1, size=(2048, 2))             # worst case: all large, one sign
    s2, exact = F(0), 0
    for a, b in n:
        h1, _ = _split(F(float(a) * float(u)), u)
        h2, _ = _split(F(float(b) * float(u)), u)
        c = F(h1 + h2)
        assert float(c) == float(h1) + float(h2)                     # the two coarse parts add exactly
        s2 = F(s2 + c)
        exact += int(round(float(c) / float(u)))
    assert int(round(float(s2) / float(u))) == exact
    assert abs(exact) < 2**36


def _widen_normal(x):
    """The FP64 product-sum's short FP32 -> FP64 widening restated on the bit
    patterns: rebias the exponent field by 1023 - 127 and keep the
    significand; zeros keep their sign."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    a = u & 0x7FFFFFFF
    hi = (u & 0x80000000) | np.where(a != 0, (a >> 3) + 0x38000000, 0)
    lo = (u << 29) & 0xFFFFFFFF
    return ((hi << 32) | lo).view(np.float64)


def test_short_widening_is_exact_for_zero_and_normal_values():
    rng = np.random.default_rng(3)
    bits = rng.integers(0, 2**32, size=400000, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    e = (bits >> 23) & 0xFF
    x = x[(e > 0) & (e < 255)]                                  # normal values only
    x = np.concatenate([x, np.float32([0.0, -0.0, 2.0**-126, -2.0**-126, 3.4028235e38, -1.0, 1.0])])
    w = _widen_normal(x)
    assert np.array_equal(w.view(np.uint64), x.astype(np.float64).view(np.uint64))
