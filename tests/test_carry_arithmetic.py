"""The arithmetic of the FP64 product-sum's carry (the drain's overflow path)
checked in IEEE FP32 on the CPU, independent of the kernel: values that are
integer multiples of a unit u with |x| <= 2^24 u (a running sum below the
exact bound, or one chunk partial) split by the add-subtract projection with
the constant 1.5 * 2^35 u into a multiple of 2^12 u and a remainder of at
most 2^11 u, both exact; a coarse sum that takes the two coarse parts of a
running sum and a partial per carry stays exact for 2^11 carries (below
2^36 u)."""
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
