"""The projections add their fp32 partial sums in 64-bit fixed point (value
x 2^32), so that the sums do not depend on the order in which contributors
arrive.  The conversion of an fp32 t to round(t) must then be exact.  The
kernels split t = h 2^31 + r with h = rint(t 2^-31), taken from the bits of a
float32 sum with 1.5 2^23, and r = t - h 2^31 (one fused multiply-add), and
round r with one 32-bit conversion.  This checks that arithmetic in float32
(numpy) against exact rounding over the whole range the sums use, ties
included: the claim behind the order-independent reductions."""
import numpy as np

MAGIC = np.float32(12582912.0)  # 1.5 * 2^23


def split_round(t: np.ndarray) -> np.ndarray:
    t = t.astype(np.float32)
    y = (t * np.float32(2.0 ** -31)).astype(np.float32) + MAGIC          # rint(t 2^-31) + magic, one rounding
    h = y.view(np.int32).astype(np.int64) - np.int64(MAGIC.view(np.int32))
    hf = (y - MAGIC).astype(np.float32)                                  # exact
    # fma(hf, -2^31, t): hf * 2^31 is exact, and so is the difference (the
    # argument of the kernel's comment), so float64 gives the fused result
    r = (t.astype(np.float64) - hf.astype(np.float64) * 2.0 ** 31).astype(np.float32)
    assert np.array_equal(r.astype(np.float64), t.astype(np.float64) - hf.astype(np.float64) * 2.0 ** 31)
    return (h << 31) + np.rint(r.astype(np.float64)).astype(np.int64)   # rint: ties to even, as the conversion


def exact_round(t: np.ndarray) -> np.ndarray:
    return np.rint(t.astype(np.float64)).astype(np.int64)  # float32 values are exact in float64


def test_split_rounding_is_exact_across_magnitudes():
    rng = np.random.default_rng(7)
    for e in range(-12, 52):
        mant = rng.uniform(1.0, 2.0, 20000)
        sign = rng.choice([-1.0, 1.0], 20000)
        t = (sign * np.ldexp(mant, e)).astype(np.float32)
        assert np.array_equal(split_round(t), exact_round(t)), e


def test_split_rounding_ties_and_edges():
    k = np.arange(-200000, 200000, dtype=np.float64)
    ties = (k + 0.5).astype(np.float32)
    assert np.array_equal(split_round(ties), exact_round(ties))
    edges = np.array([0.0, -0.0, 0.49999997, -0.49999997, 2.0 ** 30, -(2.0 ** 30), 2.0 ** 31 - 128, 2.0 ** 31,
                      -(2.0 ** 31), 2.0 ** 32 + 512, 2.0 ** 51, -(2.0 ** 51) - 2.0 ** 28], dtype=np.float32)
    assert np.array_equal(split_round(edges), exact_round(edges))


def test_integer_sums_are_order_independent():
    # the point of the exercise: fixed-point sums of the same contributions in
    # any order are identical, fp32 sums are not
    rng = np.random.default_rng(11)
    parts = (rng.standard_normal(64) * 3.0).astype(np.float32)
    fixed = split_round(parts * np.float32(2.0 ** 32))
    orders = [rng.permutation(64) for _ in range(20)]
    sums = {int(fixed[o].sum()) for o in orders}
    assert len(sums) == 1
    f32 = {float(np.float32(0) + np.cumsum(parts[o], dtype=np.float32)[-1]) for o in orders}
    assert len(f32) > 1
