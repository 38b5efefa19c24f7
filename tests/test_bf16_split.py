"""The three-term bf16 split of an fp32 value that the distillation contractions stage for
the tensor cores (CPU, numpy): hi = bf16(x), mid = bf16(x - hi), lo = bf16(x - hi - mid),
each rounded to nearest even.  Both differences are exact in fp32 and the three terms add
up to x exactly, so products of split operands carry every bit of the fp32 operands; a
two-term split (hi, mid) keeps only about 16 bits."""
import numpy as np

from paper_2608_06411_gb300 import workloads as W


def _bf16(x):
    return W.bf16_bits_to_f32(W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32)))


def _split(x):
    x = np.asarray(x, dtype=np.float32)
    hi = _bf16(x)
    r1 = (x - hi).astype(np.float32)
    mid = _bf16(r1)
    r2 = (r1 - mid).astype(np.float32)
    lo = _bf16(r2)
    return hi, mid, lo, r1, r2


def _values(seed=0, n=200_000):
    rng = np.random.default_rng(seed)
    mant = rng.uniform(1.0, 2.0, n)
    expo = rng.integers(-100, 100, n)
    sign = rng.choice([-1.0, 1.0], n)
    return (sign * mant * np.exp2(expo)).astype(np.float32)


def test_three_terms_add_up_to_x_exactly():
    x = _values()
    hi, mid, lo, r1, r2 = _split(x)
    x64 = x.astype(np.float64)
    # the fp32 differences are exact
    np.testing.assert_array_equal(r1.astype(np.float64), x64 - hi.astype(np.float64))
    np.testing.assert_array_equal(r2.astype(np.float64), r1.astype(np.float64) - mid.astype(np.float64))
    # the last remainder fits in bf16, so hi + mid + lo is x itself
    np.testing.assert_array_equal(lo, r2)
    np.testing.assert_array_equal(hi.astype(np.float64) + mid.astype(np.float64) + lo.astype(np.float64), x64)


def test_terms_shrink_by_the_bf16_precision():
    x = _values(1, 20_000)
    hi, mid, lo, _, _ = _split(x)
    nz = mid != 0
    assert np.all(np.abs(mid[nz]) <= np.abs(hi[nz]) * 2.0 ** -8)
    nz = lo != 0
    assert np.all(np.abs(lo[nz]) <= np.abs(mid[nz]) * 2.0 ** -8)


def test_two_terms_lose_the_low_bits():
    x = _values(2, 20_000)
    hi, mid, _, _, _ = _split(x)
    err = np.abs(hi.astype(np.float64) + mid.astype(np.float64) - x.astype(np.float64)) / np.abs(x.astype(np.float64))
    assert err.max() > 2.0 ** -20                  # far above fp32 rounding (2^-24)
    assert err.max() <= 2.0 ** -16
