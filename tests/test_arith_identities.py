"""The fp32 identities the decoder kernel uses to keep rounding and bf16 packing off the
conversion pipe, checked exhaustively or densely on the CPU (numpy float32 arithmetic):

* round-to-nearest-even of x through the add of 1.5 * 2^23 and the subtraction back, for the
  ranges the kernel applies it to (quantised codes |x| <= 127 (1 + 2^-24), exp2 arguments in
  [-125, 0]), and the integer in the low bits of the intermediate sum;
* the bf16 encoding of an integer of magnitude <= 127 is the high half of its fp32 encoding.
"""
import numpy as np

MAGIC = np.float32(12582912.0)  # 1.5 * 2^23


def _round_magic(x):
    t = (x + MAGIC).astype(np.float32)
    return t, (t - MAGIC).astype(np.float32)


def _dense_grid(lo, hi):
    # every float32 in [lo, hi] around the half-integers, plus a uniform sample
    halves = np.arange(2 * lo, 2 * hi + 1, dtype=np.float64) / 2
    h32 = halves.astype(np.float32)
    near = [h32]
    a, b = h32.copy(), h32.copy()
    for _ in range(64):
        a = np.nextafter(a, np.float32(-np.inf))
        b = np.nextafter(b, np.float32(np.inf))
        near += [a, b]
    rng = np.random.default_rng(1)
    near.append(rng.uniform(lo, hi, 1_000_000).astype(np.float32))
    x = np.concatenate(near)
    return x[(x >= lo) & (x <= hi)]


def test_magic_round_is_rint_ties_to_even():
    x = _dense_grid(-128, 128)
    t, n = _round_magic(x)
    assert np.array_equal(n, np.rint(x))
    # the integer n sits in the low bits of t
    assert np.array_equal(t.view(np.int32) - 0x4B400000, np.rint(x).astype(np.int32))
    # ties go to even
    ties = np.array([-2.5, -1.5, -0.5, 0.5, 1.5, 2.5, 126.5], np.float32)
    assert _round_magic(ties)[1].tolist() == [-2.0, -2.0, -0.0, 0.0, 2.0, 2.0, 126.0]


def test_magic_round_on_exp2_arguments():
    x = _dense_grid(-125, 0)
    t, n = _round_magic(x)
    assert np.array_equal(n, np.rint(x))
    f = (x - n).astype(np.float32)
    assert np.all(np.abs(f) <= 0.5)


def test_bf16_of_small_integers_is_high_half():
    v = np.arange(-127, 128, dtype=np.float32)
    bits = v.view(np.uint32)
    assert np.all((bits & 0xFFFF) == 0)  # nothing below the bf16 mantissa, so no rounding happens
    hi = (bits >> 16).astype(np.uint16)
    back = (hi.astype(np.uint32) << 16).view(np.float32)
    assert np.array_equal(back, v)
