"""The reading behind the tensor-core posterior's operand split, checked on
the CPU with an exact emulation of bf16 rounding (round to nearest, ties to
even, on the top 16 bits of an fp32 word).

Reading: an fp32 value x is split into three bf16 parts
    h = bf16(x),  m = bf16(x - h),  l = bf16(x - h - m),
each difference exact in fp32.  A bf16 holds 8 significant bits; x holds 24,
so x - h holds at most 16 and x - h - m at most 8: l takes the rest whole and
h + m + l == x exactly.  The product keeps h h, h m, m h, h l, l h and m m and
drops m l, l m and l l, each of order 2^-24 of |x y| or below.
"""
import numpy as np

from workloads import Stream


def bf16(x):
    """Round fp32 values to bf16 (returned as fp32): nearest, ties to even."""
    b = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) & 0xFFFF0000
    return b.astype(np.uint32).view(np.float32)


def split3(x):
    x = np.asarray(x, np.float32)
    h = bf16(x)
    r1 = (x - h).astype(np.float32)
    m = bf16(r1)
    r2 = (r1 - m).astype(np.float32)
    return h, m, bf16(r2), r1, r2


def samples(n, seed):
    st = Stream(seed, "split")
    mant = st.uniform(n) + 1.0
    expo = np.floor(st.uniform(n) * 120.0) - 60.0
    sign = np.where(st.uniform(n) < 0.5, -1.0, 1.0)
    return (sign * mant * np.exp2(expo)).astype(np.float32)


def test_bf16_rounding_emulation():
    # values worked by hand: 1 + 2^-8 ties to 1 (even), 1 + 3 * 2^-8 ties to 1 + 2^-6 (even), 1 + 2^-7 is exact
    x = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.0 + 2.0 ** -7, 1.0 + 2.0 ** -8 + 2.0 ** -20], np.float32)
    assert bf16(x).tolist() == [1.0, 1.0 + 2.0 ** -6, 1.0 + 2.0 ** -7, 1.0 + 2.0 ** -7]


def test_three_parts_hold_every_bit():
    x = samples(200000, 1)
    h, m, l, r1, r2 = split3(x)
    x64 = x.astype(np.float64)
    # the differences are exact in fp32 and the last part is the remainder whole
    assert np.array_equal(r1.astype(np.float64), x64 - h.astype(np.float64))
    assert np.array_equal(r2.astype(np.float64), r1.astype(np.float64) - m.astype(np.float64))
    assert np.array_equal(l, r2)
    assert np.array_equal(h.astype(np.float64) + m.astype(np.float64) + l.astype(np.float64), x64)
    # each part within 2^-8 of the remainder it rounds (relative to that remainder)
    assert np.all(np.abs(m.astype(np.float64)) <= 2.0 ** -8 * np.abs(h.astype(np.float64)))
    assert np.all(np.abs(l.astype(np.float64)) <= 2.0 ** -8 * np.abs(m.astype(np.float64)) + 0.0)


def test_two_parts_would_not_hold_them():
    """A plausible shortcut (two parts, h + m) loses the last 8 bits."""
    x = samples(20000, 2)
    h, m, l, _, _ = split3(x)
    assert np.any(h.astype(np.float64) + m.astype(np.float64) != x.astype(np.float64))


def test_dropped_products_are_below_fp32_rounding():
    x, y = samples(100000, 3), samples(100000, 4)
    hx, mx, lx, _, _ = split3(x)
    hy, my, ly, _, _ = split3(y)
    f = lambda a: a.astype(np.float64)
    kept = f(hx) * f(hy) + f(hx) * f(my) + f(mx) * f(hy) + f(hx) * f(ly) + f(lx) * f(hy) + f(mx) * f(my)
    exact = f(x) * f(y)
    rel = np.abs(exact - kept) / np.abs(exact)
    assert rel.max() <= 2.0 ** -23          # m l + l m + l l: at most about 2 * 2^-8 * 2^-16 of |x y|
    assert rel.max() > 2.0 ** -40           # and they are not all zero: the products are really dropped
