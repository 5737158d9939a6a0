"""The sums of squares' error-free step, restated with exactly rounded fp32
operations and checked against exact rational arithmetic.  No GPU.

The sweep adds each square to a running fp32 sum S by one FMA, t = fl(S + x*x),
and recovers the addition's error from zn = fl(S - t), y = fl(t + zn),
a = fl(S - y) and b = fl(x*x + zn) (a second FMA); C takes a + b.  The claim
the kernels rest on: a + b is S + x^2 - t to within about 3 u^2 t (u = 2^-24)
whether or not the square is exact in fp32, so S + C carries the sum to about
n u^2 of it after n steps -- far inside the 1e-9 relative bound the GPU sums
are held to.  Finalize adds float pairs with Knuth's TwoSum; its rounding error
is exactly recovered.
"""
from fractions import Fraction

import numpy as np
import pytest

U = Fraction(1, 1 << 24)


def r32(q: Fraction) -> Fraction:
    """q rounded to the nearest fp32 value, ties to even (normal range only)."""
    if q == 0:
        return Fraction(0)
    sign = -1 if q < 0 else 1
    a = abs(q)
    e = a.numerator.bit_length() - a.denominator.bit_length()  # 2^e <= a < 2^(e+2)
    if Fraction(2) ** e > a:
        e -= 1
    elif Fraction(2) ** (e + 1) <= a:
        e += 1
    assert -126 <= e <= 127, "outside the normal fp32 range"
    scale = Fraction(2) ** (e - 23)
    m = a / scale  # in [2^23, 2^24)
    lo = m.numerator // m.denominator
    rem = m - lo
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and lo % 2 == 1):
        lo += 1
    return sign * lo * scale


def add(a, b):
    return r32(a + b)


def sub(a, b):
    return r32(a - b)


def fma(a, b, c):
    return r32(a * b + c)


def two_sum_sq(S, C, x):
    t = fma(x, x, S)
    zn = sub(S, t)
    y = add(t, zn)
    a = sub(S, y)
    b = fma(x, x, zn)
    return t, add(C, add(a, b)), (a, b)


def f32(v):
    return Fraction(float(np.float32(v)))


def cases(seed, n, spread):
    rng = np.random.default_rng(seed)
    mags = 2.0 ** rng.uniform(-spread, spread, n)
    return [f32(v) for v in rng.standard_normal(n) * mags]


@pytest.mark.parametrize("seed,spread", [(0, 0), (1, 4), (2, 12), (3, 20)])
def test_each_step_recovers_the_addition_error(seed, spread):
    S, C = Fraction(0), Fraction(0)
    for x in cases(seed, 300, spread):
        t, C_new, (a, b) = two_sum_sq(S, C, x)
        err = S + x * x - t  # the exact rounding error of t
        assert abs(err - (a + b)) <= 3 * U * U * abs(t) + Fraction(1, 1 << 140)
        S, C = t, C_new


@pytest.mark.parametrize("seed,spread,n", [(4, 0, 128), (5, 8, 256), (6, 24, 256), (7, 2, 1024)])
def test_running_pair_carries_the_sum(seed, spread, n):
    xs = cases(seed, n, spread)
    exact = sum(x * x for x in xs)
    S, C = Fraction(0), Fraction(0)
    for x in xs:
        S, C, _ = two_sum_sq(S, C, x)
    rel = abs((S + C) - exact) / exact
    assert rel <= 4 * n * U * U  # about n u^2; a plain fp32 sum is off by up to n u
    # the same squares summed in plain fp32 are not good enough for 1e-9
    plain = Fraction(0)
    for x in xs:
        plain = fma(x, x, plain)
    if n >= 256 and spread <= 8:
        assert abs(plain - exact) / exact > Fraction(1, 10 ** 9)


def test_squares_that_are_not_exact_in_fp32():
    # fp32 inputs whose squares need 48 bits: the FMA residual carries them
    xs = [f32(1 + k * 2.0 ** -23) for k in range(1, 200, 7)]
    S, C = Fraction(0), Fraction(0)
    for x in xs:
        S, C, _ = two_sum_sq(S, C, x)
    exact = sum(x * x for x in xs)
    assert abs((S + C) - exact) / exact <= 4 * len(xs) * U * U


def two_sum(a, b):
    """Knuth's TwoSum in fp32: s = fl(a + b) and the exact error e."""
    s = add(a, b)
    z = sub(s, a)
    e = add(sub(a, sub(s, z)), sub(b, z))
    return s, e


def test_twosum_of_pairs_is_exact():
    rng = np.random.default_rng(8)
    for _ in range(400):
        a, b = (f32(v) for v in rng.standard_normal(2) * 2.0 ** rng.uniform(-30, 30, 2))
        s, e = two_sum(a, b)
        assert s + e == a + b


def test_rounding_helper_matches_numpy_float32():
    rng = np.random.default_rng(9)
    for v in rng.standard_normal(2000) * 2.0 ** rng.uniform(-60, 60, 2000):
        assert r32(Fraction(float(v))) == Fraction(float(np.float32(v)))
