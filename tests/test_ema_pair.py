"""The fp32 row EMA of the state pass's row pass, checked on the CPU with
exact rational arithmetic.

The kernel forms beta2 r + (1 - beta2) m as
    fmaf(bh, r, fmaf(bl, r, fmaf(ah, m, al * m)))
with bh + bl = beta2 and ah + al = 1 - beta2 (hi the coefficient rounded to
fp32, lo the rest rounded to fp32).  Here each fmaf is emulated exactly
(product and sum in rationals, one rounding to fp32) and the result is held
to the bar the parity tests use for the state: within 1 fp32 ulp of the
value rounded from exact arithmetic (what the fp64 oracle stores), the fixed
point r = m reproduced exactly, and rows with m = 0 decaying to the
correctly rounded beta2 r.
"""
from fractions import Fraction

import numpy as np
import pytest


def f32(x):
    """Exact rational -> nearest fp32, ties to even: the fp64 rounding gives
    a candidate, and its two fp32 neighbours settle any double rounding."""
    x = Fraction(x)
    c = np.float32(float(x))
    best = None
    for y in (np.nextafter(c, np.float32(-np.inf)), c, np.nextafter(c, np.float32(np.inf))):
        d = abs(Fraction(float(y)) - x)
        even = int(y.view(np.int32)) % 2 == 0
        if best is None or d < best[0] or (d == best[0] and even):
            best = (d, y)
    return best[1]


def fmaf(a, b, c):
    return f32(Fraction(float(a)) * Fraction(float(b)) + Fraction(float(c)))


def pair(beta2):
    bh = np.float32(beta2)
    bl = np.float32(beta2 - float(bh))
    ah = np.float32(1.0 - beta2)
    al = np.float32((1.0 - beta2) - float(ah))
    return bh, bl, ah, al


def ema_pair(c, r, m):
    bh, bl, ah, al = c
    return fmaf(bh, r, fmaf(bl, r, fmaf(ah, m, f32(Fraction(float(al)) * Fraction(float(m))))))


def ulps(a, b):
    return abs(int(np.float32(a).view(np.int32)) - int(np.float32(b).view(np.int32)))


@pytest.mark.parametrize("beta2", [0.999, 0.9, 0.5, 0.0, 0.99999])
def test_within_one_ulp_of_the_exact_value(beta2):
    rng = np.random.default_rng(int(beta2 * 1e5))
    c = pair(beta2)
    for k in range(400):
        r = np.float32(10 ** rng.uniform(-12, 0))
        m = np.float32(10 ** rng.uniform(-12, 0)) if k % 3 else np.float32(0)
        want = f32(Fraction(beta2) * Fraction(float(r)) + (1 - Fraction(beta2)) * Fraction(float(m)))
        assert ulps(ema_pair(c, r, m), want) <= 1, (beta2, r, m)


@pytest.mark.parametrize("beta2", [0.999, 0.9, 0.99999])
def test_fixed_point_is_exact(beta2):
    c = pair(beta2)
    for x in [1.0, 3.3e-7, 0.123, 7.7e-12, 2.5e-3]:
        x = np.float32(x)
        assert ema_pair(c, x, x) == x


def test_single_float_coefficients_would_drift():
    """Why the pairs: with beta2 and 1 - beta2 rounded to single floats the
    fixed point of r <- b r + a m moves to a m / (1 - b), 1.3e-5 above m at
    beta2 = 0.999, beyond the 1e-5 state bar over a long run."""
    b, a = np.float32(0.999), np.float32(1 - 0.999)
    drift = float(Fraction(float(a)) / (1 - Fraction(float(b)))) - 1.0
    assert drift > 1e-5
