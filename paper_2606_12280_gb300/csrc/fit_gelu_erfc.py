"""Fit of the Phi approximation behind the GELU in quant.cu.

GELU(h) = h * Phi(h), Phi(h) = erfc(-h / sqrt 2) / 2.  For a = |h| <= 8,

    log2 erfc(a / sqrt 2) ~= P(u),   u = a/4 - 1  (exact in fp32: a power-of-2 scale),

P a degree-12 polynomial (power basis in u, Horner in fp32), fitted by least
squares in the Chebyshev basis at 6000 Chebyshev nodes of [0, 8] to
log2 erfc(a / sqrt 2) (scipy, binary64), then converted to the power basis.
Then Phi(h) = 1 - 2^P / 2 for h >= 0 and 2^P / 2 for h < 0: one ex2, no
division, and no rounding of a scaled argument (the error that grows with a
when erfc is evaluated at a rounded a / sqrt 2).  Beyond |h| = 8, erfc < 1.3e-15
and Phi is taken as 0 or 1.  The coefficients are this fit's own.  Run it to
reproduce the constants and the maximum relative error of erfc(a / sqrt 2)
over every fp32 a in a dense grid, in binary64 and in fp32 Horner.

A second, shorter fit serves warps whose values all have |h| < 4: degree 8
in v = a/2 - 1 (again exact in fp32) over [0, 4], fitted the same way.  In
fp32 Horner its relative error is about 1e-6 there, no worse than the long
fit's on the same range, at 8 instead of 12 multiply-adds.
"""

import math

import numpy as np
from scipy.special import erfc

H1 = 8.0
DEG = 12


H_SHORT = 4.0
DEG_SHORT = 8


def fit(h1=H1, deg=DEG):
    k = np.arange(6000)
    a = 0.5 * h1 + 0.5 * h1 * np.cos(np.pi * (k + 0.5) / k.size)
    c = np.polynomial.chebyshev.chebfit(a / h1 * 2 - 1, np.log2(erfc(a / math.sqrt(2))), deg)
    return np.polynomial.chebyshev.cheb2poly(c)


def max_rel_error(c, fp32, amax=H1, h1=H1):
    f = np.float32
    a = np.linspace(0.0, amax, 800001).astype(f)
    u = (a * f(2 / h1) - f(1)).astype(f)
    if not fp32:
        p = np.polynomial.polynomial.polyval(u.astype(np.float64), c)
    else:
        cf = c.astype(f)
        p = np.full_like(u, cf[-1])
        for cc in cf[-2::-1]:          # fused multiply-add: one rounding per step
            p = (p.astype(np.float64) * u.astype(np.float64) + float(cc)).astype(f)
        p = p.astype(np.float64)
    return float(np.max(np.abs(np.exp2(p) / erfc(a.astype(np.float64) / math.sqrt(2)) - 1)))


if __name__ == "__main__":
    c = fit()
    for i, v in enumerate(c):
        print(f"C{i} = {float(np.float32(v)):.9g}f")
    print("max relative error of erfc, binary64 fit, a <= 8:", max_rel_error(c, False))
    print("max relative error of erfc, fp32 Horner,  a <= 6:", max_rel_error(c, True, 6.0))
    print("max relative error of erfc, fp32 Horner,  a <= 8:", max_rel_error(c, True))
    print("max relative error of erfc, fp32 Horner,  a <= 4:", max_rel_error(c, True, 4.0))
    cs = fit(H_SHORT, DEG_SHORT)
    for i, v in enumerate(cs):
        print(f"S{i} = {float(np.float32(v)):.9g}f")
    print("short fit, max relative error of erfc, binary64, a <= 4:", max_rel_error(cs, False, 4.0, H_SHORT))
    print("short fit, max relative error of erfc, fp32 Horner, a <= 4:", max_rel_error(cs, True, 4.0, H_SHORT))
