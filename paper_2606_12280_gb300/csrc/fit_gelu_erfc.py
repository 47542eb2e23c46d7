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
"""

import math

import numpy as np
from scipy.special import erfc

H1 = 8.0
DEG = 12


def fit():
    k = np.arange(6000)
    a = 0.5 * H1 + 0.5 * H1 * np.cos(np.pi * (k + 0.5) / k.size)
    c = np.polynomial.chebyshev.chebfit(a / H1 * 2 - 1, np.log2(erfc(a / math.sqrt(2))), DEG)
    return np.polynomial.chebyshev.cheb2poly(c)


def max_rel_error(c, fp32, amax=H1):
    f = np.float32
    a = np.linspace(0.0, amax, 800001).astype(f)
    u = (a * f(2 / H1) - f(1)).astype(f)
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
