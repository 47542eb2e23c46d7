"""The GELU fits in quant.cu are the ones fit_gelu_erfc.py computes.

The fused GELU + quantization pass evaluates log2 erfc(|h|/sqrt 2) with two
least-squares polynomials (degree 12 over [0, 8], degree 8 over [0, 4]).
This host test refits both with the script beside the kernel source and
checks that every coefficient written in quant.cu is the fit's coefficient
rounded to fp32 (the constant terms lowered by exactly 1, which halves
erfc), and that the fits meet the accuracy the kernel's comments state.
"""

import importlib.util
import os
import re

import numpy as np
import pytest

pytest.importorskip("scipy")

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                    "paper_2606_12280_gb300", "csrc")


def load_fit():
    spec = importlib.util.spec_from_file_location("fit_gelu_erfc", os.path.join(CSRC, "fit_gelu_erfc.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def kernel_coefficients(function):
    """The splat(...) constants of one GELU function in quant.cu, in source
    order (highest degree first, the Horner order)."""
    src = open(os.path.join(CSRC, "quant.cu")).read()
    start = src.index(function + "(float2 h)")
    end = src.index("return gelu_tail", start)
    vals = [float(v.rstrip("f")) for v in re.findall(r"splat\((-?[0-9.]+(?:e-?[0-9]+)?f)\)", src[start:end])]
    return vals


@pytest.mark.parametrize("function,h1,deg,skip", [("gelu_erf2_long", 8.0, 12, 2), ("gelu_erf2_short", 4.0, 8, 2)])
def test_kernel_constants_are_the_fit(function, h1, deg, skip):
    fit = load_fit()
    c = fit.fit(h1, deg)
    vals = kernel_coefficients(function)
    # the first `skip` constants are the argument map (|h| scale and -1)
    horner = vals[skip:]
    assert len(horner) == deg + 1
    want = [np.float32(v) for v in c[::-1]]
    want[-1] = np.float32(np.float32(c[0]) - np.float32(1.0))   # constant term lowered by 1
    assert np.array_equal(np.array(horner, np.float32), np.array(want, np.float32))


def test_fit_accuracy():
    fit = load_fit()
    long_fit = fit.fit(fit.H1, fit.DEG)
    short_fit = fit.fit(fit.H_SHORT, fit.DEG_SHORT)
    assert fit.max_rel_error(long_fit, True, 6.0) < 2e-6
    assert fit.max_rel_error(long_fit, True, 8.0) < 4e-6
    assert fit.max_rel_error(short_fit, True, 4.0, fit.H_SHORT) < 1.2e-6
    # on the short range the short fit is no worse than the long one
    assert fit.max_rel_error(short_fit, True, 4.0, fit.H_SHORT) <= fit.max_rel_error(long_fit, True, 4.0)
