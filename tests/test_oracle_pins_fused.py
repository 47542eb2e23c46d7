"""Pins of the oracle's GELU-fused activation quantization.

The GELU (the exact erf form, by reading: the paper does not name the FFN
activation) is checked against textbook values of the standard normal CDF
(tests/golden/handworked_fused.json), an exact identity, and an erf Taylor
series written here in binary64 (independent of the C library's erfc).  The
fused quantization reduces to the plain per-token quantization where GELU is
the identity in fp32, and obeys the rounding bound everywhere.
"""

import json
import math
import os

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                   "handworked_fused.json")))


def bf16(x):
    t = torch.tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def f32_of_bf16(h):
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def ulp32(x):
    return np.spacing(np.abs(np.float32(x))).astype(np.float64)


def erf_series(z):
    """erf(z) = 2/sqrt(pi) sum_n (-1)^n z^(2n+1) / (n! (2n+1)), |z| <= 3."""
    total, term, n = 0.0, z, 0
    while True:
        add = term / (2 * n + 1)
        total += add
        if abs(add) < 1e-18 * max(1.0, abs(total)):
            break
        n += 1
        term *= -z * z / n
    return 2.0 / math.sqrt(math.pi) * total


def test_gelu_textbook_values(oracle_mod):
    for h, phi in GOLD["phi"].items():
        h = float(h)
        g = oracle_mod.gelu_value([h])[0]
        want = np.float32(h * phi)
        assert abs(float(g) - float(want)) <= ulp32(want) + 1e-30, (h, g, want)


def test_gelu_odd_part_identity(oracle_mod):
    # GELU(h) - GELU(-h) = h exactly (erfc(-z) + erfc(z) = 2)
    h = wl.random_uniform_f32((2000,), seed=1, lo=-8.0, hi=8.0)
    gp, gm = oracle_mod.gelu_value(h), oracle_mod.gelu_value(-h)
    err = np.abs(gp.astype(np.float64) - gm - h)
    assert np.all(err <= ulp32(gp) + ulp32(gm) + ulp32(h))


def test_gelu_against_erf_series(oracle_mod):
    h = np.linspace(-4.0, 4.0, 801).astype(np.float32)
    g = oracle_mod.gelu_value(h)
    for hv, gv in zip(h, g):
        want = 0.5 * float(hv) * (1.0 + erf_series(float(hv) / math.sqrt(2.0)))
        # the oracle rounds the binary64 value once: within half an ulp, plus
        # the series' own error (cancellation at most ~1e-13 relative)
        assert abs(float(gv) - want) <= 0.5 * ulp32(want) + 1e-12 * abs(want) + 1e-45


def test_gelu_detects_sign_mistake(oracle_mod):
    # a planted mistake (erfc(+h/sqrt 2): GELU(h) becomes h * (1 - Phi(h)))
    # misses the golden value by far
    phi1 = GOLD["phi"]["1.0"]
    planted = 0.5 * 1.0 * math.erfc(1.0 / math.sqrt(2.0))
    assert abs(planted - phi1) > 0.5
    assert abs(float(oracle_mod.gelu_value([1.0])[0]) - phi1) < 1e-7


def test_gelu_quant_is_quant_where_gelu_is_identity(oracle_mod):
    # for h >= 6, erfc(-h/sqrt 2) = 2 - erfc(h/sqrt 2) rounds GELU(h) to h in fp32
    rng = np.random.default_rng(2)
    H = bf16(rng.uniform(6.0, 100.0, size=(9, 96)).astype(np.float32))
    lam = wl.random_uniform_f32((96,), seed=3, lo=0.5, hi=2.0)
    q1, s1 = oracle_mod.gelu_quant_act(H, lam)
    q2, s2 = oracle_mod.quant_act(H, lam)
    np.testing.assert_array_equal(q1, q2)
    np.testing.assert_array_equal(s1, s2)


def test_gelu_quant_invariants(oracle_mod):
    H = wl.random_bf16((17, 200), seed=4, scale=2.0)
    lam = wl.random_uniform_f32((200,), seed=5, lo=0.5, hi=2.0)
    q, sx, pre = oracle_mod.gelu_quant_act(H, lam, with_pre=True)
    h = f32_of_bf16(H).astype(np.float64)
    g = 0.5 * h * np.array([math.erfc(-v / math.sqrt(2.0)) for v in h.ravel()]).reshape(h.shape)
    xs = g / lam.astype(np.float64)
    for r in range(H.shape[0]):
        a = np.abs(xs[r]).max()
        assert abs(sx[r] * 127 - a) <= 1e-6 * a
        assert abs(int(q[r, np.argmax(np.abs(xs[r]))])) == 127
        err = np.abs(q[r].astype(np.float64) * sx[r] - xs[r])
        assert err.max() <= 0.5 * sx[r] * (1 + 1e-5) + 1e-6 * a
    # the codes are the rounded pre-values
    np.testing.assert_array_equal(q, np.clip(np.rint(pre), -127, 127).astype(np.int8))


def test_quant_act_dual_is_per_branch(oracle_mod):
    b = [(wl.random_bf16((5, 64), seed=6), wl.random_uniform_f32((64,), seed=7, lo=0.5, hi=2.0)),
         (wl.random_bf16((3, 64), seed=8), None)]
    out = oracle_mod.quant_act_dual(b)
    for (X, lam), (q, s) in zip(b, out):
        q2, s2 = oracle_mod.quant_act(X, lam)
        np.testing.assert_array_equal(q, q2)
        np.testing.assert_array_equal(s, s2)
