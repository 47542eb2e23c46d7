"""Pins of the oracle's ablation and protection functions.

The per-tensor activation quantization (naive arm of the activation-quant
ablation, Sec. 5 "What drives INT8 recovery"), the activation statistics and
the protected bf16 layer (Sec. 3, "Activation-fragility profiling and
protection") are checked against hand-worked values
(tests/golden/handworked_protect.json), exact rational arithmetic, library
routines that the oracle does not use (numpy, scipy.stats) and invariants that
hold in exact arithmetic.  ``test_*_detects_*`` plant mistakes on the CPU to
show that the checks discriminate.
"""

import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                   "handworked_protect.json")))


def bf16(x):
    t = torch.tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def f32_of_bf16(h):
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# ------------------------------------------------- per-tensor activation scale

@pytest.mark.parametrize("key", ["per_tensor_no_smoothing", "per_tensor_smoothed"])
def test_per_tensor_golden(oracle_mod, key):
    g = GOLD[key]
    lam = None if g["lambda"] is None else np.array(g["lambda"], np.float32)
    Xq, sx, amax = oracle_mod.quant_act_per_tensor(bf16(g["X"]), lam)
    np.testing.assert_array_equal(Xq, np.array(g["Xq"], np.int8))
    assert amax == g["amax"]
    # the scale is amax / 127 rounded once to fp32, on every row
    assert np.all(sx == np.float32(Fraction(g["scale_numerator"]) / 127))


def test_per_tensor_single_row_is_per_token(oracle_mod):
    # with one token the tensor is the row: both granularities coincide
    X = wl.random_bf16((1, 784), seed=5, scale=3.0)
    lam = wl.random_uniform_f32((784,), seed=6, lo=0.25, hi=4.0)
    q1, s1, _ = oracle_mod.quant_act_per_tensor(X, lam)
    q2, s2 = oracle_mod.quant_act(X, lam)
    np.testing.assert_array_equal(q1, q2)
    np.testing.assert_array_equal(s1, s2)


def test_per_tensor_invariants(oracle_mod):
    X = wl.random_bf16((37, 96), seed=7, scale=2.0)
    lam = wl.random_uniform_f32((96,), seed=8, lo=0.5, hi=2.0)
    Xq, sx, amax = oracle_mod.quant_act_per_tensor(X, lam)
    xs = (f32_of_bf16(X).astype(np.float64) / lam.astype(np.float64))
    # the largest smoothed magnitude maps to +-127, and nothing exceeds it
    i = np.unravel_index(np.argmax(np.abs(xs)), xs.shape)
    assert abs(int(Xq[i])) == 127
    assert np.all(np.abs(Xq.astype(np.int32)) <= 127)
    assert abs(amax - np.abs(xs).max()) <= 1e-6 * amax
    # dequantization error within half a step (plus fp32 rounding of x' and inv)
    s = float(sx[0])
    err = np.abs(Xq.astype(np.float64) * s - xs)
    assert err.max() <= 0.5 * s * (1 + 1e-5) + 1e-6 * amax
    # a single scale: every row carries the same one
    assert np.all(sx == sx[0])
    # rows whose own max is the tensor max quantize exactly as per-token
    qt, st = oracle_mod.quant_act(X, lam)
    for r in range(X.shape[0]):
        if st[r] == sx[0]:
            np.testing.assert_array_equal(qt[r], Xq[r])


def test_per_tensor_power_of_two_invariance(oracle_mod):
    X = wl.random_bf16((9, 64), seed=9)
    Xq, sx, amax = oracle_mod.quant_act_per_tensor(X, None)
    X4 = bf16(f32_of_bf16(X) * 4.0)           # exact: a power of two
    Xq4, sx4, amax4 = oracle_mod.quant_act_per_tensor(X4, None)
    np.testing.assert_array_equal(Xq, Xq4)
    assert amax4 == 4 * amax and np.all(sx4 == 4 * sx)


def test_per_tensor_zero_and_one_outlier(oracle_mod):
    X = np.zeros((3, 32), np.uint16)
    Xq, sx, amax = oracle_mod.quant_act_per_tensor(X, None)
    assert amax == 0 and not Xq.any() and not sx.any()
    # one outlier 1000x the rest squeezes every other code towards 0: the
    # collapse of naive per-tensor INT8 that the paper describes
    v = np.full((4, 32), 1.0, np.float32)
    v[2, 5] = 1024.0
    Xq, sx, _ = oracle_mod.quant_act_per_tensor(bf16(v), None)
    assert Xq[2, 5] == 127 and np.count_nonzero(Xq) == 1


# ------------------------------------------------------- activation statistics

def test_act_stats_golden(oracle_mod):
    g = GOLD["act_stats"]
    chan, tensor = oracle_mod.act_stats(bf16(g["X"]))
    np.testing.assert_array_equal(chan[0], g["chan_maxabs"])
    np.testing.assert_array_equal(chan[1], g["chan_mean"])
    np.testing.assert_allclose(chan[2], np.sqrt(g["chan_var"]), rtol=1e-15)
    np.testing.assert_allclose(chan[3], np.array(g["chan_kurt_num"]) / np.array(g["chan_kurt_den"]),
                               rtol=1e-15)
    t = g["tensor"]
    assert tensor[0] == t["maxabs"] and tensor[1] == t["mean"]
    assert tensor[2] == pytest.approx(np.sqrt(t["var"]), rel=1e-15)
    assert tensor[3] == pytest.approx(t["kurt"], rel=1e-15)


def test_shifted_sums_golden(oracle_mod):
    g = GOLD["act_stats"]
    S, A = oracle_mod.shifted_power_sums(bf16(g["X"]), np.array(g["shift"], np.float32))
    np.testing.assert_array_equal(S, np.array(g["shifted_sums"]))
    np.testing.assert_array_equal(A[1], S[1])          # even powers are their own size
    np.testing.assert_array_equal(A[3], S[3])


def test_act_stats_match_scipy(oracle_mod):
    scipy_stats = pytest.importorskip("scipy.stats")
    X = wl.random_bf16((301, 40), seed=11, scale=1.5)
    x = f32_of_bf16(X).astype(np.float64)
    x[:, 3] += 7.0                                  # a channel with a large mean
    x[:, 4] *= 0.0                                  # a constant channel
    X = bf16(x)
    x = f32_of_bf16(X).astype(np.float64)
    chan, tensor = oracle_mod.act_stats(X)
    np.testing.assert_allclose(chan[0], np.abs(x).max(axis=0), rtol=0)
    np.testing.assert_allclose(chan[1], x.mean(axis=0), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(chan[2], x.std(axis=0), rtol=1e-12, atol=1e-15)
    k = scipy_stats.kurtosis(x, axis=0, fisher=False, bias=True)
    nz = chan[2] > 0
    np.testing.assert_allclose(chan[3][nz], k[nz], rtol=1e-11)
    assert chan[3][4] == 0.0
    assert tensor[2] == pytest.approx(x.std(), rel=1e-12)
    assert tensor[3] == pytest.approx(scipy_stats.kurtosis(x.ravel(), fisher=False), rel=1e-11)


def test_act_stats_normal_and_student_t_kurtosis(oracle_mod):
    # large samples: Pearson kurtosis of a normal is 3; a Student-t with 5
    # degrees of freedom has 3 + 6/(5-4) = 9 (heavy tails raise it)
    rng = np.random.default_rng(3)
    z = rng.standard_normal((200000, 1)).astype(np.float32)
    t5 = rng.standard_t(5, size=(200000, 1)).astype(np.float32)
    chan, _ = oracle_mod.act_stats(bf16(np.concatenate([z, t5], axis=1)))
    assert abs(chan[3][0] - 3.0) < 0.1
    assert 6.0 < chan[3][1] < 12.0
    assert abs(chan[2][0] - 1.0) < 0.01


def test_shifted_sums_binomial_invariance(oracle_mod):
    # sums about two shifts are tied by the binomial theorem, and about shift 0
    # they are numpy's power sums
    X = wl.random_bf16((123, 24), seed=13, scale=2.0)
    x = f32_of_bf16(X).astype(np.float64)
    c = wl.random_uniform_f32((24,), seed=14, lo=-1.0, hi=1.0)
    S0, _ = oracle_mod.shifted_power_sums(X, None)
    Sc, _ = oracle_mod.shifted_power_sums(X, c)
    for p in range(1, 5):
        np.testing.assert_allclose(S0[p - 1], (x ** p).sum(axis=0), rtol=1e-12, atol=1e-9)
    T = X.shape[0]
    cd = c.astype(np.float64)
    P = [np.full(24, float(T))] + [S0[p] for p in range(4)]      # P[q] = sum x^q
    for p in range(1, 5):
        want = sum(math.comb(p, q) * (-cd) ** (p - q) * P[q] for q in range(p + 1))
        np.testing.assert_allclose(Sc[p - 1], want, rtol=1e-9, atol=1e-8)


def test_stats_detects_wrong_variance_divisor(oracle_mod):
    # a planted mistake (sample variance, divide by T-1) is caught by the golden
    g = GOLD["act_stats"]
    x = np.array(g["X"], np.float64)
    planted = x.var(axis=0, ddof=1)
    assert not np.allclose(planted, g["chan_var"])


# -------------------------------------------------------- protected bf16 layer

def test_linear_bf16_golden(oracle_mod):
    g = GOLD["linear_bf16"]
    Y, Ya = oracle_mod.linear_bf16(bf16(g["X"]), bf16(g["W"]), np.array(g["bias"], np.float32))
    np.testing.assert_array_equal(Y, np.array(g["Y"]))
    assert np.all(Ya >= np.abs(Y))


@pytest.mark.parametrize("M,N,K", [(1, 1, 1), (3, 5, 7), (4, 3, 33)])
def test_linear_bf16_exact_rationals(oracle_mod, M, N, K):
    X = wl.random_bf16((M, K), seed=M + K, scale=2.0)
    W = wl.random_bf16((N, K), seed=N + 2 * K, scale=0.5)
    b = wl.random_uniform_f32((N,), seed=K, lo=-1.0, hi=1.0)
    Y, _ = oracle_mod.linear_bf16(X, W, b)
    xf, wf = f32_of_bf16(X), f32_of_bf16(W)
    for m in range(M):
        for n in range(N):
            exact = sum(Fraction(float(xf[m, k])) * Fraction(float(wf[n, k])) for k in range(K))
            exact += Fraction(float(b[n]))
            assert abs(Fraction(Y[m, n]) - exact) <= Fraction(1, 2 ** 50) * (abs(exact) + 1)


def test_linear_bf16_numpy_and_rows(oracle_mod):
    X = wl.random_bf16((37, 200), seed=21)
    W = wl.random_bf16((19, 200), seed=22, scale=0.05)
    want = f32_of_bf16(X).astype(np.float64) @ f32_of_bf16(W).astype(np.float64).T
    Y, _ = oracle_mod.linear_bf16(X, W, None)
    np.testing.assert_allclose(Y, want, rtol=1e-13, atol=1e-13)
    Yr, _ = oracle_mod.linear_bf16(X, W, None, rows=(4, 9))
    np.testing.assert_array_equal(Yr, Y[4:9])


def test_linear_bf16_identity_and_bias(oracle_mod):
    K = 16
    X = wl.random_bf16((5, K), seed=23)
    eye = bf16(np.eye(K, dtype=np.float32))
    Y, _ = oracle_mod.linear_bf16(X, eye, None)
    np.testing.assert_array_equal(Y, f32_of_bf16(X).astype(np.float64))
    b = wl.random_f32((K,), seed=24)
    Y0, _ = oracle_mod.linear_bf16(np.zeros((2, K), np.uint16), eye, b)
    np.testing.assert_array_equal(Y0, np.tile(b.astype(np.float64), (2, 1)))


def test_layer_dispatch(oracle_mod):
    case = wl.workload_cases("single_m256_k512_n512")[0]
    X = case.X[0][:8]
    W = case.W[0]
    lam = oracle_mod.smooth_scales(oracle_mod.channel_absmax(case.X_cal), W, 0.5)
    Wq, sw = oracle_mod.quantize_weights(W, lam)
    layer = {"protect": False, "smooth": lam, "Wq": Wq, "w_scale": sw,
             "W_bf16": bf16(W), "bias": case.bias[0]}
    Yq = oracle_mod.layer_forward(X, layer)
    Xq, sx = oracle_mod.quant_act(X, lam)
    np.testing.assert_array_equal(Yq, oracle_mod.linear(Xq, sx, Wq, sw, case.bias[0]))
    layer["protect"] = True
    Yp, _ = oracle_mod.layer_forward(X, layer)
    want, _ = oracle_mod.linear_bf16(X, bf16(W), case.bias[0])
    np.testing.assert_array_equal(Yp, want)
    # the protected result is the closer one to the exact fp64 product
    exact = f32_of_bf16(X).astype(np.float64) @ W.astype(np.float64).T + case.bias[0]
    assert np.abs(Yp - exact).mean() < np.abs(f32_of_bf16(Yq) - exact).mean()
