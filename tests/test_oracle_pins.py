"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these checks re-types the oracle's own formulas: each one compares the
oracle with a hand-worked value (tests/golden/handworked.json), a brute-force
or library computation (Python integers, numpy int64 matmul, numpy rint,
torch's bf16 cast), an invariant that holds in exact arithmetic (SmoothQuant
balance, the smoothing identity) or a derived error bound.  A planted mistake
(a dropped term, a wrong sign or index, a transposed operand, the wrong
smoothing direction) fails at least one of them; ``test_bound_detects_*``
plants such mistakes on the CPU to show the bounds discriminate.
"""

import json
import os

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                   "handworked.json")))


def bf16(x):
    """float values (exactly representable) -> bf16 bit patterns via torch."""
    t = torch.tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def f32_of_bf16(h):
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# ---------------------------------------------------------------- gemm (a4)

@pytest.mark.parametrize("M,N,K", [(1, 1, 16), (7, 5, 32), (13, 9, 48), (3, 17, 64)])
def test_gemm_brute_force_python_ints(oracle_mod, M, N, K):
    Xq = wl.random_int8((M, K), seed=M * 100 + K)
    Wq = wl.random_int8((N, K), seed=N * 100 + K + 1)
    acc = oracle_mod.gemm_i32(Xq, Wq)
    for m in range(M):
        for n in range(N):
            want = sum(int(Xq[m, k]) * int(Wq[n, k]) for k in range(K))
            assert acc[m, n] == want


def test_gemm_numpy_int64(oracle_mod):
    Xq = wl.random_int8((129, 528), seed=1)
    Wq = wl.random_int8((70, 528), seed=2)
    want = Xq.astype(np.int64) @ Wq.astype(np.int64).T
    np.testing.assert_array_equal(oracle_mod.gemm_i32(Xq, Wq), want)
    # row subsets give the same rows
    np.testing.assert_array_equal(oracle_mod.gemm_i32(Xq, Wq, rows=(5, 17)), want[5:17])


def test_gemm_not_transposed(oracle_mod):
    # a non-square case where X Wq (no transpose) is not even defined the same way
    Xq = wl.random_int8((3, 32), seed=3)
    Wq = wl.random_int8((5, 32), seed=4)
    acc = oracle_mod.gemm_i32(Xq, Wq)
    assert acc.shape == (3, 5)
    assert acc[2, 4] == int(np.dot(Xq[2].astype(np.int64), Wq[4].astype(np.int64)))


def test_gemm_int32_bound(oracle_mod):
    g = GOLD["int32_bound"]
    K = g["K"]
    Xq = np.full((2, K), 127, dtype=np.int8)
    Xq[1] = -127
    Wq = np.full((1, K), 127, dtype=np.int8)
    acc = oracle_mod.gemm_i32(Xq, Wq)
    assert acc[0, 0] == g["acc_all_plus"]
    assert acc[1, 0] == g["acc_plus_minus"]


# ------------------------------------------------------------ bf16 rounding

def test_bf16_rne_handworked(oracle_mod):
    for fbits, hbits in GOLD["bf16_rne_values"]["pairs_f32bits_to_bf16bits"]:
        f = np.array([fbits], dtype=np.uint32).view(np.float32)
        assert int(oracle_mod.f32_to_bf16_rne(f)[0]) == hbits, hex(fbits)


def test_bf16_rne_matches_torch_cast(oracle_mod):
    g = torch.Generator().manual_seed(7)
    x = torch.randn(4000, generator=g) * 100
    # add exact midpoints: values with the low 16 bits == 0x8000
    mid = (torch.randint(0, 2**15, (1000,), generator=g, dtype=torch.int32) << 16) | 0x8000
    x = torch.cat([x, mid.view(torch.float32)])
    x = x[torch.isfinite(x)]
    want = x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle_mod.f32_to_bf16_rne(x.numpy())
    np.testing.assert_array_equal(got, want)


def test_quantize_value_matches_numpy_rint(oracle_mod):
    g = torch.Generator().manual_seed(8)
    v = (torch.rand(3000, generator=g) * 300 - 150).numpy().astype(np.float32)
    halves = (np.arange(-140, 140) + 0.5).astype(np.float32)
    v = np.concatenate([v, halves])
    want = np.clip(np.rint(v.astype(np.float64)), -127, 127).astype(np.int8)
    got = np.array([oracle_mod.quantize_value(float(t)) for t in v], dtype=np.int8)
    np.testing.assert_array_equal(got, want)
    assert oracle_mod.quantize_value(float("nan")) == 0
    assert oracle_mod.quantize_value(float("inf")) == 127
    assert oracle_mod.quantize_value(float("-inf")) == -127


# ------------------------------------------------- scales and quantization

def test_round_half_even_handworked(oracle_mod):
    g = GOLD["round_half_even_row"]
    Xq, sx = oracle_mod.quant_act(bf16(g["X"]), None)
    np.testing.assert_array_equal(Xq, np.array(g["Xq"], dtype=np.int8))
    assert sx[0] == np.float32(g["sx"][0])


def test_smoothed_act_handworked(oracle_mod):
    g = GOLD["smoothed_act_row"]
    Xq, sx = oracle_mod.quant_act(bf16(g["X"]), np.array(g["lambda"], np.float32))
    np.testing.assert_array_equal(Xq, np.array(g["Xq"], dtype=np.int8))
    num, den = g["sx_num_den"]
    assert sx[0] == np.float32(num / den)


def test_smooth_handworked(oracle_mod):
    g = GOLD["smooth_alpha_half"]
    lam = oracle_mod.smooth_scales(np.array(g["s"], np.float32),
                                   np.array(g["W"], np.float32), g["alpha"])
    np.testing.assert_array_equal(lam, np.array(g["lambda"], np.float32))


def test_quantize_weights_handworked(oracle_mod):
    g = GOLD["quantize_weights_row"]
    Wq, sw = oracle_mod.quantize_weights(np.array(g["W"], np.float32),
                                         np.array(g["lambda"], np.float32))
    np.testing.assert_array_equal(Wq, np.array(g["Wq"], np.int8))
    num, den = g["sw_num_den"]
    assert sw[0] == np.float32(num / den)


def test_epilogue_handworked(oracle_mod):
    g = GOLD["epilogue_value"]
    Y = oracle_mod.epilogue(np.array([[g["acc"]]], np.int32), np.array([g["sx"]], np.float32),
                            np.array([g["sw"]], np.float32), np.array([g["bias"]], np.float32))
    assert int(Y[0, 0]) == g["y_bits"]


def _check_quant_rows(xs, q, scale):
    """xs: fp32 smoothed values [R, K]; q: int8 codes; scale: fp32 [R]."""
    xs64 = xs.astype(np.float64)
    a = np.abs(xs64).max(axis=1)
    nz = a > 0
    # the closed form: scale = absmax / 127, rounded once to fp32
    np.testing.assert_array_equal(scale[nz], (a[nz] / 127.0).astype(np.float32))
    assert np.all(scale[~nz] == 0) and np.all(q[~nz] == 0)
    assert q.min() >= -127 and q.max() <= 127
    # the absmax element of every row maps to +-127 exactly
    idx = np.abs(xs64).argmax(axis=1)
    rows = np.nonzero(nz)[0]
    np.testing.assert_array_equal(np.abs(q[rows, idx[rows]]), 127)
    # round-to-nearest error bound: |x' - q*scale| <= scale/2 (1 + 2^-13)
    err = np.abs(xs64 - q.astype(np.float64) * scale.astype(np.float64)[:, None])
    bound = scale.astype(np.float64)[:, None] / 2 * (1 + 2.0 ** -13)
    assert np.all(err <= bound)


def test_quant_act_error_bound_and_scale(oracle_mod):
    c = wl.make_case(67, 528, 40, seed=11, outlier_frac=0.02)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], 0.5)
    X = c.X[0].copy()
    X[3] = 0                                   # an all-zero token
    Xq, sx = oracle_mod.quant_act(X, lam)
    r = (np.float32(1.0) / lam).astype(np.float32)   # numpy fp32 division, RN
    xs = (f32_of_bf16(X) * r[None, :]).astype(np.float32)
    _check_quant_rows(xs, Xq, sx)


def test_quant_weights_error_bound_and_scale(oracle_mod):
    W = wl.random_f32((33, 272), seed=12, scale=0.02)
    lam = np.abs(wl.random_f32((272,), seed=13)).astype(np.float32) + np.float32(0.25)
    W[5] = 0                                   # an all-zero output channel
    Wq, sw = oracle_mod.quantize_weights(W, lam)
    ws = (W * lam[None, :]).astype(np.float32)
    _check_quant_rows(ws, Wq, sw)
    Wq1, sw1 = oracle_mod.quantize_weights(W, None)
    _check_quant_rows(W, Wq1, sw1)


def test_channel_absmax_matches_numpy(oracle_mod):
    X = wl.random_bf16((50, 96), seed=14, scale=3.0)
    want = np.abs(f32_of_bf16(X)).max(axis=0)
    np.testing.assert_array_equal(oracle_mod.channel_absmax(X), want)


# ----------------------------------------------------------- smoothing (a1)

def test_smoothquant_balance_alpha_half(oracle_mod):
    """alpha = 1/2 balances the two maxima: after smoothing, the calibration
    column max and the weight column max both equal sqrt(s_j m_j)."""
    c = wl.make_case(8, 256, 96, seed=15, outlier_frac=0.03, outlier_mult=30.0)
    s = oracle_mod.channel_absmax(c.X_cal)
    W = c.W[0]
    lam = oracle_mod.smooth_scales(s, W, 0.5).astype(np.float64)
    m = np.abs(W.astype(np.float64)).max(axis=0)        # over output rows i
    act_max = np.abs(f32_of_bf16(c.X_cal).astype(np.float64)).max(axis=0) / lam
    w_max = m * lam
    geo = np.sqrt(s.astype(np.float64) * m)
    np.testing.assert_allclose(act_max, geo, rtol=4e-7)
    np.testing.assert_allclose(w_max, geo, rtol=4e-7)


def test_smooth_alpha_one_and_zero(oracle_mod):
    c = wl.make_case(4, 128, 64, seed=16)
    s = oracle_mod.channel_absmax(c.X_cal)
    W = c.W[0]
    lam1 = oracle_mod.smooth_scales(s, W, 1.0)          # lambda = s
    np.testing.assert_array_equal(lam1, s)
    lam0 = oracle_mod.smooth_scales(s, W, 0.0)          # lambda = 1/m
    m = np.abs(W).max(axis=0)
    np.testing.assert_array_equal(lam0, (np.float32(1) / m).astype(np.float32))
    # alpha = 0 puts every weight column max at 1 (up to one rounding)
    np.testing.assert_allclose(np.abs(W * lam0).max(axis=0), 1.0, rtol=2 ** -23)


def test_smooth_general_alpha_within_one_ulp(oracle_mod):
    c = wl.make_case(4, 256, 64, seed=17)
    s = oracle_mod.channel_absmax(c.X_cal)
    W = c.W[0]
    for alpha in (0.25, 0.65, 0.8):
        lam = oracle_mod.smooth_scales(s, W, alpha)
        a = float(np.float32(alpha))          # alpha crosses the ABI as fp32
        m = np.abs(W.astype(np.float64)).max(axis=0)
        want = s.astype(np.float64) ** a / m ** (1 - a)
        ulp = np.spacing(want.astype(np.float32)).astype(np.float64)
        assert np.all(np.abs(lam.astype(np.float64) - want) <= ulp)


def test_smooth_degenerate(oracle_mod):
    s = np.array([0.0, 2.0, 3.0], np.float32)
    W = np.array([[1.0, 0.0, 2.0], [-3.0, 0.0, 0.5]], np.float32)
    lam = oracle_mod.smooth_scales(s, W, 0.5)
    assert lam[0] == 1.0 and lam[1] == 1.0
    assert lam[2] == np.float32(np.sqrt(np.float32(3.0))) / np.float32(np.sqrt(np.float32(2.0)))


# ------------------------------------------------------------- epilogue (a5)

def test_epilogue_identity_small_ints(oracle_mod):
    acc = np.arange(-255, 256, dtype=np.int32).reshape(7, 73)
    Y = oracle_mod.epilogue(acc, np.ones(7, np.float32), np.ones(73, np.float32), None)
    np.testing.assert_array_equal(f32_of_bf16(Y), acc.astype(np.float32))


def test_epilogue_within_one_bf16_ulp_of_float64(oracle_mod):
    acc = (wl.random_f32((40, 64), seed=18) * 3e6).astype(np.int32)
    sx = np.abs(wl.random_f32((40,), seed=19, scale=0.05)).astype(np.float32)
    sw = np.abs(wl.random_f32((64,), seed=20, scale=2e-4)).astype(np.float32)
    b = wl.random_f32((64,), seed=21, scale=0.01)
    Y = f32_of_bf16(oracle_mod.epilogue(acc, sx, sw, b)).astype(np.float64)
    ref = acc.astype(np.float64) * sx[:, None].astype(np.float64) * sw[None, :] + b[None, :]
    # bf16 has 8 significant bits: one ulp is at most 2^-7 relative
    assert np.all(np.abs(Y - ref) <= np.abs(ref) * 2.0 ** -7 + 1e-30)
    # with the bias dropped the result moves by more than the rounding allows
    Y0 = f32_of_bf16(oracle_mod.epilogue(acc, sx, sw, None)).astype(np.float64)
    assert np.any(np.abs(Y0 - ref) > np.abs(ref) * 2.0 ** -7)


# --------------------------------------------- end to end (a1..a5) bounds

def _e2e_bound_holds(X, W, b, lam, Xq, sx, Wq, sw, Y):
    """|Y - (X W^T + b)| within the bound implied by the quantization errors."""
    x = f32_of_bf16(X).astype(np.float64)
    lam64 = lam.astype(np.float64)
    xs = x / lam64[None, :]
    ws = W.astype(np.float64) * lam64[None, :]
    ref = x @ W.astype(np.float64).T + b[None, :].astype(np.float64)
    ex = sx.astype(np.float64) / 2 * (1 + 2.0 ** -13) + np.abs(xs).max(1) * 2.0 ** -22
    ew = sw.astype(np.float64) / 2 * (1 + 2.0 ** -13) + np.abs(ws).max(1) * 2.0 ** -22
    wq_abs = (np.abs(Wq.astype(np.float64)) * sw.astype(np.float64)[:, None]).sum(1)
    bound = ex[:, None] * wq_abs[None, :] + np.abs(xs).sum(1)[:, None] * ew[None, :]
    y = f32_of_bf16(Y).astype(np.float64)
    tol = bound * (1 + 2.0 ** -7) + np.abs(ref) * 2.0 ** -7 + 1e-6
    return bool(np.all(np.abs(y - ref) <= tol)), float(np.median(bound))


def _run_layer(oracle_mod, c, alpha=0.5):
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], alpha)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    Xq, sx = oracle_mod.quant_act(c.X[0], lam)
    Y = oracle_mod.linear(Xq, sx, Wq, sw, c.bias[0])
    return lam, Xq, sx, Wq, sw, Y


def test_end_to_end_within_quantization_bound(oracle_mod):
    c = wl.make_case(48, 512, 80, seed=22, outlier_frac=0.01, outlier_mult=30.0)
    lam, Xq, sx, Wq, sw, Y = _run_layer(oracle_mod, c)
    ok, _ = _e2e_bound_holds(c.X[0], c.W[0], c.bias[0], lam, Xq, sx, Wq, sw, Y)
    assert ok


def test_smoothing_identity_exact_in_reals(oracle_mod):
    """(X diag(lambda)^-1)(diag(lambda) W^T) = X W^T in exact arithmetic."""
    c = wl.make_case(16, 256, 24, seed=23)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], 0.5).astype(np.float64)
    x = f32_of_bf16(c.X[0]).astype(np.float64)
    W = c.W[0].astype(np.float64)
    lhs = (x / lam[None, :]) @ (W * lam[None, :]).T
    np.testing.assert_allclose(lhs, x @ W.T, rtol=1e-12, atol=1e-12)


def test_bound_detects_wrong_smoothing_direction(oracle_mod):
    """Plant a mistake in the oracle's inputs: activations multiplied (not
    divided) by lambda while weights are multiplied too.  The bound must fail."""
    c = wl.make_case(48, 512, 80, seed=22, outlier_frac=0.01, outlier_mult=30.0)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], 0.5)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    inv = (np.float32(1) / lam).astype(np.float32)
    Xq, sx = oracle_mod.quant_act(c.X[0], inv)         # wrong direction
    Y = oracle_mod.linear(Xq, sx, Wq, sw, c.bias[0])
    ok, _ = _e2e_bound_holds(c.X[0], c.W[0], c.bias[0], lam, Xq, sx, Wq, sw, Y)
    assert not ok


def test_bound_detects_transposed_weight_scale(oracle_mod):
    """Plant a mistake: per-channel weight scales applied in reversed order."""
    c = wl.make_case(48, 512, 80, seed=24)
    lam, Xq, sx, Wq, sw, Y = _run_layer(oracle_mod, c)
    Ybad = oracle_mod.linear(Xq, sx, Wq, sw[::-1].copy(), c.bias[0])
    ok, _ = _e2e_bound_holds(c.X[0], c.W[0], c.bias[0], lam, Xq, sx, Wq, sw, Ybad)
    assert not ok


def test_dual_is_two_singles(oracle_mod):
    c = wl.make_case(20, 128, 32, seed=25, branches=2)
    br = []
    for i in range(2):
        s = oracle_mod.channel_absmax(c.X_cal)
        lam = oracle_mod.smooth_scales(s, c.W[i], 0.5)
        Wq, sw = oracle_mod.quantize_weights(c.W[i], lam)
        Xq, sx = oracle_mod.quant_act(c.X[i], lam)
        br.append((Xq, sx, Wq, sw, c.bias[i]))
    ys = oracle_mod.linear_dual(br)
    for i in range(2):
        np.testing.assert_array_equal(ys[i], oracle_mod.linear(*br[i]))
