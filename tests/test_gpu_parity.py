"""GPU parity: every kernel, called through the C ABI, against the CPU oracle.

Bar: INT8 codes, FP32 scales, lambda (alpha in {0, 1/2, 1}) and the INT32
product bit-exact; bf16 outputs within 1 bf16 ulp (relative 2^-8), and in fact
bit-identical because both sides follow the same pinned fp32 op order.  Sizes
span several tiles with ragged tails; edge cases cover empty and single-row
inputs, all-zero rows and columns, adversarial INT8 extremes and the largest K.
The product GEMM (tcgen05 on SM pairs) is checked through w8a8_linear and the
earlier engines kept as test anchors (tcgen05 on single SMs, mma.sync)
through the test-only entry point that takes the engine per call.
"""

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

ENGINES = ["tcgen05_pair", "tcgen05", "mma_sync"]
DEBUG_ENGINE = {"tcgen05": 1, "mma_sync": 0}


@pytest.fixture(scope="module")
def w8():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    w8a8.lib()
    yield w8a8


class Engine:
    """One GEMM engine behind the calls the tests make: the product engine
    through w8a8_linear / w8a8_linear_dual / w8a8_debug_gemm_i32, the others
    through the test-only entry point that takes the engine as an argument."""

    def __init__(self, w8, name):
        self.w8, self.name = w8, name

    def linear(self, Xq, sx, Wq, sw, b=None, Y=None):
        if self.name in DEBUG_ENGINE:
            return self.w8.debug_linear_engine(DEBUG_ENGINE[self.name], [(Xq, sx, Wq, sw, b)],
                                               Ys=None if Y is None else [Y])[0]
        return self.w8.linear(Xq, sx, Wq, sw, b, Y=Y)

    def debug_gemm_i32(self, Xq, Wq, acc=None):
        if self.name in DEBUG_ENGINE:
            return self.w8.debug_linear_engine(DEBUG_ENGINE[self.name], [(Xq, None, Wq, None, None)],
                                               Ys=None if acc is None else [acc], out_i32=True)[0]
        return self.w8.debug_gemm_i32(Xq, Wq, acc=acc)

    def linear_dual(self, brs):
        if self.name in DEBUG_ENGINE:
            return self.w8.debug_linear_engine(DEBUG_ENGINE[self.name], brs)
        return self.w8.linear_dual(brs)


@pytest.fixture(params=ENGINES)
def engine(request, w8):
    return Engine(w8, request.param)


DEV = "cuda"


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(DEV)


def t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def u16(x):
    return x.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def assert_bf16_close(got_u16, want_u16, max_ulp=1):
    g = got_u16.astype(np.int32)
    w = want_u16.astype(np.int32)
    diff = np.abs(g - w)
    assert diff.max(initial=0) <= max_ulp, f"max bf16 ulp diff {diff.max()}"


# ---------------------------------------------------------- calibration / a1

@pytest.mark.parametrize("T,K", [(1, 16), (300, 528), (256, 4096), (37, 16384 + 16)])
def test_channel_absmax(w8, oracle_mod, T, K):
    X = wl.random_bf16((T, K), seed=T + K, scale=2.0)
    got = w8.channel_absmax(bf(X)).cpu().numpy()
    np.testing.assert_array_equal(got, oracle_mod.channel_absmax(X))


@pytest.mark.parametrize("alpha", [0.5, 1.0, 0.0])
@pytest.mark.parametrize("N,K", [(8, 16), (264, 1040), (4096, 512)])
def test_smooth_scales_exact(w8, oracle_mod, alpha, N, K):
    c = wl.make_case(4, K, N, seed=N + K)
    s = oracle_mod.channel_absmax(c.X_cal)
    W = c.W[0].copy()
    W[:, 3] = 0.0                           # a zero weight column -> lambda 1
    s[5] = 0.0                              # a zero activation channel -> lambda 1
    got = w8.smooth_scales(t(s), t(W), alpha).cpu().numpy()
    np.testing.assert_array_equal(got, oracle_mod.smooth_scales(s, W, alpha))


def test_smooth_scales_general_alpha_one_ulp(w8, oracle_mod):
    c = wl.make_case(4, 1040, 264, seed=9)
    s = oracle_mod.channel_absmax(c.X_cal)
    for alpha in (0.25, 0.65):
        got = w8.smooth_scales(t(s), t(c.W[0]), alpha).cpu().numpy()
        want = oracle_mod.smooth_scales(s, c.W[0], alpha)
        ulps = np.abs(got.view(np.int32).astype(np.int64) - want.view(np.int32).astype(np.int64))
        assert ulps.max() <= 1


# ------------------------------------------------------------------ a2 / a3

@pytest.mark.parametrize("N,K", [(8, 16), (264, 1040), (520, 4096), (24, 16384), (16, 20016)])
@pytest.mark.parametrize("smooth", [True, False])
def test_quantize_weights(w8, oracle_mod, N, K, smooth):
    W = wl.random_f32((N, K), seed=N * 7 + K, scale=0.02)
    W[min(3, N - 1)] = 0.0                  # an all-zero output channel
    lam = (np.abs(wl.random_f32((K,), seed=K)) + 0.1).astype(np.float32) if smooth else None
    Wq, sw = w8.quantize_weights(t(W), t(lam) if smooth else None)
    Wq_ref, sw_ref = oracle_mod.quantize_weights(W, lam)
    np.testing.assert_array_equal(Wq.cpu().numpy(), Wq_ref)
    np.testing.assert_array_equal(sw.cpu().numpy(), sw_ref)


# K spans every team width of the warp-team kernel (K <= 256, 512, 1024, 2048,
# 4096, 8192, 16384 values per row, each with a ragged last chunk) and the
# long-row kernel beyond
@pytest.mark.parametrize("M,K", [(1, 16), (7, 48), (2, 256), (1000, 272), (129, 528), (77, 2064),
                                 (300, 4096), (513, 4112), (40, 8208), (33, 16384), (5, 20016), (4608, 512)])
@pytest.mark.parametrize("smooth", [True, False])
def test_quant_act(w8, oracle_mod, M, K, smooth):
    c = wl.make_case(M, K, 16, seed=M + K, outlier_frac=0.01, outlier_mult=30.0)
    X = c.X[0].copy()
    X[M // 2] = 0                          # an all-zero token
    lam = None
    if smooth:
        s = oracle_mod.channel_absmax(c.X_cal)
        lam = oracle_mod.smooth_scales(s, c.W[0], 0.5)
    Xq, sx = w8.quant_act(bf(X), t(lam) if smooth else None)
    Xq_ref, sx_ref = oracle_mod.quant_act(X, lam)
    np.testing.assert_array_equal(Xq.cpu().numpy(), Xq_ref)
    np.testing.assert_array_equal(sx.cpu().numpy(), sx_ref)


def test_quant_act_round_half_even_and_tiny(w8, oracle_mod):
    # ties at every half-integer, plus values so small that 127/absmax overflows
    row = np.array([127.0, 0.5, 1.5, 2.5, -0.5, -2.5, 3.5, -3.5] + [0.0] * 8, np.float32)
    tiny = np.zeros(16, np.float32)
    tiny[0] = 1e-38
    tiny[1] = -3e-39
    X = torch.tensor(np.stack([row, tiny])).to(torch.bfloat16)
    Xn = X.view(torch.int16).numpy().view(np.uint16)
    Xq, sx = w8.quant_act(X.to(DEV), None)
    Xq_ref, sx_ref = oracle_mod.quant_act(Xn, None)
    np.testing.assert_array_equal(Xq.cpu().numpy(), Xq_ref)
    np.testing.assert_array_equal(sx.cpu().numpy(), sx_ref)


# ------------------------------------------------------------------ a4 (+a5)

GEMM_SHAPES = [(1, 8, 16), (7, 24, 48), (129, 136, 528), (300, 264, 1040),
               (257, 520, 2064), (128, 256, 64), (513, 392, 4112)]


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
def test_gemm_i32_exact(w8, engine, oracle_mod, M, N, K):
    Xq = wl.random_int8((M, K), seed=M * 3 + K)
    Wq = wl.random_int8((N, K), seed=N * 5 + K)
    acc = engine.debug_gemm_i32(t(Xq), t(Wq)).cpu().numpy()
    np.testing.assert_array_equal(acc, oracle_mod.gemm_i32(Xq, Wq))


@pytest.mark.parametrize("pattern", ["all_plus", "plus_minus", "alternating", "random_extreme"])
def test_gemm_i32_adversarial_k16384(w8, engine, oracle_mod, pattern):
    M, N, K = 136, 264, 16384
    if pattern == "all_plus":
        Xq = np.full((M, K), 127, np.int8)
        Wq = np.full((N, K), 127, np.int8)
        Wq[1::2] = -127
    elif pattern == "plus_minus":
        Xq = np.full((M, K), -127, np.int8)
        Wq = np.full((N, K), 127, np.int8)
    elif pattern == "alternating":
        sgn = np.where(np.arange(K) % 2 == 0, 127, -127).astype(np.int8)
        Xq = np.tile(sgn, (M, 1))
        Wq = np.tile(sgn, (N, 1))
        Wq[::3] = -Wq[::3]
        # a block structure that makes partial sums climb then fall
        Xq[:, K // 2:] = 127
    else:
        g = np.random.default_rng(0)
        Xq = (g.integers(0, 2, (M, K)) * 254 - 127).astype(np.int8)
        Wq = (g.integers(0, 2, (N, K)) * 254 - 127).astype(np.int8)
    acc = engine.debug_gemm_i32(t(Xq), t(Wq)).cpu().numpy()
    want = oracle_mod.gemm_i32(Xq, Wq)
    np.testing.assert_array_equal(acc, want)


def test_gemm_i32_max_k(w8, engine, oracle_mod):
    K = 133136                      # largest multiple of 16 <= the int32 bound
    Xq = np.full((3, K), 127, np.int8)
    Xq[1] = -127
    Wq = np.full((8, K), 127, np.int8)
    Wq[2, ::2] = -127
    acc = engine.debug_gemm_i32(t(Xq), t(Wq)).cpu().numpy()
    np.testing.assert_array_equal(acc, oracle_mod.gemm_i32(Xq, Wq))


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
@pytest.mark.parametrize("with_bias", [True, False])
def test_linear(w8, engine, oracle_mod, M, N, K, with_bias):
    Xq = wl.random_int8((M, K), seed=M + 11 * K)
    Wq = wl.random_int8((N, K), seed=N + 13 * K)
    sx = np.abs(wl.random_f32((M,), seed=M, scale=0.03)).astype(np.float32)
    sw = np.abs(wl.random_f32((N,), seed=N, scale=1e-4)).astype(np.float32)
    b = wl.random_f32((N,), seed=N + 1, scale=0.01) if with_bias else None
    Y = engine.linear(t(Xq), t(sx), t(Wq), t(sw), t(b) if with_bias else None)
    want = oracle_mod.linear(Xq, sx, Wq, sw, b)
    assert_bf16_close(u16(Y), want)
    np.testing.assert_array_equal(u16(Y), want)   # same pinned op order


def test_linear_empty_and_dual_ragged(w8, engine, oracle_mod):
    N, K = 264, 528
    Wq = [wl.random_int8((N, K), seed=40 + i) for i in range(2)]
    sw = [np.abs(wl.random_f32((N,), seed=50 + i, scale=1e-4)).astype(np.float32) for i in range(2)]
    b = [wl.random_f32((N,), seed=60 + i, scale=0.01) for i in range(2)]
    # M = 0 is a no-op
    Y0 = engine.linear(torch.empty(0, K, dtype=torch.int8, device=DEV),
                       torch.empty(0, dtype=torch.float32, device=DEV), t(Wq[0]), t(sw[0]))
    assert Y0.shape == (0, N)
    # branches of different M (one of them ragged, one empty)
    for Ms in ((129, 300), (0, 77)):
        brs, wants = [], []
        for i, M in enumerate(Ms):
            Xq = wl.random_int8((M, K), seed=70 + i + M)
            sx = np.abs(wl.random_f32((M,), seed=80 + i + M, scale=0.03)).astype(np.float32)
            brs.append((t(Xq), t(sx), t(Wq[i]), t(sw[i]), t(b[i])))
            wants.append(oracle_mod.linear(Xq, sx, Wq[i], sw[i], b[i]) if M else None)
        Ys = engine.linear_dual(brs)
        for i, M in enumerate(Ms):
            if M:
                np.testing.assert_array_equal(u16(Ys[i]), wants[i])
                np.testing.assert_array_equal(u16(Ys[i]), u16(engine.linear(*brs[i])))


def test_no_out_of_bounds_writes(w8, engine):
    """Guard bands around Y and acc stay untouched (ragged M and N)."""
    M, N, K = 131, 136, 528
    guard = 4096
    Xq = t(wl.random_int8((M, K), seed=1))
    Wq = t(wl.random_int8((N, K), seed=2))
    sx = torch.ones(M, device=DEV)
    sw = torch.ones(N, device=DEV)
    buf = torch.full((guard + M * N + guard,), 0x7A7B, dtype=torch.int16, device=DEV)
    Y = buf[guard:guard + M * N].view(torch.bfloat16).view(M, N)
    engine.linear(Xq, sx, Wq, sw, None, Y=Y)
    torch.cuda.synchronize()
    assert torch.all(buf[:guard] == 0x7A7B) and torch.all(buf[guard + M * N:] == 0x7A7B)
    buf32 = torch.full((guard + M * N + guard,), 0x5A5A5A5A, dtype=torch.int32, device=DEV)
    acc = buf32[guard:guard + M * N].view(M, N)
    engine.debug_gemm_i32(Xq, Wq, acc=acc)
    torch.cuda.synchronize()
    assert torch.all(buf32[:guard] == 0x5A5A5A5A) and torch.all(buf32[guard + M * N:] == 0x5A5A5A5A)
    assert w8.device_status() == 0


def test_bounded_wait_reports_timeout_and_context_survives(w8):
    """A barrier wait that nothing satisfies gives up after its limit, records
    its code in the device error word, and the context keeps working."""
    assert w8.device_status() == 0
    w8.debug_wait_timeout(20000)                  # 20 ms
    assert w8.device_status() == 128             # reported once ...
    assert w8.device_status() == 0               # ... and cleared
    Xq = t(wl.random_int8((300, 528), seed=90))
    Wq = t(wl.random_int8((264, 528), seed=91))
    acc = w8.debug_gemm_i32(Xq, Wq).cpu().numpy()
    want = Xq.cpu().numpy().astype(np.int64) @ Wq.cpu().numpy().astype(np.int64).T
    np.testing.assert_array_equal(acc, want)
    assert w8.device_status() == 0
