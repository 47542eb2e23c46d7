"""GPU parity of w8a8_linear on int8 codes with a workspace.

With a workspace the int8 codes are first written as fp16 values, with each
token's sum of squared codes, by a streaming pass, and the GEMM with the
weights in tensor memory runs on them (the drain plan, the single-run bound
and the split-K area as for the fp16-code linear).  Integer products are exact
on both engines, so the bar is bitwise: the int32 product equals the int64
product of the codes (including -128, which a3 never writes but the int8
container holds), Y equals the oracle and the call without a workspace, and
the dual call equals two single calls.  The cases cover ragged M and N, a
ragged last K chunk, K = 16384, the largest accepted K (products at the int32
limit), partial sums near 2^24, fewer tiles than CTA pairs, an empty branch,
and a workspace reused across calls.
"""

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def w8():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    w8a8.lib()
    return w8a8


def t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(DEV)


def u16(x):
    return x.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def split_counters_zero(w8, ws):
    pairs = torch.cuda.get_device_properties(0).multi_processor_count // 2
    n = ((pairs * 16 * 4 + 255) // 256) * 256
    return not ws[:n].any().item()


def codes_case(M, N, K, kind, seed):
    rng = np.random.default_rng(seed)
    if kind == "random":                    # the whole int8 range, -128 included
        Xq = rng.integers(-128, 128, (M, K), dtype=np.int8)
        Wq = rng.integers(-127, 128, (N, K), dtype=np.int8)
    else:                                   # partial sums of one sign near 2^24
        Xq = np.where(rng.random((M, K)) < 0.3, 125, 127).astype(np.int8)
        Wq = np.full((N, K), 127, np.int8)
        Xq[: M // 2] = -Xq[: M // 2]
    return Xq, Wq


@pytest.mark.parametrize("M,N,K,kind", [
    (512, 1024, 4096, "random"),      # 8 tiles: fewer than the pairs
    (300, 520, 3072, "random"),       # ragged M and N
    (1000, 1000, 2064, "random"),     # ragged last K chunk
    (257, 264, 16384, "random"),      # K = 16384
    (600, 512, 4096, "extreme"),      # drains inside the runs
])
@pytest.mark.parametrize("with_plan", [True, False])
def test_int32_exact_with_workspace(w8, M, N, K, kind, with_plan):
    Xq, Wq = codes_case(M, N, K, kind, M + N + K)
    plan = w8.chunk_plan(t(Wq)) if with_plan else None
    ws = w8.linear_workspace(M, K)
    acc = w8.debug_gemm_i32(t(Xq), t(Wq), plan=plan, workspace=ws)
    want = Xq.astype(np.int64) @ Wq.astype(np.int64).T
    np.testing.assert_array_equal(acc.cpu().numpy(), want)
    assert torch.equal(acc, w8.debug_gemm_i32(t(Xq), t(Wq)))
    assert split_counters_zero(w8, ws)
    assert w8.device_status() == 0


@pytest.mark.parametrize("M,N,K", [(600, 1040, 4096), (257, 264, 2048), (1300, 776, 1040)])
@pytest.mark.parametrize("with_bias", [True, False])
def test_linear_with_workspace_matches_oracle(w8, oracle_mod, M, N, K, with_bias):
    c = wl.make_case(M, K, N, seed=M + 3 * N + K)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    b = c.bias[0] if with_bias else None
    Xq, sx = w8.quant_act(bf(c.X[0]), t(lam))
    plan = w8.chunk_plan(t(Wq))
    ws = w8.linear_workspace(M, K)
    Ys = [w8.linear(Xq, sx, t(Wq), t(sw), t(b) if with_bias else None, plan=plan, workspace=ws)
          for _ in range(3)]                                    # the workspace is reused
    Xq_ref, sx_ref = oracle_mod.quant_act(c.X[0], lam)
    want = oracle_mod.linear(Xq_ref, sx_ref, Wq, sw, b)
    np.testing.assert_array_equal(u16(Ys[0]), want)
    Y0 = w8.linear(Xq, sx, t(Wq), t(sw), t(b) if with_bias else None)
    for Y in Ys:
        assert torch.equal(Y, Y0)
    Y_noplan = w8.linear(Xq, sx, t(Wq), t(sw), t(b) if with_bias else None, workspace=ws)
    assert torch.equal(Y_noplan, Y0)
    assert split_counters_zero(w8, ws)


def test_qkv_shape_equals_unsplit(w8):
    # the benchmarked shape: 864 tiles, single-run tiles (Gaussian codes)
    M, N, K = 4608, 12288, 4096
    g = torch.Generator(device=DEV).manual_seed(12)
    Xq = torch.randint(-127, 128, (M, K), generator=g, device=DEV, dtype=torch.int32).to(torch.int8)
    Wq = (torch.randn(N, K, generator=g, device=DEV) * 40).round().clamp(-127, 127).to(torch.int8)
    sx = torch.rand(M, generator=g, device=DEV) * 1e-3
    sw = torch.rand(N, generator=g, device=DEV) * 1e-3
    bias = torch.randn(N, generator=g, device=DEV)
    plan = w8.chunk_plan(Wq)
    ws = w8.linear_workspace(M, K)
    Y1 = w8.linear(Xq, sx, Wq, sw, bias, plan=plan, workspace=ws)
    Y0 = w8.linear(Xq, sx, Wq, sw, bias)
    assert torch.equal(Y1, Y0)
    # the same codes through the fp16-code entry points give the same bits
    q16 = Xq.to(torch.float16)
    ss = (Xq.to(torch.int32) ** 2).sum(1, dtype=torch.int32)
    assert torch.equal(Y1, w8.linear_f16codes(q16, sx, Wq, sw, bias, plan=plan, x_sumsq=ss))
    acc1 = w8.debug_gemm_i32(Xq, Wq, plan=plan, workspace=ws)
    acc0 = w8.debug_gemm_i32(Xq, Wq)
    assert torch.equal(acc1, acc0)
    assert split_counters_zero(w8, ws)
    assert w8.device_status() == 0


@pytest.mark.parametrize("kind", ["random", "edge"])
def test_int32_exact_largest_k(w8, kind):
    # K = 133136, the largest accepted K: 127^2 K = 2147350544 is 133103 below
    # 2^31 - 1, so the "edge" products sit at the int32 limit, of either sign
    M, N, K = 130, 136, 133136
    rng = np.random.default_rng(kind == "edge")
    if kind == "random":
        Xq = rng.integers(-127, 128, (M, K), dtype=np.int8)
        Wq = rng.integers(-127, 128, (N, K), dtype=np.int8)
    else:
        Xq = np.full((M, K), 127, np.int8)
        Xq[::2] = -127
        Wq = np.full((N, K), 127, np.int8)
        Wq[1::3] = -127
    # every partial sum is an integer below 2^53: the float64 product is exact
    want = (Xq.astype(np.float64) @ Wq.astype(np.float64).T).astype(np.int64)
    if kind == "edge":
        assert np.abs(want).max() == 127 * 127 * K and want.min() == -127 * 127 * K
    plan = w8.chunk_plan(t(Wq))
    ws = w8.linear_workspace(M, K)
    for kw in ({}, {"plan": plan}, {"workspace": ws}, {"plan": plan, "workspace": ws}):
        acc = w8.debug_gemm_i32(t(Xq), t(Wq), **kw)
        np.testing.assert_array_equal(acc.cpu().numpy(), want)
    assert split_counters_zero(w8, ws)
    assert w8.device_status() == 0


def test_layer_forward_largest_k(w8, oracle_mod):
    # K > 16384: a3 writes int8 codes (fp16 codes are limited to K <= 16384)
    # and the workspace call expands them before the GEMM
    M, N, K = 70, 136, 133136
    c = wl.make_case(M, K, N, seed=29, calib_tokens=32)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    Xq_ref, sx_ref = oracle_mod.quant_act(c.X[0], lam)
    want = oracle_mod.linear(Xq_ref, sx_ref, Wq, sw, c.bias[0])
    args = dict(smooth=t(lam), Wq=t(Wq), w_scale=t(sw), bias=t(c.bias[0]))
    Y0 = w8.layer_forward(bf(c.X[0]), False, N, K, **args)
    np.testing.assert_array_equal(u16(Y0), want)
    ws = w8.linear_workspace(M, K)
    for _ in range(2):                                          # the workspace is reused
        Y1 = w8.layer_forward(bf(c.X[0]), False, N, K, plan=w8.chunk_plan(t(Wq)), workspace=ws, **args)
        assert torch.equal(Y1, Y0)
    assert split_counters_zero(w8, ws)


@pytest.mark.parametrize("M0,M1", [(300, 130), (2000, 800), (0, 257), (513, 0)])
def test_dual_with_workspace_equals_singles(w8, oracle_mod, M0, M1):
    N, K = 520, 2064
    branches = []
    for b, M in enumerate((M0, M1)):
        c = wl.make_case(max(M, 1), K, N, seed=5 * M + b)
        s = oracle_mod.channel_absmax(c.X_cal)
        lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
        Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
        X = c.X[0][:M]
        if M:
            Xq, sx = w8.quant_act(bf(X), t(lam))
        else:
            Xq, sx = torch.empty(0, K, dtype=torch.int8, device=DEV), torch.empty(0, device=DEV)
        branches.append((Xq, sx, t(Wq), t(sw), t(c.bias[0]), w8.chunk_plan(t(Wq))))
    ws = w8.linear_workspace(M0 + M1, K)
    Y1 = w8.linear_dual(branches, workspace=ws)
    Y0 = w8.linear_dual([br[:5] for br in branches])
    for i, (a, b) in enumerate(zip(Y1, Y0)):
        assert torch.equal(a, b)
        if branches[i][0].shape[0]:
            assert torch.equal(a, w8.linear(*branches[i][:5], plan=branches[i][5],
                                            workspace=w8.linear_workspace(branches[i][0].shape[0], K)))
    assert split_counters_zero(w8, ws)


def test_workspace_size_checked(w8):
    Xq = torch.zeros(256, 1024, dtype=torch.int8, device=DEV)
    Wq = torch.zeros(256, 1024, dtype=torch.int8, device=DEV)
    sx = torch.zeros(256, device=DEV)
    with pytest.raises(ValueError):
        w8.linear(Xq, sx, Wq, sx, workspace=w8.linear_workspace(255, 1024))
    with pytest.raises(ValueError):
        w8.linear(Xq, sx, Wq, sx, workspace=torch.zeros(w8.linear_workspace_size(256, 1024) // 4,
                                                        dtype=torch.int32, device=DEV))
    Y = w8.linear(Xq, sx, Wq, sx, workspace=w8.linear_workspace(256, 1024))
    assert not Y.float().any().item()
