"""GPU parity of the fp16-code GEMM with a split-K workspace.

With a workspace, as many output tiles as a last, partial round over the CTA
pairs would hold (all tiles, when there are fewer tiles than pairs) are split
over consecutive K chunks between pairs of the first round; the parts' int32
sums meet in the workspace and the last part to finish adds them.  Integer sums are exact in
any order, so the bar is bitwise: the int32 product equals the int64 product
of the codes, and every output equals the call without a workspace.  The
cases cover fewer tiles than pairs, a partial last round, an odd number of K
chunks, a ragged last chunk, ragged M and N, partial sums near 2^24 (drains
inside a part), the single-run path (token sums), both branches, and a
workspace reused across calls (its counters return to zero).
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


def pairs():
    return torch.cuda.get_device_properties(0).multi_processor_count // 2


def counters_zero(ws):
    n = ((pairs() * 16 * 4 + 255) // 256) * 256
    return not ws[:n].any().item()


def codes_case(M, N, K, kind, seed):
    rng = np.random.default_rng(seed)
    if kind == "random":
        Xq = rng.integers(-127, 128, (M, K), dtype=np.int8)
        Wq = rng.integers(-127, 128, (N, K), dtype=np.int8)
    else:                                   # partial sums of one sign near 2^24
        Xq = np.where(rng.random((M, K)) < 0.3, 125, 127).astype(np.int8)
        Wq = np.full((N, K), 127, np.int8)
        Xq[: M // 2] = -Xq[: M // 2]
    return Xq, Wq


@pytest.mark.parametrize("M,N,K,kind", [
    (512, 1024, 4096, "random"),      # 8 tiles: fewer than the pairs, 4 chunks
    (2560, 2304, 4096, "random"),     # 90 tiles: a partial second round
    (2560, 3072, 4096, "random"),     # 120 tiles: 44 left over, more than half the pairs: no split
    (300, 520, 3072, "random"),       # 6 tiles, 3 chunks, ragged M and N
    (1000, 1000, 2064, "random"),     # 16 tiles, ragged last chunk
    (600, 512, 4096, "extreme"),      # drains inside the parts
])
@pytest.mark.parametrize("with_plan", [True, False])
def test_split_int32_exact(w8, M, N, K, kind, with_plan):
    Xq, Wq = codes_case(M, N, K, kind, M + N + K)
    q16 = torch.from_numpy(Xq.astype(np.float16)).to(DEV)
    plan = w8.chunk_plan(t(Wq)) if with_plan else None
    ws = w8.gemm_workspace()
    acc = w8.debug_gemm_f16codes_i32(q16, t(Wq), plan=plan, workspace=ws)
    want = Xq.astype(np.int64) @ Wq.astype(np.int64).T
    np.testing.assert_array_equal(acc.cpu().numpy(), want)
    assert torch.equal(acc, w8.debug_gemm_f16codes_i32(q16, t(Wq), plan=plan))
    assert counters_zero(ws)
    assert w8.device_status() == 0


@pytest.mark.parametrize("M,N,K", [(600, 1040, 4096), (257, 264, 2048)])
def test_split_linear_bitwise_with_sumsq(w8, oracle_mod, M, N, K):
    c = wl.make_case(M, K, N, seed=M + 5 * N + K)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    ss = torch.empty(M, dtype=torch.int32, device=DEV)
    q16, sx = w8.quant_act_f16codes(bf(c.X[0]), t(lam), sumsq=ss)
    plan = w8.chunk_plan(t(Wq))
    ws = w8.gemm_workspace()
    Ys = [w8.linear_f16codes(q16, sx, t(Wq), t(sw), t(c.bias[0]), plan=plan, x_sumsq=ss, workspace=ws)
          for _ in range(3)]                                  # the workspace is reused
    Y0 = w8.linear_f16codes(q16, sx, t(Wq), t(sw), t(c.bias[0]), plan=plan, x_sumsq=ss)
    Xq, wsx = oracle_mod.quant_act(c.X[0], lam)
    np.testing.assert_array_equal(u16(Ys[0]), oracle_mod.linear(Xq, wsx, Wq, sw, c.bias[0]))
    for Y in Ys:
        assert torch.equal(Y, Y0)
    assert counters_zero(ws)


def test_split_qkv_shape_equals_unsplit(w8):
    # the benchmarked shape: 864 tiles on 76 pairs, 28 of them split in two
    M, N, K = 4608, 12288, 4096
    g = torch.Generator(device=DEV).manual_seed(11)
    q16 = torch.randint(-127, 128, (M, K), generator=g, device=DEV, dtype=torch.int32).to(torch.float16)
    Wq = torch.randint(-127, 128, (N, K), generator=g, device=DEV, dtype=torch.int32).to(torch.int8)
    sx = torch.rand(M, generator=g, device=DEV) * 1e-3
    sw = torch.rand(N, generator=g, device=DEV) * 1e-3
    bias = torch.randn(N, generator=g, device=DEV)
    ss = (q16.to(torch.int32) ** 2).sum(1, dtype=torch.int32)
    plan = w8.chunk_plan(Wq)
    ws = w8.gemm_workspace()
    for sums in (None, ss):
        Y1 = w8.linear_f16codes(q16, sx, Wq, sw, bias, plan=plan, x_sumsq=sums, workspace=ws)
        Y0 = w8.linear_f16codes(q16, sx, Wq, sw, bias, plan=plan, x_sumsq=sums)
        assert torch.equal(Y1, Y0)
    acc1 = w8.debug_gemm_f16codes_i32(q16, Wq, plan=plan, workspace=ws)
    acc0 = w8.debug_gemm_f16codes_i32(q16, Wq, plan=plan)
    assert torch.equal(acc1, acc0)
    assert counters_zero(ws)
    assert w8.device_status() == 0


@pytest.mark.parametrize("M0,M1", [(300, 130), (2000, 800), (0, 257)])
def test_split_dual_equals_unsplit(w8, oracle_mod, M0, M1):
    N, K = 520, 2064
    branches = []
    for b, M in enumerate((M0, M1)):
        c = wl.make_case(max(M, 1), K, N, seed=3 * M + b)
        s = oracle_mod.channel_absmax(c.X_cal)
        lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
        Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
        X = c.X[0][:M]
        ss = torch.empty(M, dtype=torch.int32, device=DEV)
        if M:
            q16, sx = w8.quant_act_f16codes(bf(X), t(lam), sumsq=ss)
        else:
            q16, sx = torch.empty(0, K, dtype=torch.float16, device=DEV), torch.empty(0, device=DEV)
        branches.append((q16, sx, t(Wq), t(sw), t(c.bias[0]), w8.chunk_plan(t(Wq)), ss))
    ws = w8.gemm_workspace()
    Y1 = w8.linear_dual_f16codes(branches, workspace=ws)
    Y0 = w8.linear_dual_f16codes(branches)
    for a, b in zip(Y1, Y0):
        assert torch.equal(a, b)
    assert counters_zero(ws)


def test_workspace_size_and_checks(w8):
    assert w8.gemm_workspace_size() >= pairs() * 256 * 256 * 4
    q16 = torch.zeros(256, 1024, dtype=torch.float16, device=DEV)
    Wq = torch.zeros(256, 1024, dtype=torch.int8, device=DEV)
    with pytest.raises(ValueError):
        w8.debug_gemm_f16codes_i32(q16, Wq, workspace=torch.zeros(16, dtype=torch.uint8, device=DEV))
    with pytest.raises(ValueError):
        w8.debug_gemm_f16codes_i32(q16, Wq, workspace=torch.zeros(w8.gemm_workspace_size(), dtype=torch.int32,
                                                                   device=DEV))


def test_split_dual_workload_equals_unsplit(w8):
    # the dual-branch workload's shape: 576 tiles on 76 pairs leave 44, more
    # than half the pairs, so the launch runs unsplit with the workspace too
    M, N, K = 4608, 4096, 4096
    g = torch.Generator(device=DEV).manual_seed(13)
    brs = []
    for b in range(2):
        q16 = torch.randint(-127, 128, (M, K), generator=g, device=DEV, dtype=torch.int32).to(torch.float16)
        Wq = torch.randint(-127, 128, (N, K), generator=g, device=DEV, dtype=torch.int32).to(torch.int8)
        sx = torch.rand(M, generator=g, device=DEV) * 1e-3
        sw = torch.rand(N, generator=g, device=DEV) * 1e-3
        bias = torch.randn(N, generator=g, device=DEV)
        ss = (q16.to(torch.int32) ** 2).sum(1, dtype=torch.int32)
        brs.append((q16, sx, Wq, sw, bias, w8.chunk_plan(Wq), ss))
    ws = w8.gemm_workspace()
    Y1 = w8.linear_dual_f16codes(brs, workspace=ws)
    Y0 = w8.linear_dual_f16codes(brs)
    for a, b in zip(Y1, Y0):
        assert torch.equal(a, b)
    assert counters_zero(ws)
    assert w8.device_status() == 0
