"""GPU parity of the fp16-code GEMM's tile order for large activations.

When a branch's fp16 activation codes exceed what the GEMM plans to keep in
L2 (48 MB), the tiles run in groups of feature blocks (feature block fastest
within a group) instead of token tile fastest.  The order changes which CTA
pair computes which tile and when, never the arithmetic, so the bar is
bitwise: the int32 product equals an exact product (fp64 GEMM of the integer
codes on the GPU: every partial sum is an integer below 2^53), and Y equals
the epilogue applied step by step in fp32 (float(acc), times the token scale,
times the channel scale, plus the bias, rounded once to bf16).  The cases
cover one group, several groups with a ragged last one, K = 16384, the
split-K workspace and both branches.
"""

import pytest
import torch

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def w8():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    w8a8.lib()
    return w8a8


def operands(M, N, K, seed):
    g = torch.Generator(device=DEV).manual_seed(seed)
    q = torch.randint(-127, 128, (M, K), generator=g, device=DEV, dtype=torch.int32)
    w = torch.randint(-127, 128, (N, K), generator=g, device=DEV, dtype=torch.int32)
    sx = torch.rand(M, generator=g, device=DEV) * 1e-3
    sw = torch.rand(N, generator=g, device=DEV) * 1e-3
    b = torch.randn(N, generator=g, device=DEV)
    return q, w, sx, sw, b


def exact_product(q, w):
    return (q.double() @ w.double().T).to(torch.int64)


def epilogue(acc, sx, sw, b):
    t = acc.to(torch.float32)
    t = t * sx[:, None]
    t = t * sw[None, :]
    t = t + b[None, :]
    return t.to(torch.bfloat16)


@pytest.mark.parametrize("M,N,K", [
    (6144, 1040, 4096),     # codes 50 MB: one group of all 5 feature blocks
    (1600, 2304, 16384),    # codes 52 MB, 4 MB weight blocks: one group of 9
    (1600, 12288, 16384),   # groups of 10 feature blocks, the last of 8
])
@pytest.mark.parametrize("with_ws", [False, True])
def test_grouped_order_exact(w8, M, N, K, with_ws):
    q, w, sx, sw, b = operands(M, N, K, M + N + K)
    q16 = q.to(torch.float16)
    wq = w.to(torch.int8)
    plan = w8.chunk_plan(wq)
    ws = w8.gemm_workspace() if with_ws else None
    acc = w8.debug_gemm_f16codes_i32(q16, wq, plan=plan, workspace=ws)
    want = exact_product(q, w)
    assert torch.equal(acc.to(torch.int64), want)
    Y = w8.linear_f16codes(q16, sx, wq, sw, b, plan=plan, workspace=ws)
    assert torch.equal(Y.view(torch.int16), epilogue(acc, sx, sw, b).view(torch.int16))
    assert w8.device_status() == 0


def test_grouped_order_dual(w8):
    # one branch above the threshold, one below: the order is planned for the
    # larger, and both branches' outputs match their single calls
    N, K = 1040, 4096
    brs, singles = [], []
    for i, M in enumerate((6144, 700)):
        q, w, sx, sw, b = operands(M, N, K, 7 + i)
        q16, wq = q.to(torch.float16), w.to(torch.int8)
        plan = w8.chunk_plan(wq)
        ss = (q * q).sum(1, dtype=torch.int32)
        brs.append((q16, sx, wq, sw, b, plan, ss))
        singles.append(w8.linear_f16codes(q16, sx, wq, sw, b, plan=plan, x_sumsq=ss))
    Ys = w8.linear_dual_f16codes(brs)
    for a, s in zip(Ys, singles):
        assert torch.equal(a, s)
    acc = w8.debug_gemm_f16codes_i32(brs[1][0], brs[1][2], plan=brs[1][5])
    assert torch.equal(singles[1].view(torch.int16),
                       epilogue(acc, brs[1][1], brs[1][3], brs[1][4]).view(torch.int16))


# ------------------------------------------- the other engines, same order

def test_grouped_order_int8_engine(w8):
    # int8 codes of 12800 x 4096 (52 MB): above the threshold for 1-byte codes
    M, N, K = 12800, 1040, 4096
    q, w, sx, sw, b = operands(M, N, K, 21)
    acc = w8.debug_gemm_i32(q.to(torch.int8), w.to(torch.int8))
    assert torch.equal(acc.to(torch.int64), exact_product(q, w))
    Y = w8.linear(q.to(torch.int8), sx, w.to(torch.int8), sw, b)
    assert torch.equal(Y.view(torch.int16), epilogue(acc, sx, sw, b).view(torch.int16))


def test_grouped_order_bf16_layer(w8):
    # bf16 activations of 6400 x 4096 (52 MB): within half a bf16 ulp plus the
    # fp32 accumulation bound (K/16 + 16) 2^-22 sum |x w| of the exact product
    M, N, K = 6400, 2304, 4096
    g = torch.Generator(device=DEV).manual_seed(5)
    X = torch.randn(M, K, generator=g, device=DEV).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g, device=DEV) * 0.05).to(torch.bfloat16)
    b = torch.randn(N, generator=g, device=DEV) * 0.1
    Y = w8.linear_bf16(X, W, b).double()
    Xd, Wd = X.double(), W.double()
    ref = Xd @ Wd.T + b.double()[None, :]
    absum = Xd.abs() @ Wd.abs().T
    ulp = torch.pow(2.0, torch.floor(torch.log2(ref.abs().clamp_min(1e-30))) - 7)
    bound = 0.5 * ulp + (K / 16 + 16) * 2.0 ** -22 * absum + 1e-30
    assert bool(((Y - ref).abs() <= bound).all())


@pytest.mark.parametrize("fmt", [0, 1])
def test_grouped_order_gguf_equals_bf16_layer(w8, fmt):
    # the GGUF layer equals the bf16 layer on its decoded weights bitwise,
    # whatever order either visits its tiles in
    from paper_2606_12280_gb300 import workloads as wl
    M, N, K = 6400, 1024, 4096
    raw = torch.from_numpy(wl.random_gguf(fmt, N, K, seed=fmt + 3)).to(DEV)
    g = torch.Generator(device=DEV).manual_seed(9)
    X = torch.randn(M, K, generator=g, device=DEV).to(torch.bfloat16)
    b = torch.randn(N, generator=g, device=DEV) * 0.1
    Wd = w8.debug_gguf_dequant(raw, fmt, N, K)
    assert torch.equal(w8.linear_gguf(X, raw, fmt, N, b), w8.linear_bf16(X, Wd, b))
