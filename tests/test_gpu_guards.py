"""Guard bands around every output of the library's kernels.

compute-sanitizer is not available here, so each output buffer is placed
inside a larger allocation whose leading and trailing 4096 elements hold a
fill pattern; after the call the pattern must be intact (no write outside
the output) and, where the output is checked elsewhere for its values, the
interior must equal an unguarded call bitwise.  Shapes are ragged (M, N and K
not multiples of any tile) so that tail tiles and masked rows are exercised.
"""

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"
G = 4096                         # guard elements on each side (16-byte multiple for every dtype)
FILL = {1: (torch.int8, 0x5A), 2: (torch.int16, 0x7A7B), 4: (torch.int32, 0x5A5A5A5A),
        8: (torch.int64, 0x5A5A5A5A5A5A5A5A)}


@pytest.fixture(scope="module")
def w8():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    w8a8.lib()
    return w8a8


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(DEV)


def t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


class Guarded:
    """An output tensor of `shape` and `dtype` between two guard bands."""

    def __init__(self, shape, dtype, zero=False):
        n = int(np.prod(shape))
        size = torch.empty(0, dtype=dtype).element_size()
        idt, pattern = FILL[size]
        self.raw = torch.full((G + n + G,), pattern, dtype=idt, device=DEV)
        if zero:
            self.raw[G:G + n] = 0
        self.n, self.pattern = n, pattern
        self.t = self.raw[G:G + n].view(dtype).view(*shape)

    def intact(self):
        torch.cuda.synchronize()
        return bool(torch.all(self.raw[:G] == self.pattern)) and bool(torch.all(self.raw[G + self.n:] == self.pattern))


def check(*gs):
    for g in gs:
        assert g.intact()


@pytest.mark.parametrize("M,K", [(131, 528), (1001, 4096), (37, 4112), (37, 16384 + 16)])
def test_quant_act(w8, M, K):
    X = bf(wl.random_bf16((M, K), seed=M + K, scale=2.0))
    lam = t(wl.random_uniform_f32((K,), seed=K, lo=0.25, hi=4.0))
    q, s = Guarded((M, K), torch.int8), Guarded((M,), torch.float32)
    w8.quant_act(X, lam, Xq=q.t, x_scale=s.t)
    check(q, s)
    q0, s0 = w8.quant_act(X, lam)
    assert torch.equal(q.t, q0) and torch.equal(s.t, s0)


@pytest.mark.parametrize("gelu", [False, True])
def test_quant_act_f16codes(w8, gelu):
    M, K = 131, 528
    X = bf(wl.random_bf16((M, K), seed=3, scale=2.0))
    lam = t(wl.random_uniform_f32((K,), seed=4, lo=0.25, hi=4.0))
    q, s, ss = Guarded((M, K), torch.float16), Guarded((M,), torch.float32), Guarded((M,), torch.int32)
    w8.quant_act_f16codes(X, lam, Xq16=q.t, x_scale=s.t, sumsq=ss.t, gelu=gelu)
    check(q, s, ss)
    ss0 = torch.empty(M, dtype=torch.int32, device=DEV)
    q0, s0 = w8.quant_act_f16codes(X, lam, gelu=gelu, sumsq=ss0)
    assert torch.equal(q.t, q0) and torch.equal(s.t, s0) and torch.equal(ss.t, ss0)


def test_quant_act_dual_and_dual_f16codes(w8):
    K = 528
    Ms = (131, 70)
    Xs = [bf(wl.random_bf16((M, K), seed=10 + M, scale=2.0)) for M in Ms]
    lams = [t(wl.random_uniform_f32((K,), seed=20 + i, lo=0.25, hi=4.0)) for i in range(2)]
    out8 = [(Guarded((M, K), torch.int8), Guarded((M,), torch.float32)) for M in Ms]
    w8.quant_act_dual(list(zip(Xs, lams)), out=[(a.t, b.t) for a, b in out8])
    check(*[g for pair in out8 for g in pair])
    out16 = [(Guarded((M, K), torch.float16), Guarded((M,), torch.float32), Guarded((M,), torch.int32))
             for M in Ms]
    w8.quant_act_dual_f16codes(list(zip(Xs, lams)), out=[(a.t, b.t, c.t) for a, b, c in out16])
    check(*[g for trip in out16 for g in trip])
    for i in range(2):
        q0, s0 = w8.quant_act(Xs[i], lams[i])
        assert torch.equal(out8[i][0].t, q0) and torch.equal(out16[i][0].t.to(torch.int8), q0)


def gemm_operands(M, N, K, seed):
    Xq = wl.random_int8((M, K), seed=seed)
    Wq = t(wl.random_int8((N, K), seed=seed + 1))
    sx = t(wl.random_uniform_f32((M,), seed=seed + 2, lo=1e-3, hi=2e-3))
    sw = t(wl.random_uniform_f32((N,), seed=seed + 3, lo=1e-3, hi=2e-3))
    b = t(wl.random_f32((N,), seed=seed + 4, scale=0.01))
    ss = t((Xq.astype(np.int64) ** 2).sum(1).astype(np.uint32).view(np.int32))
    return torch.from_numpy(Xq.astype(np.float16)).to(DEV), t(Xq), Wq, sx, sw, b, ss


@pytest.mark.parametrize("with_plan", [True, False])
def test_linear_f16codes_and_i32(w8, with_plan):
    M, N, K = 131, 136, 528
    q16, q8, Wq, sx, sw, b, ss = gemm_operands(M, N, K, 30)
    plan = w8.chunk_plan(Wq) if with_plan else None
    Y = Guarded((M, N), torch.bfloat16)
    w8.linear_f16codes(q16, sx, Wq, sw, b, Y=Y.t, plan=plan, x_sumsq=ss if with_plan else None)
    check(Y)
    assert torch.equal(Y.t, w8.linear(q8, sx, Wq, sw, b))
    acc = Guarded((M, N), torch.int32)
    w8.debug_gemm_f16codes_i32(q16, Wq, plan=plan, x_sumsq=ss if with_plan else None, acc=acc.t)
    check(acc)
    assert torch.equal(acc.t, w8.debug_gemm_i32(q8, Wq))



def test_linear_dual_both_containers(w8):
    N, K = 136, 528
    Ms = (131, 70)
    ops = [gemm_operands(M, N, K, 40 + 10 * i) for i, M in enumerate(Ms)]
    Ys = [Guarded((M, N), torch.bfloat16) for M in Ms]
    w8.linear_dual_f16codes([(o[0], o[3], o[2], o[4], o[5], w8.chunk_plan(o[2]), o[6]) for o in ops],
                            Ys=[y.t for y in Ys])
    check(*Ys)
    Y8 = [Guarded((M, N), torch.bfloat16) for M in Ms]
    w8.linear_dual([(o[1], o[3], o[2], o[4], o[5]) for o in ops], Ys=[y.t for y in Y8])
    check(*Y8)
    for i in range(2):
        assert torch.equal(Ys[i].t, Y8[i].t)


def test_linear_bf16(w8):
    M, N, K = 131, 136, 528
    X = bf(wl.random_bf16((M, K), seed=50))
    W = bf(wl.random_bf16((N, K), seed=51, scale=0.05))
    b = t(wl.random_f32((N,), seed=52, scale=0.01))
    Y = Guarded((M, N), torch.bfloat16)
    w8.linear_bf16(X, W, b, Y=Y.t)
    check(Y)
    assert torch.equal(Y.t, w8.linear_bf16(X, W, b))


@pytest.mark.parametrize("fmt", [0, 1], ids=["q8_0", "q4_k"])
def test_linear_gguf_and_dequant(w8, fmt):
    M, N, K = 131, 136, 512
    X = bf(wl.random_bf16((M, K), seed=60))
    raw = t(wl.random_gguf(fmt, N, K, seed=61 + fmt))
    b = t(wl.random_f32((N,), seed=63, scale=0.01))
    Y = Guarded((M, N), torch.bfloat16)
    w8.linear_gguf(X, raw, fmt, N, b, Y=Y.t)
    check(Y)
    W = Guarded((N, K), torch.bfloat16)
    w8.debug_gguf_dequant(raw, fmt, N, K, W=W.t)
    check(W)
    assert torch.equal(Y.t, w8.linear_bf16(X, W.t, b))


def test_gelu_and_per_tensor_quant(w8):
    M, K = 131, 528
    H = bf(wl.ffn_preactivation(M, K, seed=70))
    lam = t(wl.random_uniform_f32((K,), seed=71, lo=0.25, hi=4.0))
    q, s = Guarded((M, K), torch.int8), Guarded((M,), torch.float32)
    w8.gelu_quant_act(H, lam, Xq=q.t, x_scale=s.t)
    check(q, s)
    q2, s2, a2 = Guarded((M, K), torch.int8), Guarded((M,), torch.float32), Guarded((1,), torch.float32)
    w8.quant_act_per_tensor(H, lam, Xq=q2.t, x_scale=s2.t, amax=a2.t)
    check(q2, s2, a2)


def test_act_stats_and_chunk_plan(w8):
    T, K = 131, 528
    X = bf(wl.random_bf16((T, K), seed=80, scale=2.0))
    sums, amax = Guarded((4, K), torch.float64, zero=True), Guarded((K,), torch.float32, zero=True)
    w8.act_stats_update(X, sums.t, amax.t)
    check(sums, amax)
    chan, tensor = Guarded((4, K), torch.float32), Guarded((4,), torch.float32)
    w8.act_stats_finalize(sums.t, amax.t, T, chan=chan.t, tensor=tensor.t)
    check(chan, tensor)
    Wq = t(wl.random_int8((136, 5000 - 5000 % 16), seed=81))
    plan = Guarded((w8.chunk_plan_size(*Wq.shape),), torch.int32)
    w8.chunk_plan(Wq, plan=plan.t)
    check(plan)
    assert torch.equal(plan.t, w8.chunk_plan(Wq))
