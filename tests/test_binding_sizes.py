"""The Python binding refuses buffers too small for the call before anything
reaches the library (the C ABI takes plain pointers and cannot check sizes).

Every check runs before the binding turns tensors into device pointers, so
host (CPU) tensors exercise it here: buffers of the right size get as far as
the device-pointer check (TypeError: not a CUDA tensor), and one element less
in any of them is a ValueError.
"""

import pytest
import torch

from paper_2606_12280_gb300 import _build

M, N, K = 5, 16, 32
f32, bf16, i8, f16, i32, f64, u8 = (torch.float32, torch.bfloat16, torch.int8, torch.float16, torch.int32,
                                    torch.float64, torch.uint8)


@pytest.fixture(scope="module")
def w8():
    _build.build()
    from paper_2606_12280_gb300 import w8a8
    w8a8.lib()
    return w8a8


def e(n, dt):
    return torch.zeros(n, dtype=dt)


def cases(w8):
    P = w8.chunk_plan_size(N, K)
    LW, GW = w8.linear_workspace_size(M, K), w8.gemm_workspace_size()
    # the split-K area is sized by the device's SM count: 0 bytes without a GPU
    gw = {"workspace": (GW, u8)} if GW > 0 else {}
    G0, G1 = N * (K // 32) * 34, N * (256 // 256) * 144
    X, W, Xq, Wq, X16 = e((M, K), bf16), e((N, K), f32), e((M, K), i8), e((N, K), i8), e((M, K), f16)
    # (function, positional args, {sized keyword: (numel, dtype)})
    return [
        (w8.channel_absmax, (X,), {"s": (K, f32)}),
        (w8.smooth_scales, (e(K, f32), W, 0.5), {"smooth": (K, f32)}),
        (w8.quantize_weights, (W,), {"smooth": (K, f32), "Wq": (N * K, i8), "w_scale": (N, f32)}),
        (w8.quant_act, (X,), {"smooth": (K, f32), "Xq": (M * K, i8), "x_scale": (M, f32)}),
        (w8.linear, (Xq, e(M, f32), Wq, e(N, f32)), {"bias": (N, f32), "Y": (M * N, bf16)}),
        (w8.linear, (Xq, e(M, f32), Wq, e(N, f32)), {"Y": (M * N, bf16), "plan": (P, i32), "workspace": (LW, u8)}),
        (w8.debug_gemm_i32, (Xq, Wq), {"acc": (M * N, i32)}),
        (w8.debug_gemm_i32, (Xq, Wq), {"acc": (M * N, i32), "workspace": (LW, u8)}),
        (w8.gelu_quant_act, (X,), {"smooth": (K, f32), "Xq": (M * K, i8), "x_scale": (M, f32)}),
        (w8.quant_act_f16codes, (X,), {"smooth": (K, f32), "Xq16": (M * K, f16), "x_scale": (M, f32),
                                       "sumsq": (M, i32)}),
        (w8.linear_f16codes, (X16, e(M, f32), Wq, e(N, f32)), {"bias": (N, f32), "Y": (M * N, bf16),
                                                             "plan": (P, i32), "x_sumsq": (M, i32), **gw}),
        (w8.debug_gemm_f16codes_i32, (X16, Wq), {"plan": (P, i32), "x_sumsq": (M, i32), "acc": (M * N, i32),
                                                 **gw}),
        (w8.chunk_plan, (Wq,), {"plan": (P, i32)}),
        (w8.linear_gguf, (e((M, K), bf16), e(G0, u8), 0, N), {"bias": (N, f32), "Y": (M * N, bf16)}),
        (w8.linear_gguf, (e((M, 256), bf16), e(G1, u8), 1, N), {"Y": (M * N, bf16)}),
        (w8.debug_gguf_dequant, (e(G0, u8), 0, N, K), {"W": (N * K, bf16)}),
        (w8.debug_gelu, (e(7, bf16),), {"G": (7, f32)}),
        (w8.quant_act_per_tensor, (X,), {"smooth": (K, f32), "Xq": (M * K, i8), "x_scale": (M, f32),
                                         "amax": (1, f32)}),
        (w8.act_stats_finalize, (e((4, K), f64), e(K, f32), M), {"shift": (K, f32), "chan": (4 * K, f32),
                                                                 "tensor": (4, f32)}),
        (w8.act_stats_noalloc, (X,), {"shift": (K, f32), "chan": (4 * K, f32), "tensor": (4, f32)}),
        (w8.linear_bf16, (X, e((N, K), bf16)), {"bias": (N, f32), "Y": (M * N, bf16)}),
        (w8.layer_forward, (X, False, N, K), {"smooth": (K, f32), "Wq": (N * K, i8), "w_scale": (N, f32),
                                              "bias": (N, f32), "Xq_work": (M * K, i8),
                                              "x_scale_work": (M, f32), "Y": (M * N, bf16)}),
        (w8.layer_forward, (X, True, N, K), {"W_bf16": (N * K, bf16), "bias": (N, f32), "Y": (M * N, bf16)}),
        (w8.layer_forward, (X, False, N, K), {"smooth": (K, f32), "Wq": (N * K, i8), "w_scale": (N, f32),
                                              "x_scale_work": (M, f32), "Y": (M * N, bf16), "plan": (P, i32),
                                              "workspace": (LW, u8)}),
        (w8.quantized_linear_forward, (X, e(K, f32), Wq, e(N, f32)), {"workspace": (LW, u8)}),
    ]


def test_right_sizes_pass_the_checks(w8):
    for fn, args, sized in cases(w8):
        kw = {k: e(n, dt) for k, (n, dt) in sized.items()}
        with pytest.raises(TypeError, match="CUDA tensor"):
            fn(*args, **kw)


def test_one_element_short_is_refused(w8):
    for fn, args, sized in cases(w8):
        for short in sized:
            kw = {k: e(n - (1 if k == short else 0), dt) for k, (n, dt) in sized.items()}
            with pytest.raises(ValueError, match=short):
                fn(*args, **kw)


def test_inputs_sized_too(w8):
    with pytest.raises(ValueError, match="act_absmax"):
        w8.smooth_scales(e(K - 1, f32), e((N, K), f32), 0.5)
    with pytest.raises(ValueError, match="Wraw"):
        w8.linear_gguf(e((M, K), bf16), e(N * 34 - 1, u8), 0, N)
    with pytest.raises(ValueError, match="sums"):
        w8.act_stats_update(e((M, K), bf16), e(4 * K - 1, f64), e(K, f32))


def test_weights_match_the_activations(w8):
    """A weight matrix narrower than the activations' K would be read past
    its end: every GEMM entry refuses it."""
    Xq, X16, short = e((M, K), i8), e((M, K), f16), e((N, K - 16), i8)
    for call in (lambda: w8.linear(Xq, e(M, f32), short, e(N, f32)),
                 lambda: w8.debug_gemm_i32(Xq, short),
                 lambda: w8.linear_f16codes(X16, e(M, f32), short, e(N, f32)),
                 lambda: w8.debug_gemm_f16codes_i32(X16, short)):
        with pytest.raises(ValueError, match="Wq"):
            call()


def test_statistics_planes_exact_shape(w8):
    """The library addresses the four power-sum planes at stride K: a wider
    accumulator (enough elements, wrong stride) is refused, and so is an
    absmax longer than the batch's K."""
    X = e((M, K), bf16)
    with pytest.raises(ValueError, match="sums"):
        w8.act_stats_update(X, e((4, 2 * K), f64), e(K, f32))
    with pytest.raises(ValueError, match="absmax"):
        w8.act_stats_update(X, e((4, K), f64), e(2 * K, f32))
    with pytest.raises(ValueError, match="sums"):
        w8.act_stats_finalize(e((4, 2 * K), f64), e(K, f32), M)


def test_layer_forward_checks_x(w8):
    with pytest.raises(ValueError, match="X has shape"):
        w8.layer_forward(e((M, K - 16), bf16), False, N, K)


def test_dual_branches_sized(w8):
    Xq, Wq = e((M, K), i8), e((N, K), i8)
    good = (Xq, e(M, f32), Wq, e(N, f32), e(N, f32))
    bad = (Xq, e(M - 1, f32), Wq, e(N, f32), e(N, f32))
    with pytest.raises(TypeError, match="CUDA tensor"):
        w8.linear_dual([good, good], Ys=[e(M * N, bf16), e(M * N, bf16)])
    # (a branch is checked before its pointers are taken; the library is
    # called only after both, so the short one is put first here, where host
    # tensors stop at the first pointer)
    with pytest.raises(ValueError, match="x_scale"):
        w8.linear_dual([bad, good])
    with pytest.raises(ValueError, match="Y"):
        w8.linear_dual([good, good], Ys=[e(M * N - 1, bf16), e(M * N, bf16)])
    X = e((M, K), bf16)
    with pytest.raises(ValueError, match="sumsq"):
        w8.quant_act_dual_f16codes([(X, None), (X, None)],
                                   out=[(e(M * K, f16), e(M, f32), e(M - 1, i32)), (e(M * K, f16), e(M, f32), e(M, i32))])
