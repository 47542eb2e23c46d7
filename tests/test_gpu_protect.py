"""GPU parity of the pieces around the W8A8 layer, through the C ABI.

- Per-tensor activation quantization (naive arm of the activation-quant
  ablation, Sec. 5 "What drives INT8 recovery"): codes, scales and the tensor
  max bit-exact against the oracle.
- Activation statistics (Sec. 3, "Activation-fragility profiling and
  protection"): the accumulated power sums within their stated rounding
  bound of the oracle's binary64 sums, max-abs exact, the finalized
  mean / std / kurtosis within a relative 1e-4 (derived below).
- Protected bf16 layer: every output within half a bf16 ulp of the exact
  value plus the fp32 accumulation bound, and on average within 0.35 ulp.
- Per-layer dispatch: each path bitwise equal to the call it dispatches to.
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


def bf(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(DEV)


def t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def u16(x):
    return x.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def f32_of_bf16(h):
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def bf16_bits_of(x):
    return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).view(torch.int16) \
        .numpy().view(np.uint16)


# --------------------------------------------------- per-tensor activation scale

@pytest.mark.parametrize("M,K", [(1, 16), (257, 528), (64, 16384 + 16), (1031, 4096)])
@pytest.mark.parametrize("smooth", [True, False])
def test_quant_act_per_tensor_exact(w8, oracle_mod, M, K, smooth):
    X = wl.random_bf16((M, K), seed=M + 3 * K, scale=2.0)
    X[M // 2, K // 3] = bf16_bits_of([300.0])[0]          # one outlier sets the scale
    lam = wl.random_uniform_f32((K,), seed=K, lo=0.25, hi=4.0) if smooth else None
    q, sx, amax = w8.quant_act_per_tensor(bf(X), t(lam) if smooth else None)
    wq, wsx, wamax = oracle_mod.quant_act_per_tensor(X, lam)
    np.testing.assert_array_equal(q.cpu().numpy(), wq)
    np.testing.assert_array_equal(sx.cpu().numpy(), wsx)
    assert amax.item() == wamax


def test_quant_act_per_tensor_zero_and_qkv(w8, oracle_mod):
    Z = np.zeros((33, 64), np.uint16)
    q, sx, amax = w8.quant_act_per_tensor(bf(Z))
    assert amax.item() == 0.0 and not q.any().item() and not sx.any().item()
    case = wl.workload_cases("qkv_m4608_k4096_n12288")[0]
    lam = oracle_mod.smooth_scales(oracle_mod.channel_absmax(case.X_cal), case.W[0], case.alpha)
    q, sx, amax = w8.quant_act_per_tensor(bf(case.X[0]), t(lam))
    wq, wsx, wamax = oracle_mod.quant_act_per_tensor(case.X[0], lam)
    np.testing.assert_array_equal(q.cpu().numpy(), wq)
    np.testing.assert_array_equal(sx.cpu().numpy(), wsx)
    assert amax.item() == wamax


# ------------------------------------------------------------ statistics

# Each GPU power sum is within (2 * 64 + 12) * 2^-24 = 8.3e-6 of sum |x - c|^p
# (fp32 groups of at most 64 rows, at most 64 groups summed in fp32, a block's
# 8 warps added in fp32, fp64 beyond); 1e-5 leaves margin for the fp64 adds.
SUM_REL = 1e-5


def _stats_gpu(w8, chunks, K, shift):
    sums = torch.zeros(4, K, dtype=torch.float64, device=DEV)
    absmax = torch.zeros(K, dtype=torch.float32, device=DEV)
    sh = t(shift) if shift is not None else None
    for X in chunks:
        w8.act_stats_update(bf(X), sums, absmax, shift=sh)
    count = sum(x.shape[0] for x in chunks)
    chan, tensor = w8.act_stats_finalize(sums, absmax, count, shift=sh)
    return sums.cpu().numpy(), absmax.cpu().numpy(), chan.cpu().numpy(), tensor.cpu().numpy()


def _check_stats(oracle_mod, X, shift, sums, absmax, chan, tensor):
    S, A = oracle_mod.shifted_power_sums(X, shift)
    assert np.all(np.abs(sums - S) <= SUM_REL * A + 1e-30), np.max(np.abs(sums - S) / (A + 1e-30))
    wc, wt = oracle_mod.act_stats(X)
    np.testing.assert_array_equal(absmax, wc[0].astype(np.float32))
    # mean: the error of S1 / n is at most SUM_REL * mean|x - c|
    mean_tol = SUM_REL * A[0] / X.shape[0] + 1e-7 * np.abs(wc[1])
    assert np.all(np.abs(chan[1] - wc[1]) <= mean_tol + 1e-30)
    # std and kurtosis: relative 1e-4 where the variance is not tiny against
    # the squared distance to the shift (these inputs keep it above 1e-2)
    np.testing.assert_allclose(chan[2], wc[2], rtol=1e-4, atol=0)
    np.testing.assert_allclose(chan[3], wc[3], rtol=1e-4, atol=1e-6)
    assert tensor[0] == np.float32(wt[0])
    np.testing.assert_allclose(tensor[1:], wt[1:], rtol=1e-4, atol=1e-5 * wt[2])


@pytest.mark.parametrize("T,K", [(1, 16), (300, 528), (1000, 4096), (129, 16384 + 32)])
def test_act_stats(w8, oracle_mod, T, K):
    X = wl.random_bf16((T, K), seed=T + K, scale=1.5)
    x = f32_of_bf16(X)
    x[:, 1] += 5.0                       # large mean, taken out by the shift
    x[:, 2] = 0.75                       # a constant channel
    if T > 1:
        x[T // 2, 7] = 200.0             # an outlier token
    X = bf16_bits_of(x)
    shift = np.zeros(K, np.float32)
    shift[1] = 5.0
    got = _stats_gpu(w8, [X], K, shift)
    if T == 1:
        # one token: mean = x, std 0 and kurtosis 0 everywhere
        assert np.all(got[2][2] == 0) and np.all(got[2][3] == 0)
        np.testing.assert_allclose(got[2][1], f32_of_bf16(X)[0], rtol=1e-6, atol=1e-6)
        return
    _check_stats(oracle_mod, X, shift, *got)
    assert got[2][2][2] == 0.0 and got[2][3][2] == 0.0     # constant channel


def test_act_stats_accumulate_over_calls(w8, oracle_mod):
    # statistics recorded over several batches (the denoising trajectory)
    # equal those of the batches stacked
    K = 1024
    chunks = [wl.random_bf16((n, K), seed=50 + n, scale=1.0 + 0.3 * i)
              for i, n in enumerate((100, 1, 257))]
    got = _stats_gpu(w8, chunks, K, None)
    _check_stats(oracle_mod, np.concatenate(chunks), None, *got)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["qkv_m4608_k4096_n12288", "ffn_down_m4608_k16384_n4096"])
def test_act_stats_workloads(w8, oracle_mod, name):
    # the QKV input (outlier channels) and the FFN down-projection input (GELU
    # of a heavy-tailed pre-activation), full size
    case = wl.workload_cases(name)[0]
    X = case.X[0]
    got = _stats_gpu(w8, [X], X.shape[1], None)
    _check_stats(oracle_mod, X, None, *got)


# ------------------------------------------------------ protected bf16 layer

def _check_bf16_linear(Y_u16, y_exact, y_abs, K):
    """Y = bf16(fp32 sum + b): within half a bf16 ulp of the exact value plus the
    fp32 accumulation error (at most K/16 + 16 tensor-core accumulator adds of
    relative 2^-22 each, over sum |x w| + |b|), and on average within 0.35 ulp."""
    got = f32_of_bf16(Y_u16).astype(np.float64)
    mag = np.maximum(np.abs(got), np.abs(y_exact))
    ulp = np.exp2(np.floor(np.log2(np.maximum(mag, 2.0 ** -126))) - 7)
    acc_err = (K / 16 + 16) * 2.0 ** -22 * y_abs
    err = np.abs(got - y_exact)
    bad = err > 0.5 * ulp + acc_err + 2.0 ** -133
    assert not bad.any(), f"{bad.sum()} outputs outside the bound, worst {np.max(err / (0.5 * ulp + acc_err))}"
    assert np.mean(err / ulp) < 0.35


@pytest.mark.parametrize("M,N,K", [(1, 8, 16), (300, 264, 528), (257, 520, 1040), (64, 256, 16384 + 64)])
@pytest.mark.parametrize("with_bias", [True, False])
def test_linear_bf16(w8, oracle_mod, M, N, K, with_bias):
    X = wl.random_bf16((M, K), seed=M + K, scale=1.0)
    W = wl.random_bf16((N, K), seed=N + K, scale=0.05)
    b = wl.random_f32((N,), seed=N, scale=0.1) if with_bias else None
    Y = w8.linear_bf16(bf(X), bf(W), t(b) if with_bias else None)
    y, ya = oracle_mod.linear_bf16(X, W, b)
    _check_bf16_linear(u16(Y), y, ya, K)


@pytest.mark.slow
def test_linear_bf16_qkv_sampled_rows(w8, oracle_mod):
    case = wl.workload_cases("qkv_m4608_k4096_n12288")[0]
    X = case.X[0]
    Wb = bf16_bits_of(case.W[0])
    Y = w8.linear_bf16(bf(X), bf(Wb), t(case.bias[0]))
    Yh = u16(Y)
    rows = [0, 1, 255, 256, 2047, 4095, 4350, 4607]
    for r in rows:
        y, ya = oracle_mod.linear_bf16(X, Wb, case.bias[0], rows=(r, r + 1))
        _check_bf16_linear(Yh[r:r + 1], y, ya, X.shape[1])


def test_linear_bf16_empty_and_identity(w8):
    X = torch.zeros(0, 64, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(16, 64, dtype=torch.bfloat16, device=DEV)
    assert w8.linear_bf16(X, W).shape == (0, 16)
    # identity weights reproduce X exactly (one nonzero product per output)
    Xr = torch.randn(300, 256, device=DEV).to(torch.bfloat16)
    eye = torch.eye(256, device=DEV).to(torch.bfloat16)
    assert torch.equal(w8.linear_bf16(Xr, eye), Xr)


# ------------------------------------------------------------- dispatch

def test_layer_forward_dispatch(w8, oracle_mod):
    case = wl.workload_cases("single_m256_k512_n512")[0]
    M, K = case.X[0].shape
    N = case.W[0].shape[0]
    X = bf(case.X[0])
    s = w8.channel_absmax(bf(case.X_cal))
    W = t(case.W[0])
    lam = w8.smooth_scales(s, W, case.alpha)
    Wq, sw = w8.quantize_weights(W, lam)
    Wb = W.to(torch.bfloat16)
    bias = t(case.bias[0])
    Yq = w8.layer_forward(X, False, N, K, smooth=lam, Wq=Wq, w_scale=sw, bias=bias)
    Xq, sx = w8.quant_act(X, lam)
    assert torch.equal(Yq, w8.linear(Xq, sx, Wq, sw, bias))
    Yp = w8.layer_forward(X, True, N, K, W_bf16=Wb, bias=bias)
    assert torch.equal(Yp, w8.linear_bf16(X, Wb, bias))
    # with a workspace: fp16 codes written into it, the weights-in-TMEM GEMM
    ws = w8.linear_workspace(M, K)
    for plan in (None, w8.chunk_plan(Wq)):
        Yw = w8.layer_forward(X, False, N, K, smooth=lam, Wq=Wq, w_scale=sw, bias=bias, plan=plan, workspace=ws)
        assert torch.equal(Yw, Yq)
    # and against the oracle: the W8A8 path bit-exact
    lam_h = oracle_mod.smooth_scales(oracle_mod.channel_absmax(case.X_cal), case.W[0], case.alpha)
    Wq_h, sw_h = oracle_mod.quantize_weights(case.W[0], lam_h)
    want = oracle_mod.layer_forward(case.X[0], {"protect": False, "smooth": lam_h, "Wq": Wq_h,
                                                "w_scale": sw_h, "W_bf16": None,
                                                "bias": case.bias[0]})
    np.testing.assert_array_equal(u16(Yq), want)


def test_layer_forward_workspace_long_k(w8):
    # K > 16384: int8 codes, then the expansion pass in the workspace
    M, N, K = 300, 264, 16400
    g = torch.Generator(device=DEV).manual_seed(8)
    X = torch.randn(M, K, generator=g, device=DEV).to(torch.bfloat16)
    W = torch.randn(N, K, generator=g, device=DEV) * 0.02
    lam = torch.rand(K, generator=g, device=DEV) + 0.5
    Wq, sw = w8.quantize_weights(W, lam)
    bias = torch.randn(N, generator=g, device=DEV) * 0.01
    Y0 = w8.layer_forward(X, False, N, K, smooth=lam, Wq=Wq, w_scale=sw, bias=bias)
    Y1 = w8.layer_forward(X, False, N, K, smooth=lam, Wq=Wq, w_scale=sw, bias=bias, plan=w8.chunk_plan(Wq),
                          workspace=w8.linear_workspace(M, K))
    assert torch.equal(Y0, Y1)
    assert w8.device_status() == 0
