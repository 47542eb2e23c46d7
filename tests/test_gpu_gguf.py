"""GPU parity of the GGUF weight-only layer (Sec. 3, "GGUF k-quants"), through
the C ABI.

- Decoding: the bf16 weights decoded from Q8_0 and Q4_K blocks bit-exact
  against the oracle's decoder.
- The layer: every output within half a bf16 ulp of the exact value plus the
  fp32 accumulation bound (as for the protected bf16 layer), and bitwise equal
  to the bf16 layer run on the decoded weights (same tensor-core K order).
"""

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = "cuda"
FMTS = [0, 1]
FMT_IDS = ["q8_0", "q4_k"]


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


def check_linear(Y_u16, y_exact, y_abs, K):
    got = f32_of_bf16(Y_u16).astype(np.float64)
    mag = np.maximum(np.abs(got), np.abs(y_exact))
    ulp = np.exp2(np.floor(np.log2(np.maximum(mag, 2.0 ** -126))) - 7)
    acc_err = (K / 16 + 16) * 2.0 ** -22 * y_abs
    err = np.abs(got - y_exact)
    assert not np.any(err > 0.5 * ulp + acc_err + 2.0 ** -133)
    assert np.mean(err / ulp) < 0.35


@pytest.mark.parametrize("fmt", FMTS, ids=FMT_IDS)
@pytest.mark.parametrize("N,K", [(8, 256), (264, 1024), (128, 4096), (16, 16384)])
def test_gguf_dequant_exact(w8, oracle_mod, fmt, N, K):
    raw = wl.random_gguf(fmt, N, K, seed=N + K + fmt)
    got = u16(w8.debug_gguf_dequant(t(raw), fmt, N, K))
    np.testing.assert_array_equal(got, oracle_mod.gguf_dequant_bf16(raw, fmt, N, K))


@pytest.mark.parametrize("fmt", FMTS, ids=FMT_IDS)
@pytest.mark.parametrize("M,N,K", [(1, 8, 256), (300, 264, 512), (257, 520, 1024), (64, 256, 16384)])
@pytest.mark.parametrize("with_bias", [True, False])
def test_linear_gguf(w8, oracle_mod, fmt, M, N, K, with_bias):
    X = wl.random_bf16((M, K), seed=M + K, scale=1.0)
    raw = wl.random_gguf(fmt, N, K, seed=N + 3 * K + fmt)
    b = wl.random_f32((N,), seed=N, scale=0.1) if with_bias else None
    Y = w8.linear_gguf(bf(X), t(raw), fmt, N, t(b) if with_bias else None)
    y, ya = oracle_mod.linear_gguf(X, raw, fmt, N, b)
    check_linear(u16(Y), y, ya, K)
    # the same tensor-core accumulation as the bf16 layer on the decoded weights
    Wd = w8.debug_gguf_dequant(t(raw), fmt, N, K)
    assert torch.equal(Y, w8.linear_bf16(bf(X), Wd, t(b) if with_bias else None))


def test_linear_gguf_empty(w8):
    X = torch.zeros(0, 256, dtype=torch.bfloat16, device=DEV)
    raw = torch.zeros(8, 144, dtype=torch.uint8, device=DEV)
    assert w8.linear_gguf(X, raw, 1, 8).shape == (0, 8)


@pytest.mark.slow
@pytest.mark.parametrize("fmt", FMTS, ids=FMT_IDS)
def test_linear_gguf_qkv_sampled_rows(w8, oracle_mod, fmt):
    # the QKV projection at full size: 4608 tokens, 4096 -> 12288
    case = wl.workload_cases("qkv_m4608_k4096_n12288")[0]
    X = case.X[0]
    M, K = X.shape
    N = 12288
    raw = wl.random_gguf(fmt, N, K, seed=11 + fmt)
    Y = u16(w8.linear_gguf(bf(X), t(raw), fmt, N, t(case.bias[0])))
    Wb = oracle_mod.gguf_dequant_bf16(raw, fmt, N, K)
    for r in [0, 1, 255, 256, 2047, 4095, 4350, 4607]:
        y, ya = oracle_mod.linear_bf16(X, Wb, case.bias[0], rows=(r, r + 1))
        check_linear(Y[r:r + 1], y, ya, K)
