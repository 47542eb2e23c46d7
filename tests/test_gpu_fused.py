"""GPU parity of a3 fused with its neighbours, through the C ABI.

- Dual-branch activation quantization in one launch: each branch bit-exact
  against the oracle's per-branch quantization (and the single-branch call).
- GELU folded into the quantization of the FFN down-projection input: the
  GPU's GELU (a table of the binary64 GELU rounded once to fp32 at every
  bf16 input) is checked exhaustively against the oracle's, bit for bit, and
  the fused pass's codes and scales are bit-exact against the oracle.
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


def f32_of_bf16(h):
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# ------------------------------------------------------------- dual branch

@pytest.mark.parametrize("M0,M1,K", [(300, 257, 528), (0, 64, 1040), (64, 0, 1040), (1, 1, 16),
                                     (129, 77, 4096), (40, 33, 16384), (9, 5, 16384 + 16)])
def test_quant_act_dual_exact(w8, oracle_mod, M0, M1, K):
    X0 = wl.random_bf16((M0, K), seed=M0 + K, scale=2.0)
    X1 = wl.random_bf16((M1, K), seed=M1 + 2 * K, scale=0.5)
    l0 = wl.random_uniform_f32((K,), seed=K, lo=0.25, hi=4.0)
    out = w8.quant_act_dual([(bf(X0), t(l0)), (bf(X1), None)])
    want = oracle_mod.quant_act_dual([(X0, l0), (X1, None)])
    for (q, s), (wq, ws) in zip(out, want):
        np.testing.assert_array_equal(q.cpu().numpy(), wq)
        np.testing.assert_array_equal(s.cpu().numpy(), ws)


def test_quant_act_dual_workload(w8, oracle_mod):
    # the dual-branch workload: both branches' inputs, each with its own lambda
    case = wl.workload_cases("dual_m4608_k4096_n4096")[0]
    s = oracle_mod.channel_absmax(case.X_cal)
    lams = [oracle_mod.smooth_scales(s, case.W[i], case.alpha) for i in range(2)]
    out = w8.quant_act_dual([(bf(case.X[i]), t(lams[i])) for i in range(2)])
    for i in range(2):
        wq, ws = oracle_mod.quant_act(case.X[i], lams[i])
        np.testing.assert_array_equal(out[i][0].cpu().numpy(), wq)
        np.testing.assert_array_equal(out[i][1].cpu().numpy(), ws)
        q1, s1 = w8.quant_act(bf(case.X[i]), t(lams[i]))
        assert torch.equal(q1, out[i][0]) and torch.equal(s1, out[i][1])


# ---------------------------------------------------------------- GELU

def test_gelu_values_every_bf16(w8, oracle_mod):
    """The fused pass's GELU equals the oracle's (binary64, rounded once) at
    every finite bf16 input, bit for bit: the table is exact, and its
    binary64 erfc (the device's) and the oracle's (the host C library's) are
    independent implementations."""
    h = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    hv = f32_of_bf16(h)
    h = h[np.isfinite(hv)]
    hv = hv[np.isfinite(hv)]
    g = w8.debug_gelu(bf(h)).cpu().numpy()
    want = oracle_mod.gelu_value(hv)
    np.testing.assert_array_equal(g.view(np.uint32), want.view(np.uint32))


def _check_gelu_quant(q, sx, wq, wsx):
    np.testing.assert_array_equal(sx, wsx)
    np.testing.assert_array_equal(q, wq)


@pytest.mark.parametrize("M,K", [(1, 16), (300, 528), (257, 4096), (64, 16384), (33, 16384 + 16)])
@pytest.mark.parametrize("smooth", [True, False])
def test_gelu_quant_act(w8, oracle_mod, M, K, smooth):
    H = wl.ffn_preactivation(M, K, seed=M + K)
    lam = wl.random_uniform_f32((K,), seed=K + 1, lo=0.25, hi=4.0) if smooth else None
    q, sx = w8.gelu_quant_act(bf(H), t(lam) if smooth else None)
    wq, wsx = oracle_mod.gelu_quant_act(H, lam)
    _check_gelu_quant(q.cpu().numpy(), sx.cpu().numpy(), wq, wsx)


def test_gelu_quant_act_edges(w8, oracle_mod):
    # zero rows, large positive values (GELU is the identity there), large
    # negative values (GELU underflows towards 0 but stays nonzero)
    K = 64
    h = np.zeros((4, K), np.float32)
    h[1] = np.linspace(6.0, 60.0, K)
    h[2] = -np.linspace(3.0, 9.0, K)
    h[3, ::2] = 1.5
    H = torch.from_numpy(h).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    q, sx = w8.gelu_quant_act(bf(H))
    wq, wsx = oracle_mod.gelu_quant_act(H, None)
    _check_gelu_quant(q.cpu().numpy(), sx.cpu().numpy(), wq, wsx)
    assert sx[0].item() == 0.0 and not q[0].any().item()
    # where GELU is the identity the fused pass is the plain pass
    q1, s1 = w8.quant_act(bf(H[1:2]))
    assert torch.equal(q1[0], q[1]) and s1[0].item() == sx[1].item()


@pytest.mark.slow
def test_gelu_quant_act_ffn_down_full(w8, oracle_mod):
    # the FFN down-projection input at full size: 4608 tokens x 16384 channels
    M, K = 4608, 16384
    H = wl.ffn_preactivation(M, K, seed=2)
    lam = wl.random_uniform_f32((K,), seed=3, lo=0.25, hi=4.0)
    q, sx = w8.gelu_quant_act(bf(H), t(lam))
    wq, wsx = oracle_mod.gelu_quant_act(H, lam)
    _check_gelu_quant(q.cpu().numpy(), sx.cpu().numpy(), wq, wsx)
