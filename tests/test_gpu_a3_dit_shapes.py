"""GPU parity of a3 at the DiT's K = 4096 shapes and around them.

The codes and scales must equal the oracle's bit for bit in both code
containers, with the token sums of squares exact, at the full QKV input (4608
x 4096) and the 128 x 128-patch one (16896 x 4096), with fewer rows than SMs,
ragged K (a partial last chunk group), all-zero tokens, smoothing off, and
both branches in one launch with uneven token counts.
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


def inputs(M, K, seed, smooth=True):
    X = wl.random_bf16((M, K), seed=seed, scale=2.0)
    X[M // 3, :] = 0                                    # an all-zero token
    lam = wl.random_uniform_f32((K,), seed=seed + 1, lo=0.25, hi=4.0) if smooth else None
    return X, lam


@pytest.mark.parametrize("M,K", [(4608, 4096), (16896, 4096), (100, 4096), (1, 4096), (2000, 3072),
                                 (777, 2064), (153, 4080)])
@pytest.mark.parametrize("smooth", [True, False])
def test_codes_exact(w8, oracle_mod, M, K, smooth):
    X, lam = inputs(M, K, M + K, smooth)
    Xq_ref, sx_ref = oracle_mod.quant_act(X, lam)
    lam_d = t(lam) if smooth else None
    Xq, sx = w8.quant_act(bf(X), lam_d)
    np.testing.assert_array_equal(Xq.cpu().numpy(), Xq_ref)
    np.testing.assert_array_equal(sx.cpu().numpy(), sx_ref)
    ss = torch.empty(M, dtype=torch.int32, device=DEV)
    q16, sx16 = w8.quant_act_f16codes(bf(X), lam_d, sumsq=ss)
    assert torch.equal(q16.to(torch.int8), Xq) and torch.equal(sx16, sx)
    want_ss = (Xq_ref.astype(np.int64) ** 2).sum(1)
    np.testing.assert_array_equal(ss.cpu().numpy().astype(np.int64), want_ss)
    assert w8.device_status() == 0


@pytest.mark.parametrize("M0,M1", [(4608, 4608), (3000, 17), (0, 700), (250, 0)])
def test_dual_exact(w8, oracle_mod, M0, M1):
    K = 4096
    ins = [inputs(max(M, 1), K, 31 * i + M) for i, M in enumerate((M0, M1))]
    Xs = [bf(ins[i][0][:M]) for i, M in enumerate((M0, M1))]
    lams = [t(ins[i][1]) for i in range(2)]
    outs = w8.quant_act_dual([(Xs[i], lams[i]) for i in range(2)])
    outs16 = w8.quant_act_dual_f16codes([(Xs[i], lams[i]) for i in range(2)])
    for i, M in enumerate((M0, M1)):
        if M == 0:
            continue
        Xq_ref, sx_ref = oracle_mod.quant_act(ins[i][0][:M], ins[i][1])
        np.testing.assert_array_equal(outs[i][0].cpu().numpy(), Xq_ref)
        np.testing.assert_array_equal(outs[i][1].cpu().numpy(), sx_ref)
        assert torch.equal(outs16[i][0].to(torch.int8), outs[i][0])
        np.testing.assert_array_equal(outs16[i][2].cpu().numpy().astype(np.int64),
                                      (Xq_ref.astype(np.int64) ** 2).sum(1))
    assert w8.device_status() == 0
