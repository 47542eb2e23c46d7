"""Full-size parity on every benchmark workload, in the launch configuration
bench.py uses: the whole layer (calibration statistic, smoothing vector,
weight quantization, activation quantization, INT8 GEMM with fused epilogue,
the dual-branch launch where the workload has two branches) runs on the GPU
through the C ABI and is compared with the CPU oracle.  The fp16-code path
(the benchmarked one: codes as fp16 values with their token sums of squares,
the weights' drain plan, single or dual-branch launches) runs beside it and
must give the same codes and bitwise the same outputs.

lambda, Wq, w_scale, Xq and x_scale are compared in full (bit-exact); the bf16
output is compared on sampled rows (first, last and seeded random rows), which
the oracle computes one by one, within 1 bf16 ulp (and in practice exactly).
The FFN workloads also report the error of the W8A8 output against an fp32
GEMM of the unquantized operands, as information.
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


def u16(x):
    return x.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def sample_rows(M, n=12, seed=0):
    g = np.random.default_rng(seed)
    rows = {0, M - 1, M // 2}
    rows.update(int(r) for r in g.integers(0, M, n))
    return sorted(rows)


def run_case(w8, oracle_mod, case, info=False):
    M, K = case.X[0].shape
    N = case.W[0].shape[0]
    nb = len(case.X)
    s = w8.channel_absmax(bf(case.X_cal))
    s_ref = oracle_mod.channel_absmax(case.X_cal)
    np.testing.assert_array_equal(s.cpu().numpy(), s_ref)
    branches, refs = [], []
    for i in range(nb):
        W = torch.from_numpy(case.W[i]).to(DEV)
        b = torch.from_numpy(case.bias[i]).to(DEV)
        lam = w8.smooth_scales(s, W, case.alpha)
        Wq, sw = w8.quantize_weights(W, lam)
        Xq, sx = w8.quant_act(bf(case.X[i]), lam)
        lam_ref = oracle_mod.smooth_scales(s_ref, case.W[i], case.alpha)
        np.testing.assert_array_equal(lam.cpu().numpy(), lam_ref)
        Wq_ref, sw_ref = oracle_mod.quantize_weights(case.W[i], lam_ref)
        np.testing.assert_array_equal(sw.cpu().numpy(), sw_ref)
        np.testing.assert_array_equal(Wq.cpu().numpy(), Wq_ref)
        del W
        Xq_ref, sx_ref = oracle_mod.quant_act(case.X[i], lam_ref)
        np.testing.assert_array_equal(sx.cpu().numpy(), sx_ref)
        np.testing.assert_array_equal(Xq.cpu().numpy(), Xq_ref)
        branches.append((Xq, sx, Wq, sw, b))
        refs.append((Xq_ref, sx_ref, Wq_ref, sw_ref, case.bias[i]))
    if nb == 2:
        Ys = w8.linear_dual(branches)
    else:
        Ys = [w8.linear(*branches[0])]
    # the fp16-code path on the same layer
    lams = [w8.smooth_scales(s, torch.from_numpy(case.W[i]).to(DEV), case.alpha) for i in range(nb)]
    plans = [w8.chunk_plan(branches[i][2]) for i in range(nb)]
    if nb == 2:
        q = w8.quant_act_dual_f16codes([(bf(case.X[i]), lams[i]) for i in range(2)])
        Y16 = w8.linear_dual_f16codes([(q[i][0], q[i][1], branches[i][2], branches[i][3], branches[i][4],
                                        plans[i], q[i][2]) for i in range(2)])
    else:
        ss = torch.empty(M, dtype=torch.int32, device=DEV)
        q16, sx16 = w8.quant_act_f16codes(bf(case.X[0]), lams[0], sumsq=ss)
        q = [(q16, sx16, ss)]
        Y16 = [w8.linear_f16codes(q16, sx16, branches[0][2], branches[0][3], branches[0][4],
                                  plan=plans[0], x_sumsq=ss)]
    torch.cuda.synchronize()
    assert w8.device_status() == 0
    for i in range(nb):
        Xq_ref = refs[i][0]
        assert torch.equal(q[i][0].to(torch.int8), branches[i][0])
        assert torch.equal(q[i][1], branches[i][1])
        np.testing.assert_array_equal(q[i][2].cpu().numpy().view(np.uint32),
                                      (Xq_ref.astype(np.int64) ** 2).sum(1).astype(np.uint32))
        assert torch.equal(Y16[i], Ys[i]), f"branch {i}: fp16-code path differs"
    del Y16, q
    rows = sample_rows(M)
    for i in range(nb):
        got = u16(Ys[i])[rows]
        Xq_ref, sx_ref, Wq_ref, sw_ref, b_ref = refs[i]
        want = np.concatenate([oracle_mod.linear(Xq_ref, sx_ref, Wq_ref, sw_ref, b_ref,
                                                 rows=(r, r + 1)) for r in rows])
        diff = np.abs(got.astype(np.int32) - want.astype(np.int32))
        assert diff.max() <= 1, f"branch {i}: {diff.max()} bf16 ulp"
        np.testing.assert_array_equal(got, want)
        if info:
            x = (case.X[i][rows].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            ref = x @ case.W[i].astype(np.float64).T + case.bias[i][None, :]
            y = (got.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            rel = np.linalg.norm(y - ref) / np.linalg.norm(ref)
            print(f"[info] {case.shape.name} branch {i}: W8A8 vs fp64 GEMM relative "
                  f"Frobenius error {rel:.4f}, max abs {np.abs(y - ref).max():.4f}")
    return Ys


@pytest.mark.parametrize("name", ["single_m256_k512_n512", "qkv_m4608_k4096_n12288",
                                  "ffn_up_m4608_k4096_n16384", "ffn_down_m4608_k16384_n4096",
                                  "dual_m4608_k4096_n4096"])
def test_workload(w8, oracle_mod, name):
    for case in wl.workload_cases(name):
        run_case(w8, oracle_mod, case, info=name.startswith("ffn"))


@pytest.mark.slow
@pytest.mark.parametrize("name", ["block_m1280", "block_m4608", "block_m16896"])
def test_block_sweep(w8, oracle_mod, name):
    for sh in wl.WORKLOADS[name].linears:
        case = wl.workload_cases(name, only=sh.name)[0]
        run_case(w8, oracle_mod, case)
        del case
