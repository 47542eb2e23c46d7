"""GPU parity of the layer with activation codes in a 16-bit container.

`w8a8_quant_act_f16codes` writes the same integer codes as `w8a8_quant_act`
as fp16 values; `w8a8_linear_f16codes` computes the same exact INT32 product
and epilogue from them.  Bar: codes and scales bit-exact against the oracle,
outputs bit-exact against the oracle and bitwise equal to the int8-container
path.
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


def codes(Xq16):
    q = Xq16.float().cpu().numpy()
    assert np.all(q == np.rint(q)) and np.all(np.abs(q) <= 127)
    return q.astype(np.int8)


@pytest.mark.parametrize("M,K", [(1, 16), (1000, 272), (300, 528), (77, 2064), (257, 4096), (40, 4112),
                                 (64, 16384)])
def test_quant_act_f16codes_exact(w8, oracle_mod, M, K):
    X = wl.random_bf16((M, K), seed=M + K, scale=2.0)
    X[0, :] = 0                                         # an all-zero token
    lam = wl.random_uniform_f32((K,), seed=K, lo=0.25, hi=4.0)
    q16, sx = w8.quant_act_f16codes(bf(X), t(lam))
    wq, wsx = oracle_mod.quant_act(X, lam)
    np.testing.assert_array_equal(codes(q16), wq)
    np.testing.assert_array_equal(sx.cpu().numpy(), wsx)
    q8, sx8 = w8.quant_act(bf(X), t(lam))
    assert torch.equal(q16.to(torch.int8), q8) and torch.equal(sx, sx8)


def test_quant_act_f16codes_gelu_matches_int8_gelu(w8):
    H = wl.ffn_preactivation(129, 16384, seed=5)
    lam = wl.random_uniform_f32((16384,), seed=6, lo=0.25, hi=4.0)
    q16, sx = w8.quant_act_f16codes(bf(H), t(lam), gelu=True)
    q8, sx8 = w8.gelu_quant_act(bf(H), t(lam))
    assert torch.equal(q16.to(torch.int8), q8) and torch.equal(sx, sx8)


@pytest.mark.parametrize("M,N,K", [(1, 8, 16), (300, 264, 528), (513, 520, 1040), (64, 256, 16384)])
@pytest.mark.parametrize("with_bias", [True, False])
@pytest.mark.parametrize("with_plan", [True, False])
def test_linear_f16codes_exact(w8, oracle_mod, M, N, K, with_bias, with_plan):
    c = wl.make_case(M, K, N, seed=M + N + K)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    b = c.bias[0] if with_bias else None
    q16, sx = w8.quant_act_f16codes(bf(c.X[0]), t(lam))
    plan = w8.chunk_plan(t(Wq)) if with_plan else None
    Y = w8.linear_f16codes(q16, sx, t(Wq), t(sw), t(b) if with_bias else None, plan=plan)
    Xq, wsx = oracle_mod.quant_act(c.X[0], lam)
    np.testing.assert_array_equal(u16(Y), oracle_mod.linear(Xq, wsx, Wq, sw, b))
    Y8 = w8.linear(q16.to(torch.int8), sx, t(Wq), t(sw), t(b) if with_bias else None)
    assert torch.equal(Y, Y8)


def test_linear_f16codes_extremes(w8, oracle_mod):
    # all codes +-127 at the longest K the int32 chunks see in practice
    M, N, K = 256, 256, 16384
    rng = np.random.default_rng(7)
    Xq = np.where(rng.random((M, K)) < 0.5, -127, 127).astype(np.int8)
    Wq = np.where(rng.random((N, K)) < 0.5, -127, 127).astype(np.int8)
    Xq[0] = 127
    Wq[0] = 127
    sx = np.full(M, 1e-3, np.float32)
    sw = np.full(N, 1e-3, np.float32)
    q16 = torch.from_numpy(Xq.astype(np.float16)).to(DEV)
    Y = w8.linear_f16codes(q16, t(sx), t(Wq), t(sw))
    np.testing.assert_array_equal(u16(Y), oracle_mod.linear(Xq, sx, Wq, sw, None))


@pytest.mark.slow
def test_linear_f16codes_qkv_sampled_rows(w8, oracle_mod):
    case = wl.workload_cases("qkv_m4608_k4096_n12288")[0]
    s = oracle_mod.channel_absmax(case.X_cal)
    lam = oracle_mod.smooth_scales(s, case.W[0], case.alpha)
    Wq, sw = oracle_mod.quantize_weights(case.W[0], lam)
    q16, sx = w8.quant_act_f16codes(bf(case.X[0]), t(lam))
    Y = u16(w8.linear_f16codes(q16, sx, t(Wq), t(sw), t(case.bias[0]), plan=w8.chunk_plan(t(Wq))))
    Xq, wsx = oracle_mod.quant_act(case.X[0], lam)
    np.testing.assert_array_equal(codes(q16), Xq)
    for r in [0, 1, 255, 256, 2047, 4095, 4350, 4607]:
        np.testing.assert_array_equal(Y[r:r + 1], oracle_mod.linear(Xq, wsx, Wq, sw, case.bias[0],
                                                                     rows=(r, r + 1)))


# ------------------------------------------------------------------ drain plan

def plan_reference(Wq, limit=1 << 17, kc=1024, rows=256):
    """The drain plan restated: per block of `rows` weight rows, a run of K
    chunks ends before chunk c when some row's sum |w| over the run including
    c would exceed `limit` (then 128 * limit = 2^24 bounds every partial sum of
    codes |a| <= 128); the last chunk always ends a run.  Bit c of a block's
    words = a run ends after chunk c; the block's last word = the largest
    sum of squares of its rows."""
    N, K = Wq.shape
    nc = -(-K // kc)
    words = -(-nc // 32)
    nb = -(-N // rows)
    a = np.abs(Wq.astype(np.int64))
    l1 = np.stack([a[:, c * kc:(c + 1) * kc].sum(1) for c in range(nc)], 1)
    plan = np.zeros((nb, words + 1), np.uint32)
    sq = (Wq.astype(np.int64) ** 2).sum(1)
    for b in range(nb):
        blk = l1[b * rows:(b + 1) * rows]
        cur = np.zeros(blk.shape[0], np.int64)
        for c in range(nc):
            cand = cur + blk[:, c]
            if cand.max() > limit:
                plan[b, (c - 1) // 32] |= np.uint32(1 << ((c - 1) % 32))
                cur = blk[:, c].copy()
            else:
                cur = cand
        plan[b, (nc - 1) // 32] |= np.uint32(1 << ((nc - 1) % 32))
        plan[b, words] = np.uint32(sq[b * rows:(b + 1) * rows].max())
    return plan.reshape(-1)


def gauss_codes(shape, seed, sigma):
    rng = np.random.default_rng(seed)
    return np.clip(np.rint(rng.normal(0, sigma, shape)), -127, 127).astype(np.int8)


def plan_cases():
    rng = np.random.default_rng(11)
    small = gauss_codes((520, 3 * 1024 + 320), 1, 20.0)             # runs merge
    uni = rng.integers(-127, 128, (296, 5 * 1024), dtype=np.int8)    # pairs of chunks
    full = np.full((256, 4096), 127, np.int8)                       # a drain after every chunk
    mixed = np.concatenate([gauss_codes((256, 8192), 2, 12.0), np.full((200, 8192), -127, np.int8)])
    many = gauss_codes((296, 40 * 1024), 3, 8.0)                    # two plan words per block
    return {"small": small, "uniform": uni, "full": full, "mixed": mixed, "many": many}


@pytest.mark.parametrize("name", ["small", "uniform", "full", "mixed", "many"])
def test_chunk_plan_matches_reference(w8, name):
    Wq = plan_cases()[name]
    plan = w8.chunk_plan(t(Wq)).cpu().numpy().view(np.uint32)
    assert plan.size == w8.chunk_plan_size(*Wq.shape)
    np.testing.assert_array_equal(plan, plan_reference(Wq))


def test_chunk_plan_reference_needs_drains_where_fp32_would_round():
    # (host check of the plan's premise) the all-max block: a single fp32 run
    # over two chunks of positive products passes 2^24 and rounds, so the
    # plan must end a run after every chunk there
    Wq = plan_cases()["full"]
    assert plan_reference(Wq)[0] == np.uint32(0b1111)
    prod = np.full(2048, 127 * 127, np.float32)
    prod[1::3] = 127 * 125
    acc = np.float32(0)
    for v in prod:
        acc = np.float32(acc + v)
    assert int(acc) != int(prod.astype(np.int64).sum())


@pytest.mark.parametrize("name", ["small", "uniform", "full", "mixed"])
@pytest.mark.parametrize("with_plan", [True, False])
def test_gemm_f16codes_i32_exact(w8, name, with_plan):
    Wq = plan_cases()[name]
    N, K = Wq.shape
    M = 300
    rng = np.random.default_rng(N + K)
    Xq = rng.integers(-127, 128, (M, K), dtype=np.int8)
    if name in ("full", "mixed"):
        # products of one sign and near the maximum: partial sums near 2^24
        Xq = np.where(rng.random((M, K)) < 0.3, 125, 127).astype(np.int8)
        if name == "mixed":
            Xq[:150] = -Xq[:150]
    q16 = torch.from_numpy(Xq.astype(np.float16)).to(DEV)
    plan = w8.chunk_plan(t(Wq)) if with_plan else None
    acc = w8.debug_gemm_f16codes_i32(q16, t(Wq), plan=plan).cpu().numpy()
    want = Xq.astype(np.int64) @ Wq.astype(np.int64).T
    np.testing.assert_array_equal(acc, want)


# ------------------------------------------------------- token sums of squares

@pytest.mark.parametrize("M,K,gelu", [(1, 16, False), (300, 528, False), (257, 4096, False),
                                      (64, 16384, False), (129, 4096, True)])
def test_quant_act_f16codes_sumsq_exact(w8, M, K, gelu):
    X = wl.random_bf16((M, K), seed=M + 3 * K, scale=2.0)
    X[0, :] = 0                                         # an all-zero token
    lam = wl.random_uniform_f32((K,), seed=K + 1, lo=0.25, hi=4.0)
    ss = torch.empty(M, dtype=torch.int32, device=DEV)
    q16, sx = w8.quant_act_f16codes(bf(X), t(lam), gelu=gelu, sumsq=ss)
    q = codes(q16).astype(np.int64)
    np.testing.assert_array_equal(ss.cpu().numpy().view(np.uint32), (q * q).sum(1).astype(np.uint32))
    q16b, sxb = w8.quant_act_f16codes(bf(X), t(lam), gelu=gelu)
    assert torch.equal(q16, q16b) and torch.equal(sx, sxb)


def sumsq_cases():
    rng = np.random.default_rng(23)
    # 1: Gaussian codes and weights: every tile one run (bound holds)
    W1 = gauss_codes((520, 4096), 5, 30.0)
    X1 = gauss_codes((600, 4096), 6, 30.0)
    # 2: near-max codes in the second token block: those tiles fall back to
    # the plan (the bound fails), the first block's tiles run as one
    W2 = gauss_codes((264, 8192), 7, 40.0)
    X2 = gauss_codes((520, 8192), 8, 20.0)
    X2[256:] = np.where(rng.random((264, 8192)) < 0.5, -127, 127)
    # 3: worst case everywhere
    W3 = np.full((256, 3072), 127, np.int8)
    X3 = np.where(rng.random((300, 3072)) < 0.3, 125, 127).astype(np.int8)
    return {"single": (X1, W1), "mixed": (X2, W2), "worst": (X3, W3)}


@pytest.mark.parametrize("name", ["single", "mixed", "worst"])
def test_gemm_f16codes_i32_exact_with_sumsq(w8, name):
    Xq, Wq = sumsq_cases()[name]
    q16 = torch.from_numpy(Xq.astype(np.float16)).to(DEV)
    ss = torch.from_numpy(((Xq.astype(np.int64) ** 2).sum(1)).astype(np.uint32).view(np.int32)).to(DEV)
    plan = w8.chunk_plan(t(Wq))
    acc = w8.debug_gemm_f16codes_i32(q16, t(Wq), plan=plan, x_sumsq=ss).cpu().numpy()
    np.testing.assert_array_equal(acc, Xq.astype(np.int64) @ Wq.astype(np.int64).T)


def test_single_run_bound_premise():
    # (host check) the cases above exercise both sides of the bound
    X1, W1 = sumsq_cases()["single"]
    a = (X1.astype(np.int64) ** 2).sum(1).max()
    w = (W1.astype(np.int64) ** 2).sum(1).max()
    assert a * w <= 2 ** 48
    X2, W2 = sumsq_cases()["mixed"]
    w = (W2.astype(np.int64) ** 2).sum(1).max()
    assert (X2[:256].astype(np.int64) ** 2).sum(1).max() * w <= 2 ** 48
    assert (X2[256:].astype(np.int64) ** 2).sum(1).max() * w > 2 ** 48


@pytest.mark.parametrize("M,N,K", [(300, 264, 528), (513, 520, 4096)])
def test_linear_f16codes_exact_with_sumsq(w8, oracle_mod, M, N, K):
    c = wl.make_case(M, K, N, seed=M + N + 2 * K)
    s = oracle_mod.channel_absmax(c.X_cal)
    lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
    Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
    ss = torch.empty(M, dtype=torch.int32, device=DEV)
    q16, sx = w8.quant_act_f16codes(bf(c.X[0]), t(lam), sumsq=ss)
    Y = w8.linear_f16codes(q16, sx, t(Wq), t(sw), t(c.bias[0]), plan=w8.chunk_plan(t(Wq)), x_sumsq=ss)
    Xq, wsx = oracle_mod.quant_act(c.X[0], lam)
    np.testing.assert_array_equal(u16(Y), oracle_mod.linear(Xq, wsx, Wq, sw, c.bias[0]))


# ------------------------------------------------------------- dual branches

@pytest.mark.parametrize("M0,M1", [(300, 130), (0, 257), (513, 0), (256, 256), (2000, 800)])
def test_dual_f16codes_equals_singles(w8, oracle_mod, M0, M1):
    N, K = 520, 1040
    cs = [wl.make_case(max(M, 1), K, N, seed=M + 7 * b) for b, M in enumerate((M0, M1))]
    branches_q, branches_g, singles = [], [], []
    for b, (c, M) in enumerate(zip(cs, (M0, M1))):
        s = oracle_mod.channel_absmax(c.X_cal)
        lam = oracle_mod.smooth_scales(s, c.W[0], c.alpha)
        Wq, sw = oracle_mod.quantize_weights(c.W[0], lam)
        X = c.X[0][:M]
        branches_q.append((bf(X) if M else torch.empty(0, K, dtype=torch.bfloat16, device=DEV), t(lam)))
        branches_g.append((t(Wq), t(sw), t(c.bias[0]), w8.chunk_plan(t(Wq))))
        singles.append((X, lam, Wq, sw, c.bias[0]))
    q = w8.quant_act_dual_f16codes(branches_q)
    Ys = w8.linear_dual_f16codes([(q[b][0], q[b][1], *branches_g[b][:3], branches_g[b][3], q[b][2])
                                  for b in range(2)])
    for b, (X, lam, Wq, sw, bias) in enumerate(singles):
        M = X.shape[0]
        if M == 0:
            assert Ys[b].shape[0] == 0
            continue
        ss = torch.empty(M, dtype=torch.int32, device=DEV)
        q16, sx = w8.quant_act_f16codes(bf(X), t(lam), sumsq=ss)
        assert torch.equal(q16, q[b][0]) and torch.equal(sx, q[b][1]) and torch.equal(ss, q[b][2])
        Y1 = w8.linear_f16codes(q16, sx, t(Wq), t(sw), t(bias), plan=branches_g[b][3], x_sumsq=ss)
        assert torch.equal(Y1, Ys[b])
        Xq, wsx = oracle_mod.quant_act(X, lam)
        np.testing.assert_array_equal(u16(Ys[b]), oracle_mod.linear(Xq, wsx, Wq, sw, bias))


@pytest.mark.parametrize("case", ["inf_scale", "huge_scale", "nan_bias", "finite"])
def test_epilogue_non_finite_scales(w8, oracle_mod, case):
    # The epilogue rounds pairs with one conversion instruction only where no
    # output can be a NaN; tiles with a non-finite scale or bias, or a token
    # scale above 2^96 (acc * sx may overflow), take the integer rounding.
    # Either way Y matches the oracle: bit for bit where it is a number, and
    # NaN where the oracle's is NaN.
    M, N, K = 300, 520, 1040
    rng = np.random.default_rng(7)
    Xq = rng.integers(-127, 128, (M, K), dtype=np.int8)
    Wq = rng.integers(-127, 128, (N, K), dtype=np.int8)
    Xq[5] = 0                                             # acc = 0 rows: inf * 0 = NaN
    sx = rng.random(M, dtype=np.float32) * 1e-3
    sw = rng.random(N, dtype=np.float32) * 1e-3
    b = rng.standard_normal(N).astype(np.float32)
    if case == "inf_scale":
        sx[[3, 5, 260]] = np.inf
        sw[[7, 300]] = 0.0
    elif case == "huge_scale":
        sx[[4, 270]] = np.float32(2.0 ** 120)             # acc * sx overflows to inf
        sw[[9, 400]] = 0.0                                # inf * 0 = NaN
    elif case == "nan_bias":
        b[[11, 500]] = np.nan
    q16 = t(Xq.astype(np.float16))
    want = oracle_mod.linear(Xq, sx, Wq, sw, b)
    nan_w = (want & 0x7fff) > 0x7f80
    # the fp16-code engine and the int8-code engine without a workspace
    for Y in (u16(w8.linear_f16codes(q16, t(sx), t(Wq), t(sw), t(b))),
              u16(w8.linear(t(Xq), t(sx), t(Wq), t(sw), t(b)))):
        nan_g = (Y & 0x7fff) > 0x7f80
        np.testing.assert_array_equal(nan_g, nan_w)
        np.testing.assert_array_equal(Y[~nan_g], want[~nan_w])
    if case != "finite":
        assert nan_w.any()
