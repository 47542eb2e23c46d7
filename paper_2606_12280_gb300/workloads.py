"""Seeded synthetic inputs shaped like the DiT linears of the paper's workloads.

This module only draws random numbers: it holds none of the quantization
method's arithmetic, so both the CPU oracle and the CUDA path can consume its
outputs.  The model weights and prompts the paper used (Ideogram 4.0, gated)
are not available; these seeded tensors stand in for them.

Recipe (one CPU ``torch.Generator`` per workload, draws in this fixed order):
  1. outlier channel set: ``randperm(K)[:n_out]`` with ``n_out = max(1, round(p*K))``;
  2. calibration activations, 256 tokens;
  3. activations X, one tensor per branch;
  4. weights W ~ N(0, 0.02) fp32, one [N, K] matrix per branch;
  5. bias b ~ N(0, 0.01) fp32, one per branch.
Activations are N(0, 1) fp32 with the outlier channels multiplied by a factor,
then cast to bf16.  The FFN down-projection input is GELU(Z) in fp32 (exact erf
form) cast to bf16, where Z is N(0, 1) except on 1% of the channels, which draw
a Student-t with 3 degrees of freedom (heavy tails).

Token counts follow a 1024x1024 image at 64x64 latent patches plus text
tokens (4096 + 512 = 4608), the DiT hidden size 4096, QKV 12288 and FFN 16384.
"""

from __future__ import annotations

import dataclasses

import numpy as np
import torch

CALIB_TOKENS = 256
ALPHA = 0.5


@dataclasses.dataclass(frozen=True)
class LinearShape:
    name: str
    M: int
    K: int
    N: int


@dataclasses.dataclass(frozen=True)
class Workload:
    """One benchmark configuration: a list of linears run with one seed."""
    name: str
    seed: int
    linears: tuple[LinearShape, ...]
    branches: int = 1
    outlier_frac: float = 0.005
    outlier_mult: float = 20.0
    act: str = "gauss"               # "gauss" or "gelu_t" (FFN down input)


def _block(M: int) -> tuple[LinearShape, ...]:
    return (LinearShape(f"qkv_m{M}", M, 4096, 12288),
            LinearShape(f"out_m{M}", M, 4096, 4096),
            LinearShape(f"up_m{M}", M, 4096, 16384),
            LinearShape(f"down_m{M}", M, 16384, 4096))


WORKLOADS: dict[str, Workload] = {
    # a single small linear, 1% outlier channels x30, seed 0
    "single_m256_k512_n512": Workload(
        "single_m256_k512_n512", 0, (LinearShape("single", 256, 512, 512),),
        outlier_frac=0.01, outlier_mult=30.0),
    # DiT attention QKV projection at 4608 tokens, seed 1
    "qkv_m4608_k4096_n12288": Workload(
        "qkv_m4608_k4096_n12288", 1, (LinearShape("qkv", 4608, 4096, 12288),)),
    # FFN pair at 4608 tokens: up 4096 -> 16384, down 16384 -> 4096, seed 2
    "ffn_up_m4608_k4096_n16384": Workload(
        "ffn_up_m4608_k4096_n16384", 2, (LinearShape("up", 4608, 4096, 16384),)),
    "ffn_down_m4608_k16384_n4096": Workload(
        "ffn_down_m4608_k16384_n4096", 2, (LinearShape("down", 4608, 16384, 4096),),
        outlier_frac=0.01, act="gelu_t"),
    # dual-branch (conditional, unconditional) grouped launch, seed 3
    "dual_m4608_k4096_n4096": Workload(
        "dual_m4608_k4096_n4096", 3, (LinearShape("dual", 4608, 4096, 4096),),
        branches=2),
    # one DiT block's quantized linears, both branches, three token counts, seed 4
    "block_m1280": Workload("block_m1280", 4, _block(1280), branches=2),
    "block_m4608": Workload("block_m4608", 4, _block(4608), branches=2),
    "block_m16896": Workload("block_m16896", 4, _block(16896), branches=2),
}


def n_outliers(K: int, frac: float) -> int:
    return max(1, int(round(frac * K)))


def _bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _activations(g: torch.Generator, M: int, K: int, outliers: torch.Tensor,
                 mult: float, act: str) -> np.ndarray:
    if act == "gauss":
        x = torch.randn(M, K, generator=g, dtype=torch.float32)
        x[:, outliers] *= mult
        return _bf16_bits(x)
    if act in ("gelu_t", "heavy_t"):
        z = torch.randn(M, K, generator=g, dtype=torch.float32)
        # Student-t(3) on the outlier channels: z / sqrt(chi2_3 / 3)
        n = outliers.numel()
        zt = torch.randn(M, n, generator=g, dtype=torch.float32)
        chi2 = (torch.randn(M, n, 3, generator=g, dtype=torch.float32) ** 2).sum(-1)
        z[:, outliers] = zt / torch.sqrt(chi2 / 3.0)
        # "heavy_t" is the pre-activation itself (the up-projection output
        # that the GELU-fused quantization reads); "gelu_t" is the FFN
        # down-projection input built from it outside the method
        return _bf16_bits(z if act == "heavy_t" else torch.nn.functional.gelu(z))
    raise ValueError(act)


def ffn_preactivation(M: int, K: int, seed: int, frac: float = 0.01) -> np.ndarray:
    """Stand-in for the FFN up-projection output [M, K] bf16: N(0, 1) with a
    Student-t(3) on max(1, round(frac*K)) channels (outlier set drawn first)."""
    g = torch.Generator().manual_seed(seed)
    outliers = torch.randperm(K, generator=g)[:n_outliers(K, frac)]
    return _activations(g, M, K, outliers, 1.0, "heavy_t")


@dataclasses.dataclass
class LinearCase:
    """Inputs of one quantized linear: bf16 arrays are uint16 bit patterns."""
    shape: LinearShape
    X_cal: np.ndarray                  # [256, K] bf16 calibration batch
    X: list[np.ndarray]                # per branch [M, K] bf16
    W: list[np.ndarray]                # per branch [N, K] fp32
    bias: list[np.ndarray]             # per branch [N] fp32
    alpha: float = ALPHA


def make_case(M: int, K: int, N: int, seed: int, *, branches: int = 1,
              outlier_frac: float = 0.005, outlier_mult: float = 20.0,
              act: str = "gauss", name: str = "case",
              calib_tokens: int = CALIB_TOKENS) -> LinearCase:
    """Draw one linear's inputs in the fixed order given in the module doc."""
    g = torch.Generator().manual_seed(seed)
    outliers = torch.randperm(K, generator=g)[:n_outliers(K, outlier_frac)]
    X_cal = _activations(g, calib_tokens, K, outliers, outlier_mult, act)
    X = [_activations(g, M, K, outliers, outlier_mult, act) for _ in range(branches)]
    W = [(torch.randn(N, K, generator=g, dtype=torch.float32) * 0.02).numpy()
         for _ in range(branches)]
    bias = [(torch.randn(N, generator=g, dtype=torch.float32) * 0.01).numpy()
            for _ in range(branches)]
    return LinearCase(LinearShape(name, M, K, N), X_cal, X, W, bias)


def workload_cases(name: str, only: str | None = None) -> list[LinearCase]:
    """All linears of a named workload; linear i of it draws with seed*1000+i
    (the first linear uses the workload seed itself)."""
    wl = WORKLOADS[name]
    out = []
    for i, sh in enumerate(wl.linears):
        if only is not None and sh.name != only:
            continue
        seed = wl.seed if i == 0 else wl.seed * 1000 + i
        out.append(make_case(sh.M, sh.K, sh.N, seed, branches=wl.branches,
                             outlier_frac=wl.outlier_frac,
                             outlier_mult=wl.outlier_mult, act=wl.act,
                             name=sh.name))
    return out


def random_int8(shape, seed: int, lo: int = -127, hi: int = 127) -> np.ndarray:
    """Uniform integers in [lo, hi] as int8 (for direct GEMM parity cases)."""
    g = torch.Generator().manual_seed(seed)
    return torch.randint(lo, hi + 1, tuple(shape), generator=g,
                         dtype=torch.int16).to(torch.int8).numpy()


def random_f32(shape, seed: int, scale: float = 1.0) -> np.ndarray:
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(tuple(shape), generator=g, dtype=torch.float32) * scale).numpy()


def random_uniform_f32(shape, seed: int, lo: float, hi: float) -> np.ndarray:
    """Uniform fp32 in [lo, hi) (positive smoothing vectors, shifts)."""
    g = torch.Generator().manual_seed(seed)
    return (torch.rand(tuple(shape), generator=g, dtype=torch.float32) * (hi - lo) + lo).numpy()


def random_bf16(shape, seed: int, scale: float = 1.0) -> np.ndarray:
    g = torch.Generator().manual_seed(seed)
    return _bf16_bits(torch.randn(tuple(shape), generator=g, dtype=torch.float32) * scale)


def random_gguf(fmt: int, N: int, K: int, seed: int) -> np.ndarray:
    """Random but well-formed GGUF weight blocks, uint8 [N, bytes per row]:
    fmt 0 = Q8_0 (fp16 d in [1e-4, 4e-3), int8 quants), fmt 1 = Q4_K (fp16 d
    and dmin in [1e-5, 4e-4), random 6-bit scale/min bytes, random 4-bit
    quants).  Only random draws: decoding is the method's business."""
    g = torch.Generator().manual_seed(seed)
    if fmt == 0:
        nb = K // 32
        d = (torch.rand(N, nb, generator=g) * 3.9e-3 + 1e-4).to(torch.float16)
        q = torch.randint(-127, 128, (N, nb, 32), generator=g, dtype=torch.int16).to(torch.int8)
        raw = np.empty((N, nb, 34), np.uint8)
        raw[..., 0:2] = d.view(torch.int16).numpy().view(np.uint8).reshape(N, nb, 2)
        raw[..., 2:] = q.numpy().view(np.uint8)
        return raw.reshape(N, nb * 34)
    nb = K // 256
    dd = (torch.rand(N, nb, 2, generator=g) * 3.9e-4 + 1e-5).to(torch.float16)
    rest = torch.randint(0, 256, (N, nb, 140), generator=g, dtype=torch.int16).to(torch.uint8)
    raw = np.empty((N, nb, 144), np.uint8)
    raw[..., 0:4] = dd.view(torch.int16).numpy().view(np.uint8).reshape(N, nb, 4)
    raw[..., 4:] = rest.numpy()
    return raw.reshape(N, nb * 144)
