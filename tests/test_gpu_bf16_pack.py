"""The GEMM epilogue's one-instruction bf16 rounding against the library's
integer rounding, for every fp32 input that is not a NaN.

The fp16-code GEMM rounds its outputs to bf16 with cvt.rn.bf16x2.f32 in tiles
that cannot hold a NaN and with integer operations (which reproduce the
oracle's rounding, pinned by every parity test) elsewhere; the two must give
the same bits for every other input.  The check runs on the device over all
2^32 patterns in both halves of the word (tests/cuda/bf16_pack_check.cu).
"""

import os
import shutil
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_pack_bf16x2_matches_integer_rounding(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sys.path.insert(0, ROOT)
    from paper_2606_12280_gb300 import _build
    nvcc = _build.nvcc()
    if not nvcc or not shutil.which(nvcc) and not os.path.exists(nvcc):
        pytest.skip("no nvcc")
    exe = tmp_path / "bf16_pack_check"
    src = os.path.join(ROOT, "tests", "cuda", "bf16_pack_check.cu")
    subprocess.run([nvcc, *_build.ARCH, "-O3", "-std=c++17", src, "-o", str(exe)], check=True,
                   capture_output=True, text=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "mismatches 0" in r.stdout
