"""Host-side checks of the C ABI that need no GPU.

The library must build for sm_103a, load, and export every symbol that
include/w8a8.h declares.  Argument validation runs on the host before any CUDA
call, so invalid calls are exercised here with fake (never dereferenced)
pointer values and must return their status codes without touching a device.
"""

import ctypes
import os
import re

import numpy as np
import pytest

from paper_2606_12280_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "w8a8.h")

OK, INVALID, SHAPE, MISALIGNED = 0, 1, 2, 3


@pytest.fixture(scope="module")
def L():
    _build.build()
    from paper_2606_12280_gb300 import w8a8
    return w8a8.lib()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"W8A8_API\s+[\w\s\*]*?\b(w8a8_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("w8a8_smooth_scales", "w8a8_quantize_weights", "w8a8_quant_act",
                     "w8a8_linear", "w8a8_linear_dual", "w8a8_debug_gemm_i32",
                     "w8a8_channel_absmax", "w8a8_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name


def test_binding_covers_every_symbol():
    from paper_2606_12280_gb300 import w8a8
    assert set(declared_functions()) == set(w8a8.SIGNATURES)


def test_status_strings(L):
    assert L.w8a8_status_string(0) == b"W8A8_OK"
    assert L.w8a8_status_string(5) == b"W8A8_ERR_TIMEOUT"
    assert L.w8a8_status_string(99) == b"W8A8_ERR_UNKNOWN"


A = 0x100000          # a fake, 16-byte aligned "device" address (never used)
U = A + 4             # a misaligned one


def test_quant_act_validation(L):
    f = L.w8a8_quant_act
    assert f(A, None, 4, 15, A, A, None) == SHAPE        # K % 16
    assert f(A, None, 4, 0, A, A, None) == SHAPE
    assert f(A, None, -1, 16, A, A, None) == SHAPE
    assert f(A, None, 4, 133152, A, A, None) == SHAPE    # K beyond the int32 bound
    assert f(None, None, 4, 16, A, A, None) == INVALID
    assert f(A, None, 4, 16, None, A, None) == INVALID
    assert f(A, None, 4, 16, A, None, None) == INVALID
    assert f(U, None, 4, 16, A, A, None) == MISALIGNED
    assert f(A, U, 4, 16, A, A, None) == MISALIGNED
    assert f(A, None, 0, 16, A, A, None) == OK            # empty batch: no-op


def test_weight_and_smooth_validation(L):
    q = L.w8a8_quantize_weights
    assert q(A, None, 12, 16, A, A, None) == SHAPE        # N % 8
    assert q(A, None, 8, 24, A, A, None) == SHAPE         # K % 16
    assert q(None, None, 8, 16, A, A, None) == INVALID
    assert q(A, None, 8, 16, U, A, None) == MISALIGNED
    sm = L.w8a8_smooth_scales
    assert sm(A, A, 8, 16, 1.5, A, None) == INVALID       # alpha outside [0, 1]
    assert sm(A, A, 8, 16, -0.1, A, None) == INVALID
    assert sm(A, A, 8, 16, float("nan"), A, None) == INVALID
    assert sm(None, A, 8, 16, 0.5, A, None) == INVALID
    assert sm(A, A, 8, 16, 0.5, U, None) == MISALIGNED
    ca = L.w8a8_channel_absmax
    assert ca(A, 4, 8, A, None) == SHAPE
    assert ca(A, 4, 16, None, None) == INVALID


def test_linear_validation(L):
    f = L.w8a8_linear
    assert f(A, A, A, A, None, 4, 12, 16, A, None, None, None) == SHAPE     # N % 8
    assert f(A, A, A, A, None, 4, 8, 24, A, None, None, None) == SHAPE      # K % 16
    assert f(A, A, A, A, None, -2, 8, 16, A, None, None, None) == SHAPE
    assert f(None, A, A, A, None, 4, 8, 16, A, None, None, None) == INVALID
    assert f(A, None, A, A, None, 4, 8, 16, A, None, None, None) == INVALID
    assert f(A, A, A, A, None, 4, 8, 16, None, None, None, None) == INVALID
    assert f(A, A, U, A, None, 4, 8, 16, A, None, None, None) == MISALIGNED
    assert f(A, A, A, A, U, 4, 8, 16, A, None, None, None) == MISALIGNED    # bias
    assert f(A, A, A, A, None, 4, 8, 16, A, None, U, None) == MISALIGNED    # workspace
    assert f(A, A, A, A, None, 4, 8, 16, A, U, A, None) == MISALIGNED       # plan, with a workspace
    assert f(A, A, A, A, None, 0, 8, 16, A, None, None, None) == OK          # empty batch
    assert f(A, A, A, A, None, 0, 8, 16, A, None, A, None) == OK
    g = L.w8a8_debug_gemm_i32
    assert g(A, A, 4, 8, 15, A, None, None, None) == SHAPE
    assert g(A, None, 4, 8, 16, A, None, None, None) == INVALID
    assert g(A, A, 4, 8, 16, A, None, U, None) == MISALIGNED


def test_linear_workspace_size(L):
    base = L.w8a8_gemm_workspace_size()
    assert L.w8a8_linear_workspace_size(4608, 4096) == base + 2 * 4608 * 4096 + 4 * 4608 + 1024
    assert L.w8a8_linear_workspace_size(0, 4096) == base + 1024
    assert L.w8a8_linear_workspace_size(-1, 4096) == 0
    assert L.w8a8_linear_workspace_size(16, 0) == 0


def test_dual_validation(L):
    from paper_2606_12280_gb300.w8a8 import Branch
    arr = (Branch * 2)()
    for i in range(2):
        arr[i] = Branch(A, A, A, A, None, A, 4, None)
    f = L.w8a8_linear_dual
    assert f(None, 8, 16, None, None) == INVALID
    assert f(arr, 12, 16, None, None) == SHAPE
    assert f(arr, 8, 16, U, None) == MISALIGNED           # workspace
    arr[1].chunk_plan = U
    assert f(arr, 8, 16, A, None) == MISALIGNED           # plan, with a workspace
    arr[1].chunk_plan = None
    arr[1].Wq = U
    assert f(arr, 8, 16, None, None) == MISALIGNED
    arr[1].Wq = None
    assert f(arr, 8, 16, None, None) == INVALID
    arr[0].M = 0
    arr[1] = Branch(None, None, None, None, None, None, 0, None)
    assert f(arr, 8, 16, None, None) == OK                # both branches empty


def test_debug_engine_validation(L):
    """The earlier engines are reached only through the test entry point,
    per call (no process-wide switch)."""
    from paper_2606_12280_gb300.w8a8 import Branch
    arr = (Branch * 2)()
    for i in range(2):
        arr[i] = Branch(A, A, A, A, None, A, 4, None)
    f = L.w8a8_debug_linear_engine
    assert f(3, arr, 1, 8, 16, 0, None) == INVALID        # no such engine
    assert f(-1, arr, 1, 8, 16, 0, None) == INVALID
    assert f(2, arr, 0, 8, 16, 0, None) == INVALID        # one or two branches
    assert f(2, arr, 3, 8, 16, 0, None) == INVALID
    assert f(2, None, 1, 8, 16, 0, None) == INVALID
    assert f(1, arr, 2, 12, 16, 0, None) == SHAPE
    arr[0].x_scale = None
    assert f(0, arr, 1, 8, 16, 0, None) == INVALID        # scales needed for the bf16 output
    arr[0].Y = U
    assert f(0, arr, 1, 8, 16, 1, None) == MISALIGNED     # int32 output: scales unused
    arr[0].M = 0
    assert f(0, arr, 1, 8, 16, 1, None) == OK
    assert not hasattr(L, "w8a8_set_gemm_engine")


def test_wait_probe_validation(L):
    assert L.w8a8_debug_wait_timeout(0, None) == INVALID
    assert L.w8a8_debug_wait_timeout(2000001, None) == INVALID


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    from paper_2606_12280_gb300 import w8a8
    monkeypatch.setattr(w8a8, "_lib", None)
    monkeypatch.setattr(w8a8, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        w8a8.lib()


def test_per_tensor_and_stats_validation(L):
    f = L.w8a8_quant_act_per_tensor
    assert f(A, None, 4, 16, A, A, None, None) == INVALID        # amax
    assert f(A, None, 4, 16, A, A, U, None) == MISALIGNED
    assert f(A, None, 4, 24, A, A, A, None) == SHAPE
    assert f(A, None, 0, 16, A, A, A, None) == OK                 # empty batch
    u = L.w8a8_act_stats_update
    assert u(A, 4, 16, None, None, A, None) == INVALID
    assert u(A, 4, 16, None, A, None, None) == INVALID
    assert u(A, 4, 15, None, A, A, None) == SHAPE
    assert u(A, 4, 16, U, A, A, None) == MISALIGNED              # shift
    assert u(None, 0, 16, None, A, A, None) == OK                # no tokens
    fin = L.w8a8_act_stats_finalize
    assert fin(A, A, None, 0, 16, A, A, None) == INVALID          # count
    assert fin(A, A, None, 5, 16, A, None, None) == INVALID
    assert fin(A, A, None, 5, 8, A, A, None) == SHAPE
    # chan may not overlap the inputs (it carries partial sums during the call)
    base = 1 << 20
    chan = ctypes.c_void_p(base)
    assert fin(ctypes.c_void_p(base + 4 * 16 * 4 - 16), ctypes.c_void_p(base + 4096), None, 5, 16,
               chan, A, None) == INVALID                          # sums
    assert fin(ctypes.c_void_p(base + 4096), ctypes.c_void_p(base + 16), None, 5, 16,
               chan, A, None) == INVALID                          # absmax
    assert fin(ctypes.c_void_p(base + 4096), ctypes.c_void_p(base + 8192), ctypes.c_void_p(base + 128),
               5, 16, chan, A, None) == INVALID                   # shift


def test_linear_bf16_and_layer_validation(L):
    from paper_2606_12280_gb300.w8a8 import Layer
    f = L.w8a8_linear_bf16
    assert f(A, A, None, 4, 12, 16, A, None) == SHAPE
    assert f(A, None, None, 4, 8, 16, A, None) == INVALID
    assert f(A, A, U, 4, 8, 16, A, None) == MISALIGNED
    assert f(None, None, None, 0, 8, 16, None, None) == OK       # empty batch
    g = L.w8a8_layer_forward
    assert g(None, A, 4, A, A, A, None, None) == INVALID
    prot = Layer(1, 8, 16, None, None, None, None, None, None)
    assert g(ctypes.byref(prot), A, 4, None, None, A, None, None) == INVALID   # no bf16 weights
    q = Layer(0, 8, 16, None, A, A, None, None, None)
    assert g(ctypes.byref(q), A, 4, None, A, A, None, None) == INVALID        # no codes buffer
    assert g(ctypes.byref(q), A, 4, A, None, A, A, None) == INVALID           # no scales
    assert g(ctypes.byref(q), A, 4, U, A, A, None, None) == MISALIGNED
    assert g(ctypes.byref(q), A, 4, None, A, A, U, None) == MISALIGNED        # workspace
    assert g(ctypes.byref(q), U, 4, None, A, A, A, None) == MISALIGNED        # X, fp16-code path
    assert g(ctypes.byref(q), None, 4, None, A, A, A, None) == INVALID
    qp = Layer(0, 8, 16, None, A, A, None, None, U)
    assert g(ctypes.byref(qp), A, 4, None, A, A, A, None) == MISALIGNED       # plan
    assert g(ctypes.byref(q), A, 0, None, None, A, None, None) == OK
    bad = Layer(0, 12, 16, None, A, A, None, None, None)
    assert g(ctypes.byref(bad), A, 4, A, A, A, None, None) == SHAPE


def test_select_protected():
    from paper_2606_12280_gb300 import w8a8
    _build.build()
    nan = float("nan")
    # the n largest scores, NaN first, ties to the lower index
    assert w8a8.select_protected([0.5, 3.0, 1.0, 3.0, 2.0], 2) == [0, 1, 0, 1, 0]
    assert w8a8.select_protected([0.5, 3.0, 1.0, 3.0, 2.0], 1) == [0, 1, 0, 0, 0]
    assert w8a8.select_protected([1.0, nan, 5.0], 1) == [0, 1, 0]
    assert w8a8.select_protected([1.0, nan, 5.0], 3) == [1, 1, 1]
    assert w8a8.select_protected([1.0, 2.0], 0) == [0, 0]
    assert w8a8.select_protected([], 0) == []
    # the paper's setting: 17 of 211 linears
    rng = np.random.default_rng(0)
    sc = rng.standard_normal(211).astype(np.float32)
    flags = w8a8.select_protected(list(sc), 17)
    assert sum(flags) == 17
    assert min(sc[np.array(flags) == 1]) > max(sc[np.array(flags) == 0])
    L = w8a8.lib()
    assert L.w8a8_select_protected(None, 3, 1, None) == INVALID
    arr = (ctypes.c_float * 2)(1.0, 2.0)
    out = (ctypes.c_int * 2)()
    assert L.w8a8_select_protected(arr, 2, 3, out) == INVALID
    assert L.w8a8_select_protected(arr, 2, -1, out) == INVALID


def test_fused_quant_validation(L):
    from paper_2606_12280_gb300.w8a8 import ActBranch
    arr = (ActBranch * 2)()
    for i in range(2):
        arr[i] = ActBranch(A, None, 4, A, A)
    f = L.w8a8_quant_act_dual
    assert f(None, 16, None) == INVALID
    assert f(arr, 24, None) == SHAPE
    arr[1].Xq = U
    assert f(arr, 16, None) == MISALIGNED
    arr[1].Xq = None
    assert f(arr, 16, None) == INVALID
    arr[0] = ActBranch(None, None, 0, None, None)
    arr[1] = ActBranch(None, None, 0, None, None)
    assert f(arr, 16, None) == OK                        # both branches empty
    g = L.w8a8_gelu_quant_act
    assert g(A, None, 4, 15, A, A, None) == SHAPE
    assert g(None, None, 4, 16, A, A, None) == INVALID
    assert g(A, U, 4, 16, A, A, None) == MISALIGNED
    assert g(None, None, 0, 16, None, None, None) == OK  # empty batch


def test_gguf_validation(L):
    f = L.w8a8_linear_gguf
    assert f(A, A, 2, None, 4, 8, 256, A, None) == INVALID          # format
    assert f(A, A, 1, None, 4, 8, 128, A, None) == SHAPE            # K % 256
    assert f(A, A, 0, None, 4, 12, 256, A, None) == SHAPE           # N % 8
    assert f(A, None, 1, None, 4, 8, 256, A, None) == INVALID
    assert f(A, U, 1, None, 4, 8, 256, A, None) == MISALIGNED
    assert f(A, A, 1, U, 4, 8, 256, A, None) == MISALIGNED          # bias
    assert f(None, A, 1, None, 0, 8, 256, None, None) == OK        # empty batch
    g = L.w8a8_debug_gguf_dequant
    assert g(A, 1, 8, 256, None, None) == INVALID
    assert g(A, 0, 8, 256, U, None) == MISALIGNED


def test_f16codes_validation(L):
    f = L.w8a8_quant_act_f16codes
    assert f(A, None, 4, 16400, A, A, None, 0, None) == SHAPE         # K beyond 16384
    assert f(A, None, 4, 24, A, A, None, 0, None) == SHAPE
    assert f(None, None, 4, 16, A, A, None, 0, None) == INVALID
    assert f(A, None, 4, 16, U, A, None, 0, None) == MISALIGNED
    assert f(A, None, 4, 16, A, A, U, 0, None) == MISALIGNED          # sumsq
    assert f(None, None, 0, 16, None, None, None, 0, None) == OK
    g = L.w8a8_linear_f16codes
    assert g(A, A, A, A, None, 4, 12, 16, None, None, A, None, None) == SHAPE
    assert g(None, A, A, A, None, 4, 8, 16, None, None, A, None, None) == INVALID
    assert g(A, A, U, A, None, 4, 8, 16, None, None, A, None, None) == MISALIGNED
    assert g(A, A, A, A, None, 4, 8, 16, U, None, A, None, None) == MISALIGNED      # plan
    assert g(A, A, A, A, None, 4, 8, 16, A, U, A, None, None) == MISALIGNED         # token sums
    assert g(A, A, A, A, None, 0, 8, 16, None, None, A, None, None) == OK
    assert g(A, A, A, A, None, 4, 8, 16, None, None, A, U, None) == MISALIGNED   # workspace
    d = L.w8a8_debug_gemm_f16codes_i32
    assert d(A, A, 4, 12, 16, None, None, A, None, None) == SHAPE
    assert d(None, A, 4, 8, 16, None, None, A, None, None) == INVALID
    assert d(A, U, 4, 8, 16, None, None, A, None, None) == MISALIGNED
    assert d(A, A, 4, 8, 16, None, U, A, None, None) == MISALIGNED
    assert d(A, A, 0, 8, 16, None, None, A, None, None) == OK
    assert d(A, A, 4, 8, 16, None, None, A, U, None) == MISALIGNED             # workspace


def test_chunk_plan_validation(L):
    size = L.w8a8_chunk_plan_size
    # one word per 256-row block up to 32 chunks of 1024
    # per 256-row block: one word per 32 chunks of 1024, plus one
    assert size(256, 4096) == 2
    assert size(257, 4096) == 4
    assert size(12288, 4096) == 96
    assert size(256, 32 * 1024) == 2
    assert size(256, 32 * 1024 + 16) == 3
    assert size(0, 16) == 1
    f = L.w8a8_chunk_plan
    assert f(A, 12, 16, A, None) == SHAPE
    assert f(None, 8, 16, A, None) == INVALID
    assert f(A, 8, 16, None, None) == INVALID
    assert f(U, 8, 16, A, None) == MISALIGNED


def test_noalloc_stats_validation(L):
    f = L.w8a8_act_stats_noalloc
    assert f(A, 4, 32768 + 16, None, A, A, None) == SHAPE       # beyond the static scratch
    assert f(A, 4, 24, None, A, A, None) == SHAPE
    assert f(A, 0, 16, None, A, A, None) == INVALID            # no tokens
    assert f(A, -3, 16, None, A, A, None) == INVALID           # negative count: T >= 1
    assert f(None, 4, 16, None, A, A, None) == INVALID
    assert f(A, 4, 16, None, U, A, None) == MISALIGNED


def test_dual_f16codes_validation(L):
    from paper_2606_12280_gb300.w8a8 import ActBranch16, Branch16
    qa = (ActBranch16 * 2)()
    for i in range(2):
        qa[i] = ActBranch16(A, None, 4, A, A, None)
    f = L.w8a8_quant_act_dual_f16codes
    assert f(None, 16, None) == INVALID
    assert f(qa, 24, None) == SHAPE
    assert f(qa, 16400, None) == SHAPE                   # K beyond 16384
    qa[1].x_sumsq = U
    assert f(qa, 16, None) == MISALIGNED
    qa[1].x_sumsq = None
    qa[1].Xq16 = None
    assert f(qa, 16, None) == INVALID
    qa[0] = ActBranch16(None, None, 0, None, None, None)
    qa[1] = ActBranch16(None, None, 0, None, None, None)
    assert f(qa, 16, None) == OK                         # both branches empty
    ga = (Branch16 * 2)()
    for i in range(2):
        ga[i] = Branch16(A, A, A, A, None, A, 4, None, None)
    g = L.w8a8_linear_dual_f16codes
    assert g(None, 8, 16, None, None) == INVALID
    assert g(ga, 12, 16, None, None) == SHAPE
    assert g(ga, 8, 16, U, None) == MISALIGNED                # workspace
    ga[1].chunk_plan = U
    assert g(ga, 8, 16, None, None) == MISALIGNED
    ga[1].chunk_plan = None
    ga[1].Wq = None
    assert g(ga, 8, 16, None, None) == INVALID
    ga[0] = Branch16(None, None, None, None, None, None, 0, None, None)
    ga[1] = Branch16(None, None, None, None, None, None, 0, None, None)
    assert g(ga, 8, 16, None, None) == OK                      # both branches empty
