"""Python binding of the W8A8 C ABI (include/w8a8.h).

Argument marshalling only: each function takes CUDA tensors, checks dtype,
device and contiguity, and passes ``data_ptr()`` plus the current CUDA stream
to the function of the same name in ``libw8a8.so``.  Every step of the layer
runs in the library's CUDA kernels; there is no fallback.  If the library has
not been built, or cannot be loaded, the first call raises.
"""

from __future__ import annotations

import ctypes
import os
import threading

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libw8a8.so")

W8A8_OK = 0
STATUS_NAMES = {0: "W8A8_OK", 1: "W8A8_ERR_INVALID_ARG", 2: "W8A8_ERR_UNSUPPORTED_SHAPE",
                3: "W8A8_ERR_MISALIGNED", 4: "W8A8_ERR_CUDA", 5: "W8A8_ERR_TIMEOUT"}

# name -> argument types, in header order
_P, _I, _F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
SIGNATURES = {
    "w8a8_channel_absmax": [_P, _I, _I, _P, _P],
    "w8a8_smooth_scales": [_P, _P, _I, _I, _F, _P, _P],
    "w8a8_quantize_weights": [_P, _P, _I, _I, _P, _P, _P],
    "w8a8_quant_act": [_P, _P, _I, _I, _P, _P, _P],
    "w8a8_linear": [_P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P],
    "w8a8_linear_workspace_size": [ctypes.c_longlong, _I],
    "w8a8_linear_dual": [_P, _I, _I, _P, _P],
    "w8a8_debug_gemm_i32": [_P, _P, _I, _I, _I, _P, _P, _P, _P],
    "w8a8_debug_linear_engine": [_I, _P, _I, _I, _I, _I, _P],
    "w8a8_device_status": [_P, ctypes.POINTER(ctypes.c_uint32)],
    "w8a8_debug_wait_timeout": [ctypes.c_uint32, _P],
    "w8a8_status_string": [_I],
    "w8a8_quant_act_per_tensor": [_P, _P, _I, _I, _P, _P, _P, _P],
    "w8a8_act_stats_update": [_P, _I, _I, _P, _P, _P, _P],
    "w8a8_act_stats_finalize": [_P, _P, _P, ctypes.c_longlong, _I, _P, _P, _P],
    "w8a8_linear_bf16": [_P, _P, _P, _I, _I, _I, _P, _P],
    "w8a8_layer_forward": [_P, _P, _I, _P, _P, _P, _P, _P],
    "w8a8_select_protected": [_P, _I, _I, _P],
    "w8a8_quant_act_dual": [_P, _I, _P],
    "w8a8_gelu_quant_act": [_P, _P, _I, _I, _P, _P, _P],
    "w8a8_debug_gelu": [_P, _I, _P, _P],
    "w8a8_linear_gguf": [_P, _P, _I, _P, _I, _I, _I, _P, _P],
    "w8a8_debug_gguf_dequant": [_P, _I, _I, _I, _P, _P],
    "w8a8_quant_act_f16codes": [_P, _P, _I, _I, _P, _P, _P, _I, _P],
    "w8a8_linear_f16codes": [_P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P],
    "w8a8_gemm_workspace_size": [],
    "w8a8_debug_gemm_f16codes_i32": [_P, _P, _I, _I, _I, _P, _P, _P, _P, _P],
    "w8a8_chunk_plan_size": [_I, _I],
    "w8a8_quant_act_dual_f16codes": [_P, _I, _P],
    "w8a8_linear_dual_f16codes": [_P, _I, _I, _P, _P],
    "w8a8_chunk_plan": [_P, _I, _I, _P, _P],
    "w8a8_act_stats_noalloc": [_P, _I, _I, _P, _P, _P, _P],
}

NOALLOC_STATS_MAX_K = 32768

GGUF_Q8_0, GGUF_Q4_K = 0, 1


class W8A8Error(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} returned {STATUS_NAMES.get(status, status)}")
        self.status = status


class Branch(ctypes.Structure):
    """Mirror of ``w8a8_branch``."""
    _fields_ = [("Xq", _P), ("x_scale", _P), ("Wq", _P), ("w_scale", _P),
                ("bias", _P), ("Y", _P), ("M", _I), ("chunk_plan", _P)]


class ActBranch(ctypes.Structure):
    """Mirror of ``w8a8_act_branch``."""
    _fields_ = [("X", _P), ("smooth", _P), ("M", _I), ("Xq", _P), ("x_scale", _P)]


class ActBranch16(ctypes.Structure):
    """Mirror of ``w8a8_act_branch16``."""
    _fields_ = [("X", _P), ("smooth", _P), ("M", _I), ("Xq16", _P), ("x_scale", _P), ("x_sumsq", _P)]


class Branch16(ctypes.Structure):
    """Mirror of ``w8a8_branch16``."""
    _fields_ = [("Xq16", _P), ("x_scale", _P), ("Wq", _P), ("w_scale", _P), ("bias", _P), ("Y", _P),
                ("M", _I), ("chunk_plan", _P), ("x_sumsq", _P)]


class Layer(ctypes.Structure):
    """Mirror of ``w8a8_layer``."""
    _fields_ = [("protect", _I), ("N", _I), ("K", _I), ("smooth", _P), ("Wq", _P),
                ("w_scale", _P), ("W_bf16", _P), ("bias", _P), ("chunk_plan", _P)]


_lock = threading.Lock()
_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library (raises if it is missing: there is no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"W8A8 CUDA library not built ({LIB_PATH} missing); run "
                    "`python -c 'import __graft_entry__ as g; g.build()'`")
            L = ctypes.CDLL(LIB_PATH)
            for name, args in SIGNATURES.items():
                fn = getattr(L, name)
                fn.argtypes = args
                fn.restype = ctypes.c_int
            L.w8a8_status_string.restype = ctypes.c_char_p
            L.w8a8_chunk_plan_size.restype = ctypes.c_longlong
            L.w8a8_gemm_workspace_size.restype = ctypes.c_longlong
            L.w8a8_linear_workspace_size.restype = ctypes.c_longlong
            _lib = L
    return _lib


def _check(name: str, status: int) -> None:
    if status != W8A8_OK:
        raise W8A8Error(name, status)


def _stream(stream=None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _ptr(t, dtype, name):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    # the library launches on the current device and dereferences every
    # pointer there
    if t.device.index != torch.cuda.current_device():
        raise ValueError(f"{name} is on {t.device}, the current device is cuda:{torch.cuda.current_device()}")
    return t.data_ptr()


def _shape(t, shape, name):
    """Refuse a tensor whose shape is not exactly `shape` (where the library
    addresses it with strides that the shape fixes)."""
    if t is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, the call needs {tuple(shape)}")


def _room(t, n, name):
    """Refuse a tensor with fewer than n elements where the library reads or
    writes n (the C ABI takes plain pointers and cannot check sizes)."""
    if t is not None and t.numel() < n:
        raise ValueError(f"{name} holds {t.numel()} elements, the call needs {n}")


def _gguf_row_bytes(fmt: int, K: int) -> int:
    return (K // 32) * 34 if int(fmt) == 0 else (K // 256) * 144


def channel_absmax(X, s=None, stream=None):
    """s_j = max_t |X_tj| (calibration statistic).  X [T,K] bf16 -> s [K] fp32."""
    T, K = X.shape
    if s is None:
        s = torch.empty(K, dtype=torch.float32, device=X.device)
    _room(s, K, "s")
    _check("w8a8_channel_absmax", lib().w8a8_channel_absmax(
        _ptr(X, torch.bfloat16, "X"), T, K, _ptr(s, torch.float32, "s"), _stream(stream)))
    return s


def smooth_scales(act_absmax, W, alpha: float, smooth=None, stream=None):
    """lambda_j = s_j^alpha / max_i |W_ij|^(1-alpha).  W [N,K] fp32 -> [K] fp32."""
    N, K = W.shape
    if smooth is None:
        smooth = torch.empty(K, dtype=torch.float32, device=W.device)
    _room(act_absmax, K, "act_absmax")
    _room(smooth, K, "smooth")
    _check("w8a8_smooth_scales", lib().w8a8_smooth_scales(
        _ptr(act_absmax, torch.float32, "act_absmax"), _ptr(W, torch.float32, "W"), N, K,
        float(alpha), _ptr(smooth, torch.float32, "smooth"), _stream(stream)))
    return smooth


def quantize_weights(W, smooth=None, Wq=None, w_scale=None, stream=None):
    """Per-output-channel INT8 of W diag(lambda): returns (Wq [N,K] int8, sw [N] fp32)."""
    N, K = W.shape
    if Wq is None:
        Wq = torch.empty(N, K, dtype=torch.int8, device=W.device)
    if w_scale is None:
        w_scale = torch.empty(N, dtype=torch.float32, device=W.device)
    _room(smooth, K, "smooth")
    _room(Wq, N * K, "Wq")
    _room(w_scale, N, "w_scale")
    _check("w8a8_quantize_weights", lib().w8a8_quantize_weights(
        _ptr(W, torch.float32, "W"), _ptr(smooth, torch.float32, "smooth"), N, K,
        _ptr(Wq, torch.int8, "Wq"), _ptr(w_scale, torch.float32, "w_scale"), _stream(stream)))
    return Wq, w_scale


def quant_act(X, smooth=None, Xq=None, x_scale=None, stream=None):
    """Per-token INT8 of X diag(lambda)^-1: returns (Xq [M,K] int8, sx [M] fp32)."""
    M, K = X.shape
    if Xq is None:
        Xq = torch.empty(M, K, dtype=torch.int8, device=X.device)
    if x_scale is None:
        x_scale = torch.empty(M, dtype=torch.float32, device=X.device)
    _room(smooth, K, "smooth")
    _room(Xq, M * K, "Xq")
    _room(x_scale, M, "x_scale")
    _check("w8a8_quant_act", lib().w8a8_quant_act(
        _ptr(X, torch.bfloat16, "X"), _ptr(smooth, torch.float32, "smooth"), M, K,
        _ptr(Xq, torch.int8, "Xq"), _ptr(x_scale, torch.float32, "x_scale"), _stream(stream)))
    return Xq, x_scale


def _check_weights(Wq, N, K):
    if tuple(Wq.shape) != (N, K):
        raise ValueError(f"Wq has shape {tuple(Wq.shape)}, the activations need ({N}, {K})")


def linear(Xq, x_scale, Wq, w_scale, bias=None, Y=None, plan=None, workspace=None, stream=None):
    """Y = bf16((Xq Wq^T) * sx * sw + b): [M,N] bf16.  workspace: None, or
    ``linear_workspace(M, K)`` (the codes are then expanded to fp16 values
    and run on the GEMM of ``linear_f16codes``, with ``plan`` =
    ``chunk_plan(Wq)`` or None; same bits)."""
    M, K = Xq.shape
    N = Wq.shape[0]
    _check_weights(Wq, N, K)
    if Y is None:
        Y = torch.empty(M, N, dtype=torch.bfloat16, device=Xq.device)
    _room(x_scale, M, "x_scale")
    _room(w_scale, N, "w_scale")
    _room(bias, N, "bias")
    _room(Y, M * N, "Y")
    if plan is not None:
        _room(plan, chunk_plan_size(N, K), "plan")
    ws = _linear_ws(workspace, M, K)
    _check("w8a8_linear", lib().w8a8_linear(
        _ptr(Xq, torch.int8, "Xq"), _ptr(x_scale, torch.float32, "x_scale"),
        _ptr(Wq, torch.int8, "Wq"), _ptr(w_scale, torch.float32, "w_scale"),
        _ptr(bias, torch.float32, "bias"), M, N, K, _ptr(Y, torch.bfloat16, "Y"),
        _ptr(plan, torch.int32, "plan"), ws, _stream(stream)))
    return Y


def linear_workspace_size(tokens: int, K: int) -> int:
    """Bytes of the workspace of ``linear`` (tokens = M) or ``linear_dual``
    (tokens = M0 + M1) on the current device."""
    return int(lib().w8a8_linear_workspace_size(int(tokens), int(K)))


def linear_workspace(tokens: int, K: int, device=None):
    """A zeroed workspace for ``linear`` / ``linear_dual`` with up to `tokens`
    tokens of K channels (a uint8 tensor; calls that overlap in time need
    their own)."""
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        return torch.zeros(linear_workspace_size(tokens, K), dtype=torch.uint8, device=device)


def _linear_ws(ws, tokens, K):
    if ws is None:
        return None
    if ws.dtype != torch.uint8 or ws.numel() < linear_workspace_size(tokens, K):
        raise ValueError("workspace: a uint8 tensor of linear_workspace_size(tokens, K) bytes "
                         "(linear_workspace())")
    return _ptr(ws, torch.uint8, "workspace")


def _branch_array(branches, Ys, out_dtype=torch.bfloat16):
    """Branch structs for two (or one) branches (Xq, x_scale, Wq, w_scale,
    bias[, plan]); returns (array, outputs, N, K)."""
    N, K = branches[0][2].shape
    arr = (Branch * len(branches))()
    out = []
    for i, br in enumerate(branches):
        Xq, sx, Wq, sw, b = br[:5]
        plan = br[5] if len(br) > 5 else None
        if tuple(Wq.shape) != (N, K) or Xq.shape[1] != K:
            raise ValueError("branches must share N and K")
        M = Xq.shape[0]
        Y = Ys[i] if Ys is not None else torch.empty(M, N, dtype=out_dtype, device=Xq.device)
        _room(sx, M, "x_scale")
        _room(sw, N, "w_scale")
        _room(b, N, "bias")
        _room(Y, M * N, "Y")
        if plan is not None:
            _room(plan, chunk_plan_size(N, K), "plan")
        arr[i] = Branch(_ptr(Xq, torch.int8, "Xq"), _ptr(sx, torch.float32, "x_scale"),
                        _ptr(Wq, torch.int8, "Wq"), _ptr(sw, torch.float32, "w_scale"),
                        _ptr(b, torch.float32, "bias"), _ptr(Y, out_dtype, "Y"), M,
                        _ptr(plan, torch.int32, "plan"))
        out.append(Y)
    return arr, out, N, K


def linear_dual(branches, Ys=None, workspace=None, stream=None):
    """One grouped launch over two branches.  branches: two tuples
    (Xq, x_scale, Wq, w_scale, bias[, plan]); workspace: None or
    ``linear_workspace(M0 + M1, K)``; returns [Y_cond, Y_uncond]."""
    if len(branches) != 2:
        raise ValueError("linear_dual takes exactly two branches")
    tokens = sum(int(br[0].shape[0]) for br in branches)
    ws = _linear_ws(workspace, tokens, int(branches[0][0].shape[1]))
    arr, out, N, K = _branch_array(branches, Ys)
    _check("w8a8_linear_dual", lib().w8a8_linear_dual(arr, N, K, ws, _stream(stream)))
    return out


def debug_gemm_i32(Xq, Wq, acc=None, plan=None, workspace=None, stream=None):
    """Exact int32 acc = Xq Wq^T (test export of the GEMM alone; plan and
    workspace as for ``linear``)."""
    M, K = Xq.shape
    N = Wq.shape[0]
    _check_weights(Wq, N, K)
    if acc is None:
        acc = torch.empty(M, N, dtype=torch.int32, device=Xq.device)
    _room(acc, M * N, "acc")
    if plan is not None:
        _room(plan, chunk_plan_size(N, K), "plan")
    ws = _linear_ws(workspace, M, K)
    _check("w8a8_debug_gemm_i32", lib().w8a8_debug_gemm_i32(
        _ptr(Xq, torch.int8, "Xq"), _ptr(Wq, torch.int8, "Wq"), M, N, K,
        _ptr(acc, torch.int32, "acc"), _ptr(plan, torch.int32, "plan"), ws, _stream(stream)))
    return acc


def debug_linear_engine(engine: int, branches, Ys=None, out_i32=False, stream=None):
    """Test anchor: the exact-integer product on a chosen int8-code engine (2
    the product's tcgen05 CTA pairs, 1 tcgen05 single SMs, 0 mma.sync), per
    call, on one or two branches (Xq, x_scale, Wq, w_scale, bias); returns the
    outputs (bf16 Y, or int32 products when out_i32)."""
    if len(branches) not in (1, 2):
        raise ValueError("one or two branches")
    arr, out, N, K = _branch_array(branches, Ys, torch.int32 if out_i32 else torch.bfloat16)
    _check("w8a8_debug_linear_engine", lib().w8a8_debug_linear_engine(
        int(engine), arr, len(branches), N, K, 1 if out_i32 else 0, _stream(stream)))
    return out


def device_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device error word."""
    detail = ctypes.c_uint32(0)
    st = lib().w8a8_device_status(_stream(stream), ctypes.byref(detail))
    if st not in (W8A8_OK, 5):
        raise W8A8Error("w8a8_device_status", st)
    return int(detail.value)


def debug_wait_timeout(limit_us: int, stream=None) -> None:
    """Enqueue a bounded wait that can only time out (failure-detection test)."""
    _check("w8a8_debug_wait_timeout", lib().w8a8_debug_wait_timeout(int(limit_us), _stream(stream)))


def quant_act_dual(branches, out=None, stream=None):
    """a3 for two branches in one launch: branches = [(X, smooth), (X, smooth)]
    (smooth may be None); returns [(Xq, sx), (Xq, sx)] (written into `out`
    when given)."""
    if len(branches) != 2:
        raise ValueError("quant_act_dual takes exactly two branches")
    K = branches[0][0].shape[1]
    arr = (ActBranch * 2)()
    res = []
    for i, (X, sm) in enumerate(branches):
        if X.shape[1] != K:
            raise ValueError("branches must share K")
        M = X.shape[0]
        if out is not None:
            Xq, sx = out[i]
        else:
            Xq = torch.empty(M, K, dtype=torch.int8, device=X.device)
            sx = torch.empty(M, dtype=torch.float32, device=X.device)
        _room(sm, K, "smooth")
        _room(Xq, M * K, "Xq")
        _room(sx, M, "x_scale")
        arr[i] = ActBranch(_ptr(X, torch.bfloat16, "X"), _ptr(sm, torch.float32, "smooth"), M,
                           _ptr(Xq, torch.int8, "Xq"), _ptr(sx, torch.float32, "x_scale"))
        res.append((Xq, sx))
    _check("w8a8_quant_act_dual", lib().w8a8_quant_act_dual(arr, K, _stream(stream)))
    return res


def quant_act_dual_f16codes(branches, out=None, stream=None):
    """a3 with fp16 codes for two branches in one launch: branches = [(X,
    smooth), (X, smooth)]; returns [(Xq16, sx, sumsq), ...] (written into
    `out` when given; sumsq int32 [M] holding the uint32 token sums)."""
    if len(branches) != 2:
        raise ValueError("quant_act_dual_f16codes takes exactly two branches")
    K = branches[0][0].shape[1]
    arr = (ActBranch16 * 2)()
    res = []
    for i, (X, sm) in enumerate(branches):
        if X.shape[1] != K:
            raise ValueError("branches must share K")
        M = X.shape[0]
        if out is not None:
            Xq16, sx, ss = out[i]
        else:
            Xq16 = torch.empty(M, K, dtype=torch.float16, device=X.device)
            sx = torch.empty(M, dtype=torch.float32, device=X.device)
            ss = torch.empty(M, dtype=torch.int32, device=X.device)
        _room(sm, K, "smooth")
        _room(Xq16, M * K, "Xq16")
        _room(sx, M, "x_scale")
        _room(ss, M, "sumsq")
        arr[i] = ActBranch16(_ptr(X, torch.bfloat16, "X"), _ptr(sm, torch.float32, "smooth"), M,
                             _ptr(Xq16, torch.float16, "Xq16"), _ptr(sx, torch.float32, "x_scale"),
                             _ptr(ss, torch.int32, "sumsq"))
        res.append((Xq16, sx, ss))
    _check("w8a8_quant_act_dual_f16codes", lib().w8a8_quant_act_dual_f16codes(arr, K, _stream(stream)))
    return res


def linear_dual_f16codes(branches, Ys=None, workspace=None, stream=None):
    """One grouped launch over two branches with fp16 codes.  branches: two
    tuples (Xq16, x_scale, Wq, w_scale, bias, plan, x_sumsq) (plan and x_sumsq
    may be None); returns [Y_cond, Y_uncond].  workspace: None or
    ``gemm_workspace()`` (see ``linear_f16codes``)."""
    if len(branches) != 2:
        raise ValueError("linear_dual_f16codes takes exactly two branches")
    ws = _workspace(workspace)
    N, K = branches[0][2].shape
    arr = (Branch16 * 2)()
    out = []
    for i, (Xq16, sx, Wq, sw, b, plan, ss) in enumerate(branches):
        if tuple(Wq.shape) != (N, K) or Xq16.shape[1] != K:
            raise ValueError("branches must share N and K")
        Y = Ys[i] if Ys is not None else torch.empty(Xq16.shape[0], N, dtype=torch.bfloat16,
                                                     device=Xq16.device)
        M = Xq16.shape[0]
        _room(sx, M, "x_scale")
        _room(sw, N, "w_scale")
        _room(b, N, "bias")
        if plan is not None:
            _room(plan, chunk_plan_size(N, K), "plan")
        _room(ss, M, "x_sumsq")
        _room(Y, M * N, "Y")
        arr[i] = Branch16(_ptr(Xq16, torch.float16, "Xq16"), _ptr(sx, torch.float32, "x_scale"),
                          _ptr(Wq, torch.int8, "Wq"), _ptr(sw, torch.float32, "w_scale"),
                          _ptr(b, torch.float32, "bias"), _ptr(Y, torch.bfloat16, "Y"), Xq16.shape[0],
                          _ptr(plan, torch.int32, "plan"), _ptr(ss, torch.int32, "x_sumsq"))
        out.append(Y)
    _check("w8a8_linear_dual_f16codes", lib().w8a8_linear_dual_f16codes(arr, N, K, ws, _stream(stream)))
    return out


def gelu_quant_act(H, smooth=None, Xq=None, x_scale=None, stream=None):
    """Per-token INT8 of GELU(H) diag(lambda)^-1 in one pass: returns (Xq, sx)."""
    M, K = H.shape
    if Xq is None:
        Xq = torch.empty(M, K, dtype=torch.int8, device=H.device)
    if x_scale is None:
        x_scale = torch.empty(M, dtype=torch.float32, device=H.device)
    _room(smooth, K, "smooth")
    _room(Xq, M * K, "Xq")
    _room(x_scale, M, "x_scale")
    _check("w8a8_gelu_quant_act", lib().w8a8_gelu_quant_act(
        _ptr(H, torch.bfloat16, "H"), _ptr(smooth, torch.float32, "smooth"), M, K,
        _ptr(Xq, torch.int8, "Xq"), _ptr(x_scale, torch.float32, "x_scale"), _stream(stream)))
    return Xq, x_scale


def quant_act_f16codes(X, smooth=None, Xq16=None, x_scale=None, gelu=False, sumsq=None, stream=None):
    """a3 with the codes as fp16 values: returns (Xq16 [M,K] float16, sx [M]).
    sumsq: None, or an int32 [M] tensor that receives sum_j Xq_mj^2 per token
    (uint32 values; for ``linear_f16codes(..., x_sumsq=)``)."""
    M, K = X.shape
    if Xq16 is None:
        Xq16 = torch.empty(M, K, dtype=torch.float16, device=X.device)
    if x_scale is None:
        x_scale = torch.empty(M, dtype=torch.float32, device=X.device)
    _room(smooth, K, "smooth")
    _room(Xq16, M * K, "Xq16")
    _room(x_scale, M, "x_scale")
    _room(sumsq, M, "sumsq")
    _check("w8a8_quant_act_f16codes", lib().w8a8_quant_act_f16codes(
        _ptr(X, torch.bfloat16, "X"), _ptr(smooth, torch.float32, "smooth"), M, K,
        _ptr(Xq16, torch.float16, "Xq16"), _ptr(x_scale, torch.float32, "x_scale"),
        _ptr(sumsq, torch.int32, "sumsq"), 1 if gelu else 0, _stream(stream)))
    return Xq16, x_scale


def linear_f16codes(Xq16, x_scale, Wq, w_scale, bias=None, Y=None, plan=None, x_sumsq=None, workspace=None,
                    stream=None):
    """a4 + a5 with fp16-coded activations: Y = bf16((Xq Wq^T) * sx * sw + b).
    plan: None or ``chunk_plan(Wq)``; x_sumsq: None or the token sums that
    ``quant_act_f16codes(..., sumsq=)`` wrote for these codes; workspace: None
    or ``gemm_workspace()`` (the last round of tiles is then split over K
    between idle SM pairs; same bits)."""
    M, K = Xq16.shape
    N = Wq.shape[0]
    _check_weights(Wq, N, K)
    if Y is None:
        Y = torch.empty(M, N, dtype=torch.bfloat16, device=Xq16.device)
    _room(x_scale, M, "x_scale")
    _room(w_scale, N, "w_scale")
    _room(bias, N, "bias")
    if plan is not None:
        _room(plan, chunk_plan_size(N, K), "plan")
    _room(x_sumsq, M, "x_sumsq")
    _room(Y, M * N, "Y")
    ws = _workspace(workspace)
    _check("w8a8_linear_f16codes", lib().w8a8_linear_f16codes(
        _ptr(Xq16, torch.float16, "Xq16"), _ptr(x_scale, torch.float32, "x_scale"),
        _ptr(Wq, torch.int8, "Wq"), _ptr(w_scale, torch.float32, "w_scale"),
        _ptr(bias, torch.float32, "bias"), M, N, K, _ptr(plan, torch.int32, "plan"),
        _ptr(x_sumsq, torch.int32, "x_sumsq"), _ptr(Y, torch.bfloat16, "Y"), ws, _stream(stream)))
    return Y


def debug_gemm_f16codes_i32(Xq16, Wq, plan=None, x_sumsq=None, acc=None, workspace=None, stream=None):
    """Exact int32 acc = Xq16 Wq^T (test export of the fp16-code GEMM)."""
    M, K = Xq16.shape
    N = Wq.shape[0]
    _check_weights(Wq, N, K)
    if acc is None:
        acc = torch.empty(M, N, dtype=torch.int32, device=Xq16.device)
    if plan is not None:
        _room(plan, chunk_plan_size(N, K), "plan")
    _room(x_sumsq, M, "x_sumsq")
    _room(acc, M * N, "acc")
    ws = _workspace(workspace)
    _check("w8a8_debug_gemm_f16codes_i32", lib().w8a8_debug_gemm_f16codes_i32(
        _ptr(Xq16, torch.float16, "Xq16"), _ptr(Wq, torch.int8, "Wq"), M, N, K,
        _ptr(plan, torch.int32, "plan"), _ptr(x_sumsq, torch.int32, "x_sumsq"),
        _ptr(acc, torch.int32, "acc"), ws, _stream(stream)))
    return acc


def gemm_workspace_size() -> int:
    """Bytes of the fp16-code GEMM's workspace on the current device."""
    return int(lib().w8a8_gemm_workspace_size())


def gemm_workspace(device=None):
    """A zeroed workspace for ``linear_f16codes`` / ``linear_dual_f16codes``
    on `device` (a uint8 tensor; calls that overlap in time need their own)."""
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        return torch.zeros(gemm_workspace_size(), dtype=torch.uint8, device=device)


def _workspace(ws):
    if ws is None:
        return None
    if ws.dtype != torch.uint8 or ws.numel() < gemm_workspace_size():
        raise ValueError("workspace: a uint8 tensor of gemm_workspace_size() bytes (gemm_workspace())")
    return _ptr(ws, torch.uint8, "workspace")


def chunk_plan_size(N: int, K: int) -> int:
    """Words of the drain plan of an [N, K] int8 weight."""
    return int(lib().w8a8_chunk_plan_size(int(N), int(K)))


def chunk_plan(Wq, plan=None, stream=None):
    """Drain plan of the int8 weights Wq [N, K] for ``linear_f16codes`` (an
    int32 tensor holding the library's uint32 words)."""
    N, K = Wq.shape
    if plan is None:
        plan = torch.empty(chunk_plan_size(N, K), dtype=torch.int32, device=Wq.device)
    _room(plan, chunk_plan_size(N, K), "plan")
    _check("w8a8_chunk_plan", lib().w8a8_chunk_plan(
        _ptr(Wq, torch.int8, "Wq"), N, K, _ptr(plan, torch.int32, "plan"), _stream(stream)))
    return plan


def linear_gguf(X, Wraw, fmt: int, N: int, bias=None, Y=None, stream=None):
    """GGUF weight-only layer: Y = bf16(X dequant(W)^T + b); Wraw uint8 blocks
    (Q8_0: fmt 0, Q4_K: fmt 1) of N rows."""
    M, K = X.shape
    if Y is None:
        Y = torch.empty(M, N, dtype=torch.bfloat16, device=X.device)
    if int(fmt) in (0, 1):
        _room(Wraw, N * _gguf_row_bytes(fmt, K), "Wraw")
    _room(bias, N, "bias")
    _room(Y, M * N, "Y")
    _check("w8a8_linear_gguf", lib().w8a8_linear_gguf(
        _ptr(X, torch.bfloat16, "X"), _ptr(Wraw, torch.uint8, "Wraw"), int(fmt),
        _ptr(bias, torch.float32, "bias"), M, N, K, _ptr(Y, torch.bfloat16, "Y"), _stream(stream)))
    return Y


def debug_gguf_dequant(Wraw, fmt: int, N: int, K: int, W=None, stream=None):
    """The decoded weights [N, K] bf16."""
    if W is None:
        W = torch.empty(N, K, dtype=torch.bfloat16, device=Wraw.device)
    if int(fmt) in (0, 1):
        _room(Wraw, N * _gguf_row_bytes(fmt, K), "Wraw")
    _room(W, N * K, "W")
    _check("w8a8_debug_gguf_dequant", lib().w8a8_debug_gguf_dequant(
        _ptr(Wraw, torch.uint8, "Wraw"), int(fmt), N, K, _ptr(W, torch.bfloat16, "W"),
        _stream(stream)))
    return W


def debug_gelu(H, G=None, stream=None):
    """The fp32 GELU values of the fused pass, for a flat bf16 tensor H."""
    n = H.numel()
    if G is None:
        G = torch.empty(n, dtype=torch.float32, device=H.device)
    _room(G, n, "G")
    _check("w8a8_debug_gelu", lib().w8a8_debug_gelu(
        _ptr(H, torch.bfloat16, "H"), n, _ptr(G, torch.float32, "G"), _stream(stream)))
    return G


def quant_act_per_tensor(X, smooth=None, Xq=None, x_scale=None, amax=None, stream=None):
    """One INT8 scale for all of X diag(lambda)^-1: returns (Xq, sx [M], amax [1])."""
    M, K = X.shape
    if Xq is None:
        Xq = torch.empty(M, K, dtype=torch.int8, device=X.device)
    if x_scale is None:
        x_scale = torch.empty(M, dtype=torch.float32, device=X.device)
    if amax is None:
        amax = torch.empty(1, dtype=torch.float32, device=X.device)
    _room(smooth, K, "smooth")
    _room(Xq, M * K, "Xq")
    _room(x_scale, M, "x_scale")
    _room(amax, 1, "amax")
    _check("w8a8_quant_act_per_tensor", lib().w8a8_quant_act_per_tensor(
        _ptr(X, torch.bfloat16, "X"), _ptr(smooth, torch.float32, "smooth"), M, K,
        _ptr(Xq, torch.int8, "Xq"), _ptr(x_scale, torch.float32, "x_scale"),
        _ptr(amax, torch.float32, "amax"), _stream(stream)))
    return Xq, x_scale, amax


def act_stats_update(X, sums, absmax, shift=None, stream=None):
    """Accumulate the per-channel power sums [4,K] fp64 and absmax [K] of X [T,K] bf16."""
    T, K = X.shape
    _room(shift, K, "shift")
    # the library addresses the four planes at stride K
    _shape(sums, (4, K), "sums")
    _shape(absmax, (K,), "absmax")
    _check("w8a8_act_stats_update", lib().w8a8_act_stats_update(
        _ptr(X, torch.bfloat16, "X"), T, K, _ptr(shift, torch.float32, "shift"),
        _ptr(sums, torch.float64, "sums"), _ptr(absmax, torch.float32, "absmax"),
        _stream(stream)))


def act_stats_finalize(sums, absmax, count: int, shift=None, chan=None, tensor=None, stream=None):
    """(chan [4,K], tensor [4]) fp32: max-abs, mean, std, kurtosis."""
    K = absmax.shape[0]
    if chan is None:
        chan = torch.empty(4, K, dtype=torch.float32, device=absmax.device)
    if tensor is None:
        tensor = torch.empty(4, dtype=torch.float32, device=absmax.device)
    _shape(absmax, (K,), "absmax")
    _shape(sums, (4, K), "sums")
    _room(shift, K, "shift")
    _room(chan, 4 * K, "chan")
    _room(tensor, 4, "tensor")
    _check("w8a8_act_stats_finalize", lib().w8a8_act_stats_finalize(
        _ptr(sums, torch.float64, "sums"), _ptr(absmax, torch.float32, "absmax"),
        _ptr(shift, torch.float32, "shift"), int(count), K, _ptr(chan, torch.float32, "chan"),
        _ptr(tensor, torch.float32, "tensor"), _stream(stream)))
    return chan, tensor


def act_stats_noalloc(X, shift=None, chan=None, tensor=None, stream=None):
    """Statistics of one batch X [T,K] bf16 with the library's static scratch:
    (chan [4,K], tensor [4]) fp32.  Overlapping calls race (shared scratch)."""
    T, K = X.shape
    if chan is None:
        chan = torch.empty(4, K, dtype=torch.float32, device=X.device)
    if tensor is None:
        tensor = torch.empty(4, dtype=torch.float32, device=X.device)
    _room(shift, K, "shift")
    _room(chan, 4 * K, "chan")
    _room(tensor, 4, "tensor")
    _check("w8a8_act_stats_noalloc", lib().w8a8_act_stats_noalloc(
        _ptr(X, torch.bfloat16, "X"), T, K, _ptr(shift, torch.float32, "shift"),
        _ptr(chan, torch.float32, "chan"), _ptr(tensor, torch.float32, "tensor"), _stream(stream)))
    return chan, tensor


def linear_bf16(X, W, bias=None, Y=None, stream=None):
    """Protected layer: Y = bf16(X W^T + b), X [M,K] and W [N,K] bf16."""
    M, K = X.shape
    N = W.shape[0]
    if W.shape[1] != K:
        raise ValueError("X and W disagree on K")
    if Y is None:
        Y = torch.empty(M, N, dtype=torch.bfloat16, device=X.device)
    _room(bias, N, "bias")
    _room(Y, M * N, "Y")
    _check("w8a8_linear_bf16", lib().w8a8_linear_bf16(
        _ptr(X, torch.bfloat16, "X"), _ptr(W, torch.bfloat16, "W"),
        _ptr(bias, torch.float32, "bias"), M, N, K, _ptr(Y, torch.bfloat16, "Y"),
        _stream(stream)))
    return Y


def layer_forward(X, protect: bool, N: int, K: int, smooth=None, Wq=None, w_scale=None,
                  W_bf16=None, bias=None, Xq_work=None, x_scale_work=None, Y=None, plan=None,
                  workspace=None, stream=None):
    """Per-layer dispatch (protected -> bf16 linear, else a3 + a4 + a5).
    workspace: None or ``linear_workspace(M, K)``; with it (K <= 16384) a3
    writes fp16 codes into it and Xq_work is not needed; plan: None or
    ``chunk_plan(Wq)``."""
    M = X.shape[0]
    if tuple(X.shape) != (M, K):
        raise ValueError(f"X has shape {tuple(X.shape)}, the layer needs ({M}, {K})")
    if Y is None:
        Y = torch.empty(M, N, dtype=torch.bfloat16, device=X.device)
    _room(bias, N, "bias")
    _room(Y, M * N, "Y")
    if protect:
        _room(W_bf16, N * K, "W_bf16")
    else:
        if Xq_work is None and (workspace is None or K > 16384):
            Xq_work = torch.empty(M, K, dtype=torch.int8, device=X.device)
        if x_scale_work is None:
            x_scale_work = torch.empty(M, dtype=torch.float32, device=X.device)
        _room(smooth, K, "smooth")
        _room(Wq, N * K, "Wq")
        _room(w_scale, N, "w_scale")
        _room(Xq_work, M * K, "Xq_work")
        _room(x_scale_work, M, "x_scale_work")
        if plan is not None:
            _room(plan, chunk_plan_size(N, K), "plan")
    ws = None if protect else _linear_ws(workspace, M, K)
    layer = Layer(1 if protect else 0, N, K, _ptr(smooth, torch.float32, "smooth"),
                  _ptr(Wq, torch.int8, "Wq"), _ptr(w_scale, torch.float32, "w_scale"),
                  _ptr(W_bf16, torch.bfloat16, "W_bf16"), _ptr(bias, torch.float32, "bias"),
                  None if protect else _ptr(plan, torch.int32, "plan"))
    _check("w8a8_layer_forward", lib().w8a8_layer_forward(
        ctypes.byref(layer), _ptr(X, torch.bfloat16, "X"), M,
        _ptr(Xq_work, torch.int8, "Xq_work"), _ptr(x_scale_work, torch.float32, "x_scale_work"),
        _ptr(Y, torch.bfloat16, "Y"), ws, _stream(stream)))
    return Y


def select_protected(scores, n_protect: int):
    """Host: flags (list of 0/1) marking the n_protect most fragile layers."""
    L = len(scores)
    sc = (ctypes.c_float * L)(*[float(x) for x in scores])
    flags = (ctypes.c_int * L)()
    _check("w8a8_select_protected", lib().w8a8_select_protected(sc, L, int(n_protect), flags))
    return [int(f) for f in flags]


def quantized_linear_forward(X, smooth, Wq, w_scale, bias=None, plan=None, codes="f16", workspace=None,
                             stream=None):
    """The per-call hot path of one quantized linear: a3 then a4+a5.  codes:
    "f16" (the codes as fp16 values, the faster GEMM; K <= 16384, else the
    int8 container is used) or "int8"; plan: ``chunk_plan(Wq)`` or None;
    workspace: None, or ``linear_workspace(M, K)`` (the int8 container's
    faster GEMM; the fp16 codes use its split-K area).  Same bits in every
    combination."""
    if codes not in ("f16", "int8"):
        raise ValueError("codes must be 'f16' or 'int8'")
    M, K = X.shape
    _linear_ws(workspace, M, K)                 # checked before anything is launched
    if codes == "f16" and K <= 16384:
        ss = torch.empty(M, dtype=torch.int32, device=X.device) if plan is not None else None
        Xq16, sx = quant_act_f16codes(X, smooth, sumsq=ss, stream=stream)
        return linear_f16codes(Xq16, sx, Wq, w_scale, bias, plan=plan, x_sumsq=ss, workspace=workspace,
                               stream=stream)
    Xq, sx = quant_act(X, smooth, stream=stream)
    return linear(Xq, sx, Wq, w_scale, bias, plan=plan, workspace=workspace, stream=stream)
