"""CPU oracle of the W8A8 quantized linear layer (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never does, and the
oracle never imports the product: the two share only the seeded input
generators, which hold none of the method's arithmetic.

The arithmetic lives in ``w8a8_oracle.c``, ``protect_oracle.c``,
``fused_oracle.c`` and ``gguf_oracle.c`` (plain C,
``-O2 -ffp-contract=off``, no intrinsics), compiled with gcc into
``oracle/_build/liboracle.so`` and called through ctypes on numpy arrays.  Each
function follows the "INT8 W8A8" paragraph of the paper's Method section
(Sec. 3); the INT8 GEMM and dequantizing epilogue are the fused kernel the
paper lists as missing (Sec. 7, Limitations).  The activation statistics and
the protected bf16 layer follow Sec. 3, "Activation-fragility profiling and
protection"; the per-tensor activation scale is the naive arm of the
activation-quant ablation (Sec. 5, "What drives INT8 recovery"); the GELU
fused into the quantization of the FFN down-projection input takes the exact
erf GELU (the paper does not name the activation); the GGUF Q8_0 / Q4_K
weight-only layer decodes the public block formats (Sec. 3, "GGUF k-quants").
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRCS = [os.path.join(_HERE, f) for f in ("w8a8_oracle.c", "protect_oracle.c", "fused_oracle.c",
                                          "gguf_oracle.c")]
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP over GEMM rows when available)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and all(os.path.getmtime(_LIB_PATH) >= os.path.getmtime(f) for f in _SRCS)):
        return _LIB_PATH
    base = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11",
            "-shared", "-fPIC", *_SRCS, "-o", _LIB_PATH + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            lib = ctypes.CDLL(path)
            P = ctypes.c_void_p
            I64 = ctypes.c_int64
            lib.oracle_channel_absmax.argtypes = [P, I64, I64, P]
            lib.oracle_smooth_scales.argtypes = [P, P, I64, I64, ctypes.c_float, P]
            lib.oracle_quantize_weights.argtypes = [P, P, I64, I64, P, P]
            lib.oracle_quant_act.argtypes = [P, P, I64, I64, P, P, P]
            lib.oracle_gemm_i32.argtypes = [P, P, I64, I64, I64, I64, I64, P]
            lib.oracle_epilogue.argtypes = [P, P, P, P, I64, I64, P]
            lib.oracle_linear_rows.argtypes = [P, P, P, P, P, I64, I64, I64,
                                               I64, I64, P, P]
            lib.oracle_f32_to_bf16_rne.argtypes = [ctypes.c_float]
            lib.oracle_f32_to_bf16_rne.restype = ctypes.c_uint16
            lib.oracle_bf16_to_f32.argtypes = [ctypes.c_uint16]
            lib.oracle_bf16_to_f32.restype = ctypes.c_float
            lib.oracle_quantize_value.argtypes = [ctypes.c_float]
            lib.oracle_quantize_value.restype = ctypes.c_int8
            lib.oracle_epilogue_value.argtypes = [ctypes.c_int32, ctypes.c_float,
                                                  ctypes.c_float, P]
            lib.oracle_epilogue_value.restype = ctypes.c_uint16
            lib.oracle_num_threads.restype = ctypes.c_int
            lib.oracle_quant_act_per_tensor.argtypes = [P, P, I64, I64, P, P, P, P]
            lib.oracle_act_stats.argtypes = [P, I64, I64, P, P]
            lib.oracle_shifted_power_sums.argtypes = [P, I64, I64, P, P, P]
            lib.oracle_linear_bf16_rows.argtypes = [P, P, P, I64, I64, I64, I64, I64, P, P]
            lib.oracle_gelu_value.argtypes = [ctypes.c_float]
            lib.oracle_gelu_value.restype = ctypes.c_float
            lib.oracle_gelu_quant_act.argtypes = [P, P, I64, I64, P, P, P, P, P]
            lib.oracle_f32_to_bf16_rne_array.argtypes = [P, I64, P]
            lib.oracle_f16_to_f32.argtypes = [ctypes.c_uint16]
            lib.oracle_f16_to_f32.restype = ctypes.c_float
            lib.oracle_dequant_q8_0.argtypes = [P, I64, I64, P]
            lib.oracle_dequant_q4_k.argtypes = [P, I64, I64, P]
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    """Threads the oracle's GEMM row loop uses."""
    return int(_load().oracle_num_threads())


# --------------------------------------------------------------------------
# scalar helpers (bit patterns of bf16 are carried as uint16)
# --------------------------------------------------------------------------

def f32_to_bf16_rne(x) -> np.ndarray:
    """fp32 -> bf16 bit pattern, round to nearest, ties to even."""
    lib = _load()
    x = np.asarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    flat_in, flat_out = x.reshape(-1), out.reshape(-1)
    for i in range(flat_in.size):
        flat_out[i] = lib.oracle_f32_to_bf16_rne(float(flat_in[i]))
    return out


def bf16_to_f32(h) -> np.ndarray:
    """bf16 bit pattern -> fp32 (exact)."""
    h = np.asarray(h, dtype=np.uint16)
    return (h.astype(np.uint32) << 16).view(np.float32)


def quantize_value(v: float) -> int:
    """clamp(round_half_even(v), -127, 127) in fp32."""
    return int(_load().oracle_quantize_value(float(np.float32(v))))


# --------------------------------------------------------------------------
# the layer, step by step (Sec. 3, "INT8 W8A8")
# --------------------------------------------------------------------------

def channel_absmax(X_bf16: np.ndarray) -> np.ndarray:
    """Calibration statistic s_j = max_t |X_tj| over a [T, K] bf16 batch."""
    X = _c(X_bf16, np.uint16)
    M, K = X.shape
    s = np.empty(K, dtype=np.float32)
    _load().oracle_channel_absmax(_ptr(X), M, K, _ptr(s))
    return s


def smooth_scales(s: np.ndarray, W: np.ndarray, alpha: float) -> np.ndarray:
    """lambda_j = s_j^alpha / max_i |W_ij|^(1 - alpha)  (W is [N, K])."""
    s = _c(s, np.float32)
    W = _c(W, np.float32)
    N, K = W.shape
    lam = np.empty(K, dtype=np.float32)
    _load().oracle_smooth_scales(_ptr(s), _ptr(W), N, K, float(alpha), _ptr(lam))
    return lam


def quantize_weights(W: np.ndarray, lam: np.ndarray | None):
    """Per-output-row symmetric INT8 of W diag(lambda): returns (Wq, sw)."""
    W = _c(W, np.float32)
    lam = _c(lam, np.float32)
    N, K = W.shape
    Wq = np.empty((N, K), dtype=np.int8)
    sw = np.empty(N, dtype=np.float32)
    _load().oracle_quantize_weights(_ptr(W), _ptr(lam), N, K, _ptr(Wq), _ptr(sw))
    return Wq, sw


def quant_act(X_bf16: np.ndarray, lam: np.ndarray | None):
    """Per-token dynamic INT8 of X diag(lambda)^-1: returns (Xq, sx)."""
    X = _c(X_bf16, np.uint16)
    lam = _c(lam, np.float32)
    M, K = X.shape
    Xq = np.empty((M, K), dtype=np.int8)
    sx = np.empty(M, dtype=np.float32)
    tmp = np.empty(K, dtype=np.float32)
    _load().oracle_quant_act(_ptr(X), _ptr(lam), M, K, _ptr(Xq), _ptr(sx), _ptr(tmp))
    return Xq, sx


def gemm_i32(Xq: np.ndarray, Wq: np.ndarray, rows: tuple[int, int] | None = None):
    """Exact acc = Xq Wq^T (int32) for the rows [m0, m1) of Xq."""
    Xq = _c(Xq, np.int8)
    Wq = _c(Wq, np.int8)
    M, K = Xq.shape
    N, K2 = Wq.shape
    assert K == K2
    m0, m1 = rows if rows is not None else (0, M)
    acc = np.empty((m1 - m0, N), dtype=np.int32)
    _load().oracle_gemm_i32(_ptr(Xq), _ptr(Wq), M, N, K, m0, m1, _ptr(acc))
    return acc


def epilogue(acc: np.ndarray, sx: np.ndarray, sw: np.ndarray, bias: np.ndarray | None):
    """y = bf16_rne(((float)acc * sx_m) * sw_n + b_n), as uint16 bit patterns."""
    acc = _c(acc, np.int32)
    sx = _c(sx, np.float32)
    sw = _c(sw, np.float32)
    bias = _c(bias, np.float32)
    rows, N = acc.shape
    Y = np.empty((rows, N), dtype=np.uint16)
    _load().oracle_epilogue(_ptr(acc), _ptr(sx), _ptr(sw), _ptr(bias), rows, N, _ptr(Y))
    return Y


def linear(Xq, sx, Wq, sw, bias, rows: tuple[int, int] | None = None):
    """Quantized linear a4+a5 for rows [m0, m1): bf16 bit patterns [m1-m0, N]."""
    Xq = _c(Xq, np.int8)
    Wq = _c(Wq, np.int8)
    sx = _c(sx, np.float32)
    sw = _c(sw, np.float32)
    bias = _c(bias, np.float32)
    M, K = Xq.shape
    N = Wq.shape[0]
    m0, m1 = rows if rows is not None else (0, M)
    acc = np.empty((m1 - m0, N), dtype=np.int32)
    Y = np.empty((m1 - m0, N), dtype=np.uint16)
    _load().oracle_linear_rows(_ptr(Xq), _ptr(sx), _ptr(Wq), _ptr(sw), _ptr(bias),
                               M, N, K, m0, m1, _ptr(acc), _ptr(Y))
    return Y


def linear_dual(branches, rows=None):
    """The dual-branch layer is the single-branch layer applied to each branch."""
    return [linear(*br, rows=rows) for br in branches]


def full_layer(X_bf16, W, bias, s, alpha):
    """Offline a1+a2, then per-call a3+a4+a5; returns a dict of every stage."""
    lam = smooth_scales(s, W, alpha)
    Wq, sw = quantize_weights(W, lam)
    Xq, sx = quant_act(X_bf16, lam)
    Y = linear(Xq, sx, Wq, sw, bias)
    return {"lambda": lam, "Wq": Wq, "sw": sw, "Xq": Xq, "sx": sx, "Y": Y}


# --------------------------------------------------------------------------
# ablation arm: per-tensor activation scale (Sec. 5, "What drives INT8
# recovery"; the naive per-tensor INT8 of Sec. 2)
# --------------------------------------------------------------------------

def quant_act_per_tensor(X_bf16: np.ndarray, lam: np.ndarray | None):
    """One INT8 scale for all of X diag(lambda)^-1: returns (Xq, sx [M], amax)."""
    X = _c(X_bf16, np.uint16)
    lam = _c(lam, np.float32)
    M, K = X.shape
    Xq = np.empty((M, K), dtype=np.int8)
    sx = np.empty(M, dtype=np.float32)
    amax = np.empty(1, dtype=np.float32)
    tmp = np.empty(K, dtype=np.float32)
    _load().oracle_quant_act_per_tensor(_ptr(X), _ptr(lam), M, K, _ptr(Xq), _ptr(sx),
                                        _ptr(amax), _ptr(tmp))
    return Xq, sx, float(amax[0])


# --------------------------------------------------------------------------
# fragility profiling and protection (Sec. 3, "Activation-fragility
# profiling and protection")
# --------------------------------------------------------------------------

def act_stats(X_bf16: np.ndarray):
    """(per-channel [4, K], whole-tensor [4]) of maxabs, mean, std, kurtosis
    over the rows of a [T, K] bf16 batch, in binary64."""
    X = _c(X_bf16, np.uint16)
    T, K = X.shape
    chan = np.empty((4, K), dtype=np.float64)
    tensor = np.empty(4, dtype=np.float64)
    _load().oracle_act_stats(_ptr(X), T, K, _ptr(chan), _ptr(tensor))
    return chan, tensor


def shifted_power_sums(X_bf16: np.ndarray, shift: np.ndarray | None):
    """(S, A) [4, K]: S[p-1, j] = sum_t (x_tj - c_j)^p and A the same over |.|."""
    X = _c(X_bf16, np.uint16)
    shift = _c(shift, np.float32)
    T, K = X.shape
    S = np.empty((4, K), dtype=np.float64)
    A = np.empty((4, K), dtype=np.float64)
    _load().oracle_shifted_power_sums(_ptr(X), T, K, _ptr(shift), _ptr(S), _ptr(A))
    return S, A


def linear_bf16(X_bf16, W_bf16, bias, rows: tuple[int, int] | None = None):
    """Protected layer, rows [m0, m1): (y, yabs) in binary64, y = X W^T + b exactly
    up to binary64 summation, yabs = sum |x w| + |b|."""
    X = _c(X_bf16, np.uint16)
    W = _c(W_bf16, np.uint16)
    bias = _c(bias, np.float32)
    M, K = X.shape
    N = W.shape[0]
    m0, m1 = rows if rows is not None else (0, M)
    Y = np.empty((m1 - m0, N), dtype=np.float64)
    Ya = np.empty((m1 - m0, N), dtype=np.float64)
    _load().oracle_linear_bf16_rows(_ptr(X), _ptr(W), _ptr(bias), M, N, K, m0, m1,
                                    _ptr(Y), _ptr(Ya))
    return Y, Ya


def layer_forward(X_bf16, layer: dict, rows: tuple[int, int] | None = None):
    """Per-layer dispatch: a protected layer is the bf16 linear (no activation
    quantization); any other layer is a3 + a4 + a5.  Returns the bf16 result
    for W8A8 layers (bit patterns) or the binary64 (y, yabs) pair for
    protected ones."""
    if layer["protect"]:
        return linear_bf16(X_bf16, layer["W_bf16"], layer["bias"], rows=rows)
    Xq, sx = quant_act(X_bf16, layer["smooth"])
    return linear(Xq, sx, layer["Wq"], layer["w_scale"], layer["bias"], rows=rows)


# --------------------------------------------------------------------------
# fused neighbours of a3: both branches in one call, GELU folded in
# --------------------------------------------------------------------------

def quant_act_dual(branches):
    """The dual-branch activation quantization is a3 applied to each branch:
    branches = [(X_bf16, lam), (X_bf16, lam)] -> [(Xq, sx), (Xq, sx)]."""
    return [quant_act(X, lam) for X, lam in branches]


def gelu_value(h) -> np.ndarray:
    """fl32(GELU(h)), GELU(h) = (h/2) erfc(-h/sqrt(2)) in binary64."""
    lib = _load()
    h = np.asarray(h, dtype=np.float32)
    out = np.empty(h.shape, dtype=np.float32)
    fi, fo = h.reshape(-1), out.reshape(-1)
    for i in range(fi.size):
        fo[i] = lib.oracle_gelu_value(float(fi[i]))
    return out


def gelu_quant_act(H_bf16: np.ndarray, lam: np.ndarray | None, with_pre: bool = False):
    """Per-token INT8 of GELU(H) diag(lambda)^-1 (GELU in fp32, no bf16 rounding
    in between): returns (Xq, sx) or (Xq, sx, pre) with pre the fp32 value
    each code is rounded from."""
    H = _c(H_bf16, np.uint16)
    lam = _c(lam, np.float32)
    M, K = H.shape
    Xq = np.empty((M, K), dtype=np.int8)
    sx = np.empty(M, dtype=np.float32)
    tmp = np.empty(K, dtype=np.float32)
    row = np.empty(K, dtype=np.float32)
    pre = np.empty((M, K), dtype=np.float32) if with_pre else None
    _load().oracle_gelu_quant_act(_ptr(H), _ptr(lam), M, K, _ptr(Xq), _ptr(sx), _ptr(tmp),
                                  _ptr(row), _ptr(pre))
    return (Xq, sx, pre) if with_pre else (Xq, sx)


# --------------------------------------------------------------------------
# GGUF weight-only layer (Sec. 3, "GGUF k-quants")
# --------------------------------------------------------------------------

GGUF_Q8_0, GGUF_Q4_K = 0, 1
GGUF_BLOCK = {GGUF_Q8_0: (32, 34), GGUF_Q4_K: (256, 144)}   # weights, bytes


def f32_to_bf16_array(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (round to nearest even), any shape."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().oracle_f32_to_bf16_rne_array(_ptr(x), x.size, _ptr(out))
    return out


def f16_to_f32(h) -> np.ndarray:
    lib = _load()
    h = np.asarray(h, dtype=np.uint16)
    return np.array([lib.oracle_f16_to_f32(int(v)) for v in h.ravel()], np.float32).reshape(h.shape)


def gguf_dequant(raw: np.ndarray, fmt: int, N: int, K: int) -> np.ndarray:
    """Decode N rows of K weights from raw GGUF blocks (uint8 [N, K/QK*bytes]) to fp32."""
    qk, nbytes = GGUF_BLOCK[fmt]
    raw = np.ascontiguousarray(raw, dtype=np.uint8).reshape(N, K // qk * nbytes)
    out = np.empty((N, K), dtype=np.float32)
    fn = _load().oracle_dequant_q8_0 if fmt == GGUF_Q8_0 else _load().oracle_dequant_q4_k
    fn(_ptr(raw), N, K, _ptr(out))
    return out


def gguf_dequant_bf16(raw, fmt, N, K) -> np.ndarray:
    """The decoded weights as the layer consumes them: bf16 (nearest even)."""
    return f32_to_bf16_array(gguf_dequant(raw, fmt, N, K))


def linear_gguf(X_bf16, raw, fmt, N, bias, rows=None):
    """Weight-only layer: y = X dequant(W)^T + b with the decoded weights in
    bf16, as (y, yabs) in binary64 for rows [m0, m1)."""
    K = X_bf16.shape[1]
    return linear_bf16(X_bf16, gguf_dequant_bf16(raw, fmt, N, K), bias, rows=rows)
