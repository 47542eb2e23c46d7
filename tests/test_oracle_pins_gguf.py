"""Pins of the oracle's GGUF decoding (Sec. 3, "GGUF k-quants").

Hand-built blocks (tests/golden/handworked_gguf.json) pin the byte layout,
including the split 6-bit scales and mins of Q4_K sub-blocks 4-7; a
round-to-nearest encoder written here (independent of the oracle) pins the
decoder on random weights: decoding what it packed gives back exactly the
value its integers define.
"""

import json
import os

import numpy as np
import pytest

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "handworked_gguf.json")))


def f16_bits(x):
    return np.asarray(x, np.float16).view(np.uint16)


def f16_val(bits):
    return np.asarray(bits, np.uint16).view(np.float16).astype(np.float32)


def test_q8_0_golden(oracle_mod):
    g = GOLD["q8_0"]
    raw = np.zeros(34, np.uint8)
    raw[0:2] = np.array([g["d_f16"]], np.uint16).view(np.uint8)
    raw[2:] = np.array(g["q"], np.int8).view(np.uint8)
    w = oracle_mod.gguf_dequant(raw, oracle_mod.GGUF_Q8_0, 1, 32)[0]
    np.testing.assert_array_equal(w[:8], g["w_first8"])
    assert not w[8:].any()


def _q4k_golden_block():
    g = GOLD["q4_k"]
    raw = np.zeros(144, np.uint8)
    raw[0:2] = np.array([g["d_f16"]], np.uint16).view(np.uint8)
    raw[2:4] = np.array([g["dmin_f16"]], np.uint16).view(np.uint8)
    raw[4:16] = g["scale_bytes"]
    raw[16:] = np.arange(128, dtype=np.uint8)
    return g, raw


def test_q4_k_golden(oracle_mod):
    g, raw = _q4k_golden_block()
    w = oracle_mod.gguf_dequant(raw, oracle_mod.GGUF_Q4_K, 1, 256)[0]
    for k, v in g["spot"].items():
        assert w[int(k)] == v
    # every weight from the intended parameters (not from the bytes)
    qs = np.arange(128)
    want = np.empty(256)
    for c in range(4):
        want[64 * c:64 * c + 32] = g["d"] * g["sc"][2 * c] * (qs[32 * c:32 * c + 32] & 15) - g["dmin"] * g["m"][2 * c]
        want[64 * c + 32:64 * c + 64] = (g["d"] * g["sc"][2 * c + 1] * (qs[32 * c:32 * c + 32] >> 4)
                                         - g["dmin"] * g["m"][2 * c + 1])
    np.testing.assert_array_equal(w, want.astype(np.float32))


def test_q4_k_zero_quants_give_minus_mins(oracle_mod):
    g, raw = _q4k_golden_block()
    raw[16:] = 0
    w = oracle_mod.gguf_dequant(raw, oracle_mod.GGUF_Q4_K, 1, 256)[0]
    for j in range(8):
        np.testing.assert_array_equal(w[32 * j:32 * j + 32], np.float32(-g["dmin"] * g["m"][j]))


# ---- an independent round-to-nearest encoder (plain numpy, written here) ----

def encode_q8_0(W):
    N, K = W.shape
    blocks = W.reshape(N, K // 32, 32)
    d16 = f16_bits(np.abs(blocks).max(-1) / 127.0)
    d = f16_val(d16)
    q = np.clip(np.rint(blocks / np.where(d == 0, 1, d)[..., None]), -127, 127).astype(np.int8)
    raw = np.zeros((N, K // 32, 34), np.uint8)
    raw[..., 0:2] = d16[..., None].view(np.uint8).reshape(N, K // 32, 2)
    raw[..., 2:] = q.view(np.uint8)
    return raw.reshape(N, -1), d, q


def encode_q4_k(W):
    N, K = W.shape
    nb = K // 256
    sub = W.reshape(N, nb, 8, 32).astype(np.float64)
    mn = np.minimum(sub.min(-1), 0.0)
    scale = (sub.max(-1) - mn) / 15.0
    d = f16_val(f16_bits(scale.max(-1) / 63.0)).astype(np.float64)
    dmin = f16_val(f16_bits((-mn).max(-1) / 63.0)).astype(np.float64)
    sc = np.clip(np.rint(scale / np.where(d == 0, 1, d)[..., None]), 0, 63).astype(np.int64)
    m = np.clip(np.rint(-mn / np.where(dmin == 0, 1, dmin)[..., None]), 0, 63).astype(np.int64)
    step = d[..., None] * sc
    q = np.clip(np.rint((sub + (dmin[..., None] * m)[..., None]) / np.where(step == 0, 1, step)[..., None]),
                0, 15).astype(np.int64)
    raw = np.zeros((N, nb, 144), np.uint8)
    raw[..., 0:2] = f16_bits(d).reshape(N, nb, 1).view(np.uint8).reshape(N, nb, 2)
    raw[..., 2:4] = f16_bits(dmin).reshape(N, nb, 1).view(np.uint8).reshape(N, nb, 2)
    s = np.zeros((N, nb, 12), np.int64)
    s[..., 0:4] = sc[..., 0:4] | ((sc[..., 4:8] >> 4) << 6)
    s[..., 4:8] = m[..., 0:4] | ((m[..., 4:8] >> 4) << 6)
    s[..., 8:12] = (sc[..., 4:8] & 15) | ((m[..., 4:8] & 15) << 4)
    raw[..., 4:16] = s.astype(np.uint8)
    for c in range(4):
        raw[..., 16 + 32 * c:16 + 32 * c + 32] = (q[:, :, 2 * c, :] | (q[:, :, 2 * c + 1, :] << 4)).astype(np.uint8)
    return raw.reshape(N, -1), d, dmin, sc, m, q


def test_q8_0_round_trip(oracle_mod):
    rng = np.random.default_rng(0)
    W = (rng.standard_normal((13, 256)) * 0.02).astype(np.float32)
    raw, d, q = encode_q8_0(W)
    w = oracle_mod.gguf_dequant(raw, oracle_mod.GGUF_Q8_0, 13, 256)
    want = (d[..., None] * q.astype(np.float32)).reshape(13, 256)
    np.testing.assert_array_equal(w, want)
    assert np.all(np.abs(w - W) <= np.repeat(d, 32, axis=1) * 0.5 + 1e-9)


def test_q4_k_round_trip(oracle_mod):
    rng = np.random.default_rng(1)
    W = (rng.standard_normal((11, 512)) * 0.02).astype(np.float32)
    W[3, 300] = 0.3                                   # an outlier weight
    raw, d, dmin, sc, m, q = encode_q4_k(W)
    w = oracle_mod.gguf_dequant(raw, oracle_mod.GGUF_Q4_K, 11, 512)
    d32 = d.astype(np.float32)[..., None, None]
    dm32 = dmin.astype(np.float32)[..., None, None]
    want = ((d32 * sc.astype(np.float32)[..., None]) * q.astype(np.float32)
            - (dm32 * m.astype(np.float32)[..., None]))
    np.testing.assert_array_equal(w, want.reshape(11, 512).astype(np.float32))
    rel = np.sqrt(np.mean((w - W) ** 2) / np.mean(W ** 2))
    assert rel < 0.15                                  # 4-bit round to nearest


def test_gguf_linear_uses_bf16_weights(oracle_mod):
    rng = np.random.default_rng(2)
    W = (rng.standard_normal((5, 256)) * 0.02).astype(np.float32)
    raw = encode_q8_0(W)[0]
    X = (np.arange(3 * 256, dtype=np.uint32).reshape(3, 256) % 7 + 0x3f80).astype(np.uint16)
    y, _ = oracle_mod.linear_gguf(X, raw, oracle_mod.GGUF_Q8_0, 5, None)
    Wb = oracle_mod.gguf_dequant_bf16(raw, oracle_mod.GGUF_Q8_0, 5, 256)
    y2, _ = oracle_mod.linear_bf16(X, Wb, None)
    np.testing.assert_array_equal(y, y2)
    # the bf16 rounding of the decoded weights is round to nearest even
    w32 = oracle_mod.gguf_dequant(raw, oracle_mod.GGUF_Q8_0, 5, 256)
    back = (Wb.astype(np.uint32) << 16).view(np.float32)
    assert np.all(np.abs(back - w32) <= np.spacing(np.abs(back).astype(np.float32)) * 2 ** 15)
