// common.cuh -- small device helpers shared by the library's CUDA sources.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/w8a8.h"

namespace w8a8 {

// bf16 bit pattern -> fp32 (exact).
__device__ __forceinline__ float bf16_bits_to_f32(uint32_t h16) {
    return __uint_as_float(h16 << 16);
}

// fp32 -> bf16 bit pattern, round to nearest even (NaN stays a quiet NaN).
__device__ __forceinline__ uint32_t f32_to_bf16_bits_rn(float t) {
    uint32_t u = __float_as_uint(t);
    if ((u & 0x7fffffffu) > 0x7f800000u) return (u >> 16) | 0x40u;
    return (u + 0x7fffu + ((u >> 16) & 1u)) >> 16;
}

// clamp(round_half_even(v), -127, 127); NaN -> 0.
__device__ __forceinline__ int quantize_rne_clamp(float v) {
    if (v != v) return 0;
    float r = rintf(v);  // round to nearest, ties to even
    r = fminf(fmaxf(r, -127.0f), 127.0f);
    return static_cast<int>(r);
}

// Two fp32 -> one bf16x2 word (lo in bits 0-15), both rounded to nearest
// even by one conversion instruction: the same bits as two
// f32_to_bf16_bits_rn calls for every input that is not a NaN (a GPU test
// checks all 2^32 patterns in each half); a NaN becomes the canonical one
// instead of keeping its payload, so callers use it only where no value can
// be a NaN.
__device__ __forceinline__ uint32_t pack_bf16x2_cvt(float lo, float hi) {
    uint32_t w;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(w) : "f"(hi), "f"(lo));
    return w;
}

// The epilogue's value before the rounding to bf16: (t * sx) * sw + b, each
// step rounded to nearest even, no contraction.
__device__ __forceinline__ float epilogue_f32(float t, float sx, float sw, float b, bool has_bias) {
    t = __fmul_rn(t, sx);
    t = __fmul_rn(t, sw);
    if (has_bias) t = __fadd_rn(t, b);
    return t;
}

// Dequantizing epilogue for one output from the int32 accumulator:
// bf16(((float)acc * sx) * sw + b), each step rounded to nearest even.
__device__ __forceinline__ uint32_t epilogue_value(int32_t acc, float sx, float sw,
                                                   float b, bool has_bias) {
    return f32_to_bf16_bits_rn(epilogue_f32(__int2float_rn(acc), sx, sw, b, has_bias));
}

constexpr int kMaxK = W8A8_MAX_K;

}  // namespace w8a8
