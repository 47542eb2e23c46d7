// quant.cu -- the quantization passes of the W8A8 layer (Sec. 3, "INT8 W8A8").
//
//   act_quant_team_kernel a3 per-token activation quant (bf16 in, x / lambda),
//                         the per-call HBM-bound pass (K <= 16384)
//   row_quant_kernel      a2 per-output-channel weight quant (fp32 in,
//                         w * lambda), offline; also a3 for K > 16384 through
//   row_quant_long_kernel the two-pass variant for very long rows
//   col_absmax_kernel     column max |.| of a row-major matrix: the calibration
//                         statistic s_j and the weight column max m_j of a1
//   smooth_finalize       a1 lambda_j = s_j^alpha / m_j^(1-alpha)
//
// In row_quant_kernel a "team" of G threads owns one row at a time; each
// thread owns CPT chunks of 8 consecutive columns at a stride of 8*G columns,
// so every warp-wide load is a fully coalesced segment, and keeps its
// per-column factors (1/lambda_j or lambda_j) in registers for every row.
#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"
#include "host_once.h"
#include "launch.h"

namespace w8a8 {
namespace {

// ---------------------------------------------------------------- loading

template <typename InT> struct Chunk;

template <> struct Chunk<uint16_t> {        // 8 bf16 = 16 bytes
    uint4 v;
    __device__ __forceinline__ void load(const uint16_t *p) {
        v = __ldcs(reinterpret_cast<const uint4 *>(p));
    }
    __device__ __forceinline__ void zero() { v = make_uint4(0, 0, 0, 0); }
    __device__ __forceinline__ uint32_t bits(int e) const {
        uint32_t w = (e < 2) ? v.x : (e < 4) ? v.y : (e < 6) ? v.z : v.w;
        return (e & 1) ? (w >> 16) : (w & 0xffffu);
    }
    __device__ __forceinline__ float get(int e) const { return bf16_bits_to_f32(bits(e)); }
};

template <> struct Chunk<float> {           // 8 fp32 = 32 bytes
    float4 a, b;
    __device__ __forceinline__ void load(const float *p) {
        a = __ldcs(reinterpret_cast<const float4 *>(p));
        b = __ldcs(reinterpret_cast<const float4 *>(p) + 1);
    }
    __device__ __forceinline__ void zero() {
        a = make_float4(0.f, 0.f, 0.f, 0.f);
        b = a;
    }
    __device__ __forceinline__ float get(int e) const {
        switch (e) {
            case 0: return a.x; case 1: return a.y; case 2: return a.z;
            case 3: return a.w; case 4: return b.x; case 5: return b.y;
            case 6: return b.z; default: return b.w;
        }
    }
};

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ uint64_t pk(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}

__device__ __forceinline__ float2 upk(uint64_t v) {
    float2 r;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
    return r;
}

__device__ __forceinline__ uint64_t fma_pk(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

__device__ __forceinline__ uint64_t add_pk(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

}  // namespace

// GELU(h) = h Phi(h) = (h/2) erfc(-h/sqrt 2), the exact (erf) form, for the
// FFN down-projection input.  The fused pass only ever evaluates it at bf16
// inputs, so it reads a table holding, for each of the 65536 bf16 bit
// patterns, the value evaluated in binary64 and rounded once to fp32: exact
// as defined, no approximation.  The table (256 KB) is built on each device
// the first time a GELU pass runs there (build_gelu_table below) and then
// only read.
__device__ float g_gelu_table[65536];

namespace {

__global__ void gelu_table_kernel() {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < 65536) {
        const double x = static_cast<double>(__uint_as_float(static_cast<uint32_t>(i) << 16));
        g_gelu_table[i] = __double2float_rn(0.5 * x * erfc(-x / sqrt(2.0)));
    }
}

// GELU of a bf16 bit pattern (the table holds every one).
__device__ __forceinline__ float gelu_of_bits(uint32_t h16) { return __ldg(&g_gelu_table[h16 & 0xffffu]); }

cudaError_t build_gelu_table();

// The hot range of the table, |h| in [2^-10, 2^5) (bf16 patterns 0x3A80 ..
// 0x41FF and their negatives: 15 KB), which a block copies into shared
// memory; values outside it (rare) read the global table.
constexpr uint32_t kGeluLo = 0x3A80u, kGeluN = 0x4200u - 0x3A80u;

// GELU of the 8 bf16 values of a chunk (word q holds columns 2q, 2q+1, the
// low half first).  Each value's table index is computed without a branch
// (a value outside the hot range reads entry 0 for now), the 8 lookups go
// out together, and only a chunk holding a value outside the range (rare)
// takes the branch that reads those from the global table: a branch per
// value cost more issue slots than the lookups themselves.
__device__ __forceinline__ void gelu_chunk(const float *tab, const uint32_t (&wd)[4], float2 (&out)[4]) {
    uint32_t h[8], idx[8];
    bool all_hot = true;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        h[e] = (e & 1) ? (wd[e >> 1] >> 16) : (wd[e >> 1] & 0xffffu);
        const uint32_t t = (h[e] & 0x7fffu) - kGeluLo;      // wraps below the range
        const bool hot = t < kGeluN;
        all_hot = all_hot && hot;
        idx[e] = hot ? t + (h[e] >> 15) * kGeluN : 0u;
    }
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = tab[idx[e]];
    if (!all_hot) {
#pragma unroll
        for (int e = 0; e < 8; ++e)
            if ((h[e] & 0x7fffu) - kGeluLo >= kGeluN) v[e] = gelu_of_bits(h[e]);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) out[q] = make_float2(v[2 * q], v[2 * q + 1]);
}

// Element e of a chunk as the pass reads it: the value, or GELU of it.
template <bool GELU, typename C>
__device__ __forceinline__ float input_value(const C &ch, int e) {
    if constexpr (GELU) return gelu_of_bits(ch.bits(e));
    else return ch.get(e);
}

// ------------------------------------------------------------- row quant
//
// IS_ACT:  factor f_j = 1/lambda_j (activations are divided by lambda);
// else:    factor f_j = lambda_j   (weights are multiplied by lambda).
// Smoothed value x'_j = in_j * f_j (RN), absmax over the row, scale = a/127,
// codes = clamp(rne(x'_j * (127/a)), +-127).
template <typename InT, bool IS_ACT, int CPT>
__global__ void __launch_bounds__(512)
row_quant_kernel(const InT *__restrict__ in, const float *__restrict__ lam,
                 int M, int K, int G, int8_t *__restrict__ q,
                 float *__restrict__ scale) {
    __shared__ float red[2][32];
    const int tid = threadIdx.x;
    const int teams = blockDim.x / G;
    const int team = tid / G;
    const int tl = tid - team * G;          // index inside the team
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int team_warp0 = (team * G) >> 5;
    const int team_warps = G >> 5;

    // per-column factors, once per thread
    float f[CPT][8];
#pragma unroll
    for (int c = 0; c < CPT; ++c) {
        const int col0 = 8 * (tl + c * G);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            float fe = 1.0f;
            if (lam != nullptr && col0 < K) {
                const float l = __ldg(lam + col0 + e);
                fe = IS_ACT ? __frcp_rn(l) : l;
            }
            f[c][e] = fe;
        }
    }

    Chunk<InT> cur[CPT], nxt[CPT];
    const int row_stride = gridDim.x * teams;
    int row = blockIdx.x * teams + team;
#pragma unroll
    for (int c = 0; c < CPT; ++c) {
        const int col0 = 8 * (tl + c * G);
        if (row < M && col0 < K) cur[c].load(in + (size_t)row * K + col0);
        else cur[c].zero();
    }

    int parity = 0;
    for (int base = blockIdx.x * teams; base < M; base += row_stride) {
        row = base + team;
        const int nrow = row + row_stride;
        // prefetch the next row this team will visit
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
            const int col0 = 8 * (tl + c * G);
            if (IS_ACT && nrow < M && col0 < K) nxt[c].load(in + (size_t)nrow * K + col0);
            else nxt[c].zero();
        }
        // row absmax of the smoothed values
        float a = 0.0f;
#pragma unroll
        for (int c = 0; c < CPT; ++c)
#pragma unroll
            for (int e = 0; e < 8; ++e)
                a = fmaxf(a, fabsf(__fmul_rn(cur[c].get(e), f[c][e])));
        a = warp_max(a);
        if (G > 32) {
            if (lane == 0) red[parity][warp] = a;
            __syncthreads();
            a = 0.0f;
            for (int w = 0; w < team_warps; ++w) a = fmaxf(a, red[parity][team_warp0 + w]);
            parity ^= 1;
        }
        if (row < M) {
            const bool zero_row = (a == 0.0f);
            const float inv = zero_row ? 0.0f : __fdiv_rn(127.0f, a);
            if (tl == 0) scale[row] = zero_row ? 0.0f : __fdiv_rn(a, 127.0f);
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col0 = 8 * (tl + c * G);
                if (col0 >= K) continue;
                uint32_t lo = 0, hi = 0;
                if (!zero_row) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float xs = __fmul_rn(cur[c].get(e), f[c][e]);
                        const uint32_t b = static_cast<uint32_t>(quantize_rne_clamp(__fmul_rn(xs, inv))) & 0xffu;
                        if (e < 4) lo |= b << (8 * e);
                        else hi |= b << (8 * (e - 4));
                    }
                }
                *reinterpret_cast<uint2 *>(q + (size_t)row * K + col0) = make_uint2(lo, hi);
            }
        }
        if (IS_ACT) {
#pragma unroll
            for (int c = 0; c < CPT; ++c) cur[c] = nxt[c];
        } else {
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col0 = 8 * (tl + c * G);
                if (nrow < M && col0 < K) cur[c].load(in + (size_t)nrow * K + col0);
                else cur[c].zero();
            }
        }
    }
}

// Rows too long to hold in registers (K > 4 * 512 * 8 = 16384): two passes
// over the row, one for the absmax and one for the codes.  One block of 512
// threads per row at a time.
template <typename InT, bool IS_ACT, bool GELU = false>
__global__ void __launch_bounds__(512)
row_quant_long_kernel(const InT *__restrict__ in, const float *__restrict__ lam,
                      int M, int K, int8_t *__restrict__ q,
                      float *__restrict__ scale) {
    __shared__ float red[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int row = blockIdx.x; row < M; row += gridDim.x) {
        const InT *r = in + (size_t)row * K;
        float a = 0.0f;
        for (int col0 = 8 * tid; col0 < K; col0 += 8 * blockDim.x) {
            Chunk<InT> ch;
            ch.load(r + col0);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float fe = 1.0f;
                if (lam) { const float l = __ldg(lam + col0 + e); fe = IS_ACT ? __frcp_rn(l) : l; }
                a = fmaxf(a, fabsf(__fmul_rn(input_value<GELU>(ch, e), fe)));
            }
        }
        a = warp_max(a);
        if (lane == 0) red[warp] = a;
        __syncthreads();
        a = 0.0f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) a = fmaxf(a, red[w]);
        __syncthreads();
        const bool zero_row = (a == 0.0f);
        const float inv = zero_row ? 0.0f : __fdiv_rn(127.0f, a);
        if (tid == 0) scale[row] = zero_row ? 0.0f : __fdiv_rn(a, 127.0f);
        for (int col0 = 8 * tid; col0 < K; col0 += 8 * blockDim.x) {
            Chunk<InT> ch;
            ch.load(r + col0);
            uint32_t lo = 0, hi = 0;
            if (!zero_row) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    float fe = 1.0f;
                    if (lam) { const float l = __ldg(lam + col0 + e); fe = IS_ACT ? __frcp_rn(l) : l; }
                    const float xs = __fmul_rn(input_value<GELU>(ch, e), fe);
                    const uint32_t b = static_cast<uint32_t>(quantize_rne_clamp(__fmul_rn(xs, inv))) & 0xffu;
                    if (e < 4) lo |= b << (8 * e);
                    else hi |= b << (8 * (e - 4));
                }
            }
            *reinterpret_cast<uint2 *>(q + (size_t)row * K + col0) = make_uint2(lo, hi);
        }
    }
}

int num_sms() { return device_sms(); }

template <typename InT, bool IS_ACT, int CPT>
cudaError_t launch_row_quant_cpt(const InT *in, const float *lam, int M, int K, int G,
                                 int8_t *q, float *scale, cudaStream_t st) {
    const int block = G < 256 ? 256 : G;
    const int teams = block / G;
    const int groups = (M + teams - 1) / teams;
    static PerDevice<int> setup[2];            // block = 256 or 512
    int per_sm = 1;
    cudaError_t e = setup[block == 256 ? 0 : 1].get([&](int &v) {
        cudaError_t r = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, row_quant_kernel<InT, IS_ACT, CPT>,
                                                                      block, 0);
        if (v < 1) v = 1;
        return r;
    }, &per_sm);
    if (e != cudaSuccess) return e;
    int grid = num_sms() * per_sm;
    if (grid > groups) grid = groups;
    if (grid < 1) grid = 1;
    row_quant_kernel<InT, IS_ACT, CPT><<<grid, block, 0, st>>>(in, lam, M, K, G, q, scale);
    return cudaGetLastError();
}

// Team size: the smallest power of two in [32, 512] that covers the row in at
// most 4 chunks of 8 per thread; longer rows take the two-pass kernel.
template <typename InT, bool IS_ACT>
cudaError_t launch_row_quant(const InT *in, const float *lam, int M, int K,
                             int8_t *q, float *scale, cudaStream_t st) {
    const int chunks = K / 8;
    int G = 32;
    while (G < 512 && G * 4 < chunks) G *= 2;
    const int cpt = (chunks + G - 1) / G;
    if (cpt <= 1) return launch_row_quant_cpt<InT, IS_ACT, 1>(in, lam, M, K, G, q, scale, st);
    if (cpt <= 2) return launch_row_quant_cpt<InT, IS_ACT, 2>(in, lam, M, K, G, q, scale, st);
    if (cpt <= 4) return launch_row_quant_cpt<InT, IS_ACT, 4>(in, lam, M, K, G, q, scale, st);
    int g2 = num_sms() * 2;
    if (g2 > M) g2 = M;
    row_quant_long_kernel<InT, IS_ACT><<<g2, 512, 0, st>>>(in, lam, M, K, q, scale);
    return cudaGetLastError();
}

// Low byte of the fp32 sum 1.5*2^23 + y is round_half_even(y) in two's
// complement whenever |y| < 2^22: the sum lies in [2^23, 2^24), where the
// spacing of fp32 is exactly 1, so the addition itself rounds y to the nearest
// integer, ties to even.
constexpr float kRoundMagic = 12582912.0f;

// Packed fp32 multiply, round to nearest even.  Only used where no add
// follows: a packed multiply followed by a packed add was observed to lose the
// intermediate rounding (the quantized codes then differed at exact ties), so
// the rounding step below uses scalar __fmul_rn / __fadd_rn, which are never
// contracted.
__device__ __forceinline__ float2 mul2_rn(float2 a, float2 b) {
    float2 r;
    asm("{\n.reg .b64 ra, rb, rr;\nmov.b64 ra, {%2, %3};\nmov.b64 rb, {%4, %5};\n"
        "mul.rn.f32x2 rr, ra, rb;\nmov.b64 {%0, %1}, rr;\n}"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ uint32_t pack4_low_bytes(float a, float b, float c, float d) {
    const uint32_t ab = __byte_perm(__float_as_uint(a), __float_as_uint(b), 0x0040);
    const uint32_t cd = __byte_perm(__float_as_uint(c), __float_as_uint(d), 0x0040);
    return __byte_perm(ab, cd, 0x5410);
}

// ---------------------------------------------- activation quant, warp teams
//
// a3 with a team of TW warps per token row.  Every warp always owns the same
// columns of the row (U chunks of 8 values per lane, chunk c = (u*TW + w)*32
// + lane), so each lane computes its 8U factors 1/lambda_j once and keeps
// them in registers for every row it visits, and keeps the smoothed values x'
// in registers between the absmax and the quantization.  The bytes in flight
// that HBM needs come from a per-warp ring of S row slices in shared memory
// filled with cp.async (each lane reads back only the 16-byte chunks it
// copied, so no block-level synchronisation is needed); the team combines its
// warps' maxima through one named barrier per row.  Loads and stores are 512
// B per warp instruction.
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void *src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(valid ? 16 : 0) : "memory");
}

struct ActBranch {
    const uint16_t *X;
    const float *lam;
    int8_t *Xq;
    float *x_scale;
    int M;
    uint32_t *sumsq;      // fp16-code variant, optional: sum of the row's squared codes
};

// One launch covers up to two independent row sets (the conditional and
// unconditional branches): teams [0, teams0) of the grid take branch 0, the
// others branch 1, so every team keeps one branch's 1/lambda in registers.
struct ActParams {
    ActBranch br[2];
    int K;
    int teams0;
};

// two fp32 -> one f16x2 word (low = a), each rounded to nearest even (exact
// for the integer codes |q| <= 127)
__device__ __forceinline__ uint32_t pack_f16(float a, float b) {
    uint32_t r;
    asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(b), "f"(a));
    return r;
}

// The codes of one chunk of 8 smoothed values x' (x[q] = columns 2q, 2q+1)
// with inv = 127/a: int8 bytes packed in .x/.y, or (OUT16) fp16 values in
// .x .. .w.  OUT16 with want_ss adds the squared codes: exactly, as fp32
// pairs in ssq on the fast path (integers below 2^24: a lane's U <= 4 chunks
// give at most 4U codes of at most 127^2 per component) or as integers in ss.
template <bool OUT16>
__device__ __forceinline__ uint4 quant_chunk(const float2 (&x)[4], float inv, bool zero_row, bool fast,
                                             bool want_ss, uint32_t &ss, uint64_t &ssq) {
    uint4 o = make_uint4(0u, 0u, 0u, 0u);
    if (zero_row) return o;
    if (OUT16) {
        uint32_t hw[4];
        if (fast) {
            // rne(x' * inv) as an fp32 integer: the product rounded once
            // (scalar multiplies, never fused), the magic sum (in [2^23,
            // 2^24], where one packed add rounds both values to integers as
            // the scalar add would), minus the magic (exact)
            const uint64_t magic = pk(kRoundMagic, kRoundMagic);
            const uint64_t nmagic = pk(-kRoundMagic, -kRoundMagic);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint64_t c = add_pk(add_pk(pk(__fmul_rn(x[q].x, inv), __fmul_rn(x[q].y, inv)), magic), nmagic);
                const float2 cf = upk(c);
                hw[q] = pack_f16(cf.x, cf.y);
                if (want_ss) ssq = fma_pk(c, c, ssq);
            }
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int q0 = quantize_rne_clamp(__fmul_rn(x[q].x, inv));
                const int q1 = quantize_rne_clamp(__fmul_rn(x[q].y, inv));
                hw[q] = pack_f16(static_cast<float>(q0), static_cast<float>(q1));
                ss += static_cast<uint32_t>(q0 * q0 + q1 * q1);
            }
        }
        return make_uint4(hw[0], hw[1], hw[2], hw[3]);
    }
    uint32_t word[2] = {0u, 0u};
    if (fast) {
        // the products rounded once (scalar multiplies), their magic sums two
        // at a time (one packed add, each value rounded to an integer as the
        // scalar add would)
        const uint64_t magic = pk(kRoundMagic, kRoundMagic);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const float2 s0 = upk(add_pk(pk(__fmul_rn(x[2 * h].x, inv), __fmul_rn(x[2 * h].y, inv)), magic));
            const float2 s1 = upk(add_pk(pk(__fmul_rn(x[2 * h + 1].x, inv), __fmul_rn(x[2 * h + 1].y, inv)), magic));
            word[h] = pack4_low_bytes(s0.x, s0.y, s1.x, s1.y);
        }
    } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float xv = (e & 1) ? x[e >> 1].y : x[e >> 1].x;
            const uint32_t q8 = static_cast<uint32_t>(quantize_rne_clamp(__fmul_rn(xv, inv))) & 0xffu;
            word[e >> 2] |= q8 << (8 * (e & 3));
        }
    }
    o.x = word[0];
    o.y = word[1];
    return o;
}

// OUT16: the codes are written as fp16 values (uint16 bit patterns, 2 bytes
// each) instead of int8, for the GEMM that takes A without converting it.
template <int U, int TW, int S, bool GELU, bool OUT16>
__global__ void __launch_bounds__(TW > 8 ? 32 * TW : 256)
act_quant_team_kernel(const __grid_constant__ ActParams p) {
    // a dependent GEMM launched programmatically may set itself up on SMs as
    // they free up; it reads nothing of this pass before the pass completes
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    constexpr int kThreads = TW > 8 ? 32 * TW : 256;
    constexpr int kTeams = kThreads / (32 * TW);
    extern __shared__ __align__(16) uint4 ring_s[];
    __shared__ float red[2][kThreads / 32];
    __shared__ uint32_t sred[2][kThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int team = warp / TW, tw = warp % TW;
    const int K = p.K;
    const int cpr = K / 8;                                  // 16-byte chunks per row
    const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(ring_s)) +
                          static_cast<uint32_t>((warp * S * U * 32 + lane) * 16);

    // GELU: the hot range of the table in shared memory (see gelu_chunk)
    __shared__ float gtab[GELU ? 2 * kGeluN : 1];
    const int gteam = blockIdx.x * kTeams + team;
    const bool second = gteam >= p.teams0;
    const ActBranch b = second ? p.br[1] : p.br[0];
    const uint16_t *__restrict__ X = b.X;
    const int M = b.M;
    const int teams = second ? gridDim.x * kTeams - p.teams0 : p.teams0;
    const int first = second ? gteam - p.teams0 : gteam;
    auto issue = [&](int k) {                               // row slice k of this team -> slot k % S
        const int row = first + k * teams;
        const uint32_t slot = ring + static_cast<uint32_t>((k % S) * U * 32 * 16);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int c = (u * TW + tw) * 32 + lane;
            const bool ok = row < M && c < cpr;
            cp_async_16(slot + u * 32 * 16, ok ? (const void *)(X + (size_t)row * K + 8 * c) : (const void *)X, ok);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
#pragma unroll
    for (int k = 0; k < S - 1; ++k) issue(k);           // first rows in flight before the setup

    if (GELU) {
        for (int i = tid; i < static_cast<int>(2 * kGeluN); i += kThreads)
            gtab[i] = __ldg(&g_gelu_table[i < static_cast<int>(kGeluN) ? kGeluLo + i
                                                                       : 0x8000u + kGeluLo + (i - kGeluN)]);
        __syncthreads();
    }
    float2 r[U][4];                                         // 1/lambda of this lane's columns
#pragma unroll
    for (int u = 0; u < U; ++u) {
        const int c = (u * TW + tw) * 32 + lane;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            float f0 = 1.0f, f1 = 1.0f;
            if (b.lam != nullptr && c < cpr) {
                f0 = __frcp_rn(__ldg(b.lam + 8 * c + 2 * q));
                f1 = __frcp_rn(__ldg(b.lam + 8 * c + 2 * q + 1));
            }
            r[u][q] = make_float2(f0, f1);
        }
    }

    // OUT16: the squared codes of a row are summed (exactly, in int32: at most
    // 16384 * 127^2 < 2^31) for the GEMM's bound on its partial sums; the
    // team's per-warp sums of row k are combined after row k + 1's barrier
    const bool want_ss = OUT16 && b.sumsq != nullptr;
    int parity = 0, prev_row = -1;
    for (int k = 0;; ++k, parity ^= 1) {
        const int row = first + k * teams;                  // uniform across the team
        if (row >= M) break;
        issue(k + S - 1);
        asm volatile("cp.async.wait_group %0;" ::"n"(S - 1) : "memory");
        const uint32_t slot = ring + static_cast<uint32_t>((k % S) * U * 32 * 16);
        float2 xs[U][4];
        float a = 0.0f;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            uint4 v;
            asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                         : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(slot + u * 32 * 16));
            const uint32_t wd[4] = {v.x, v.y, v.z, v.w};
            if (GELU) {
                gelu_chunk(gtab, wd, xs[u]);
            } else {
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    xs[u][q] = make_float2(__uint_as_float(wd[q] << 16), __uint_as_float(wd[q] & 0xffff0000u));
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                xs[u][q] = mul2_rn(xs[u][q], r[u][q]);
                a = fmaxf(a, fmaxf(fabsf(xs[u][q].x), fabsf(xs[u][q].y)));
            }
        }
        a = warp_max(a);
        if (TW > 1) {
            if (lane == 0) red[parity][warp] = a;
            asm volatile("bar.sync %0, %1;" ::"r"(1 + team), "r"(TW * 32) : "memory");
#pragma unroll
            for (int w = 0; w < TW; ++w) a = fmaxf(a, red[parity][team * TW + w]);
            if (want_ss && prev_row >= 0 && tw == 0 && lane == 0) {
                uint32_t t = 0;
#pragma unroll
                for (int w = 0; w < TW; ++w) t += sred[parity ^ 1][team * TW + w];
                b.sumsq[prev_row] = t;
            }
        }
        const bool zero_row = (a == 0.0f);
        const float inv = zero_row ? 0.0f : __fdiv_rn(127.0f, a);
        if (tw == 0 && lane == 0) b.x_scale[row] = zero_row ? 0.0f : __fdiv_rn(a, 127.0f);
        // a and 127/a finite: |x' * inv| <= 127 (1 + 2^-23), no clamp needed
        const bool fast = (a <= 3.402823466e38f) && (inv <= 3.402823466e38f);
        uint2 *qr = reinterpret_cast<uint2 *>(b.Xq + (size_t)row * K);
        uint4 *qr16 = reinterpret_cast<uint4 *>(b.Xq + 2 * (size_t)row * K);
        uint32_t ss = 0;
        uint64_t ssq = 0;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int c = (u * TW + tw) * 32 + lane;
            if (c >= cpr) continue;
            const uint4 o = quant_chunk<OUT16>(xs[u], inv, zero_row, fast, want_ss, ss, ssq);
            if (OUT16) qr16[c] = o;
            else qr[c] = make_uint2(o.x, o.y);
        }
        if (want_ss) {
            const float2 sf = upk(ssq);
            ss += __float2uint_rn(__fadd_rn(sf.x, sf.y));
            ss = __reduce_add_sync(0xffffffffu, ss);
            if (TW > 1) {
                if (lane == 0) sred[parity][warp] = ss;
            } else if (lane == 0) {
                b.sumsq[row] = ss;
            }
            prev_row = row;
        }
    }
    if (TW > 1 && want_ss && prev_row >= 0) {
        // the last row's sums: one more team barrier
        asm volatile("bar.sync %0, %1;" ::"r"(1 + team), "r"(TW * 32) : "memory");
        if (tw == 0 && lane == 0) {
            uint32_t t = 0;
#pragma unroll
            for (int w = 0; w < TW; ++w) t += sred[parity ^ 1][team * TW + w];
            b.sumsq[prev_row] = t;
        }
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
}

template <int U, int TW, bool GELU, bool OUT16>
cudaError_t launch_act_quant_team(ActParams p, cudaStream_t st) {
    // ring depth, from timed sweeps on the workload shapes: every team has
    // S - 1 rows in flight from its start and visits only a handful of rows
    // (4608 rows on 608 teams for K = 4096), so a deeper ring only front-loads
    // the reads; 2 slices suit the 256-thread teams writing fp16 codes, 3
    // the int8 codes and the 16-warp teams of K > 8192
    constexpr int S = GELU ? 3 : ((OUT16 && TW <= 8) ? 2 : 3);
    constexpr int kThreads = TW > 8 ? 32 * TW : 256;
    constexpr int kTeams = kThreads / (32 * TW);
    constexpr size_t smem = (size_t)(kThreads / 32) * S * U * 32 * 16;
    auto kern = act_quant_team_kernel<U, TW, S, GELU, OUT16>;
    static PerDevice<int> setup;
    int per_sm = 1;
    cudaError_t e = setup.get([&](int &v) {
        // always opted in: the static reduction array counts against the
        // 48 KB default too
        cudaError_t r = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (r != cudaSuccess) return r;
        r = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, kern, kThreads, smem);
        if (v < 1) v = 1;
        return r;
    }, &per_sm);
    if (e != cudaSuccess) return e;
    const int M0 = p.br[0].M, M1 = p.br[1].M;
    int grid = num_sms() * per_sm;
    const int blocks_needed = (M0 + M1 + kTeams - 1) / kTeams;
    if (grid > blocks_needed) grid = blocks_needed;
    const bool both = M0 > 0 && M1 > 0;
    if (both && grid * kTeams < 2) grid = 2;            // at least one team per branch
    const int nteams = grid * kTeams;
    if (!both) {
        p.teams0 = M1 == 0 ? nteams : 0;
    } else {
        int t0 = static_cast<int>((static_cast<long long>(nteams) * M0 + (M0 + M1) / 2) / (M0 + M1));
        p.teams0 = t0 < 1 ? 1 : (t0 > nteams - 1 ? nteams - 1 : t0);
    }
    kern<<<grid, kThreads, smem, st>>>(p);
    return cudaGetLastError();
}

template <bool GELU, bool OUT16 = false>
cudaError_t launch_act_quant_teams(const ActParams &p, cudaStream_t st) {
    // team of TW warps per row, U chunks of 8 values per lane: K <= 256 U TW
    const int K = p.K;
    if (K <= 256) return launch_act_quant_team<1, 1, GELU, OUT16>(p, st);
    if (K <= 512) return launch_act_quant_team<2, 1, GELU, OUT16>(p, st);
    if (K <= 1024) return launch_act_quant_team<2, 2, GELU, OUT16>(p, st);
    if (K <= 2048) return launch_act_quant_team<2, 4, GELU, OUT16>(p, st);
    if (K <= 4096) return launch_act_quant_team<2, 8, GELU, OUT16>(p, st);
    if (K <= 8192) return launch_act_quant_team<2, 16, GELU, OUT16>(p, st);
    return launch_act_quant_team<4, 16, GELU, OUT16>(p, st);
}

// ----------------------------------------------------------- column absmax
//
// out_j = max_i |in_ij| over rows [0, R).  Each thread owns 8 consecutive
// columns and a slab of rows; slabs combine with an integer atomicMax on the
// bit patterns (non-negative floats order like their bit patterns).  `out`
// must be zeroed first.
template <typename InT>
__global__ void col_absmax_kernel(const InT *__restrict__ in, int R, int C,
                                  int rows_per_slab, float *__restrict__ out) {
    const int cg = blockIdx.x * blockDim.x + threadIdx.x;
    const int col0 = 8 * cg;
    if (col0 >= C) return;
    const int r0 = blockIdx.y * rows_per_slab;
    int r1 = r0 + rows_per_slab;
    if (r1 > R) r1 = R;
    float m[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) m[e] = 0.0f;
    for (int r = r0; r < r1; ++r) {
        Chunk<InT> ch;
        ch.load(in + (size_t)r * C + col0);
#pragma unroll
        for (int e = 0; e < 8; ++e) m[e] = fmaxf(m[e], fabsf(ch.get(e)));
    }
    if (r0 < r1) {
#pragma unroll
        for (int e = 0; e < 8; ++e)
            atomicMax(reinterpret_cast<unsigned int *>(out + col0 + e), __float_as_uint(m[e]));
    }
}

template <typename InT>
cudaError_t launch_col_absmax(const InT *in, int R, int C, float *out, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(out, 0, sizeof(float) * (size_t)C, st);
    if (e != cudaSuccess) return e;
    if (R <= 0) return cudaSuccess;
    const int threads = 128;
    const int gx = (C / 8 + threads - 1) / threads;
    int gy = (num_sms() * 8 + gx - 1) / gx;
    if (gy > R) gy = R;
    if (gy < 1) gy = 1;
    const int rows_per_slab = (R + gy - 1) / gy;
    gy = (R + rows_per_slab - 1) / rows_per_slab;
    col_absmax_kernel<InT><<<dim3(gx, gy), threads, 0, st>>>(in, R, C, rows_per_slab, out);
    return cudaGetLastError();
}

// lambda_j = s_j^alpha / m_j^(1-alpha), m_j already stored in lambda[j].
__global__ void smooth_finalize_kernel(const float *__restrict__ s, float alpha,
                                       int K, float *__restrict__ lambda) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= K) return;
    const float sj = s[j];
    const float m = lambda[j];
    float l;
    if (sj == 0.0f || m == 0.0f) l = 1.0f;
    else if (alpha == 0.5f) l = __fdiv_rn(__fsqrt_rn(sj), __fsqrt_rn(m));
    else if (alpha == 1.0f) l = sj;
    else if (alpha == 0.0f) l = __fdiv_rn(1.0f, m);
    else l = __double2float_rn(exp2((double)alpha * log2((double)sj) -
                                    (1.0 - (double)alpha) * log2((double)m)));
    lambda[j] = l;
}

}  // namespace

cudaError_t launch_channel_absmax(const uint16_t *X, int T, int K, float *s, cudaStream_t st) {
    return launch_col_absmax<uint16_t>(X, T, K, s, st);
}

cudaError_t launch_smooth_scales(const float *s, const float *W, int N, int K,
                                 float alpha, float *lambda, cudaStream_t st) {
    cudaError_t e = launch_col_absmax<float>(W, N, K, lambda, st);
    if (e != cudaSuccess) return e;
    smooth_finalize_kernel<<<(K + 255) / 256, 256, 0, st>>>(s, alpha, K, lambda);
    return cudaGetLastError();
}

cudaError_t launch_quantize_weights(const float *W, const float *lambda, int N, int K,
                                    int8_t *Wq, float *w_scale, cudaStream_t st) {
    return launch_row_quant<float, false>(W, lambda, N, K, Wq, w_scale, st);
}

cudaError_t launch_quant_act(const uint16_t *X, const float *lambda, int M, int K,
                             int8_t *Xq, float *x_scale, unsigned int *err, cudaStream_t st) {
    (void)err;  // no kernel of this pass waits on a barrier
    if (K <= 16384) {
        ActParams p{};
        p.br[0] = ActBranch{X, lambda, Xq, x_scale, M};
        p.K = K;
        return launch_act_quant_teams<false>(p, st);
    }
    return launch_row_quant<uint16_t, true>(X, lambda, M, K, Xq, x_scale, st);
}

cudaError_t launch_quant_act_f16codes(const uint16_t *X, const float *lambda, int M, int K,
                                     uint16_t *Xq16, float *x_scale, uint32_t *sumsq, bool gelu,
                                     cudaStream_t st) {
    if (gelu)
        if (cudaError_t e = build_gelu_table()) return e;
    ActParams p{};
    p.br[0] = ActBranch{X, lambda, reinterpret_cast<int8_t *>(Xq16), x_scale, M, sumsq};
    p.K = K;
    return gelu ? launch_act_quant_teams<true, true>(p, st) : launch_act_quant_teams<false, true>(p, st);
}

cudaError_t launch_quant_act_dual_f16codes(const QuantActBranch16 *br, int K, cudaStream_t st) {
    ActParams p{};
    for (int i = 0; i < 2; ++i)
        p.br[i] = ActBranch{br[i].X, br[i].lambda, reinterpret_cast<int8_t *>(br[i].Xq16), br[i].x_scale,
                            br[i].M, br[i].sumsq};
    p.K = K;
    return launch_act_quant_teams<false, true>(p, st);
}

cudaError_t launch_quant_act_dual(const QuantActBranch *br, int K, cudaStream_t st) {
    if (K <= 16384) {
        ActParams p{};
        for (int i = 0; i < 2; ++i)
            p.br[i] = ActBranch{br[i].X, br[i].lambda, br[i].Xq, br[i].x_scale, br[i].M, nullptr};
        p.K = K;
        return launch_act_quant_teams<false>(p, st);
    }
    for (int i = 0; i < 2; ++i) {
        if (br[i].M == 0) continue;
        cudaError_t e = launch_row_quant<uint16_t, true>(br[i].X, br[i].lambda, br[i].M, K, br[i].Xq,
                                                         br[i].x_scale, st);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

namespace {
__global__ void gelu_values_kernel(const uint16_t *__restrict__ H, int n, float *__restrict__ G) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        G[i] = gelu_of_bits(H[i]);
}

// The GELU table of the current device, built once (synchronously, on a
// stream of its own, so that every later launch on any stream finds it
// complete; this first build is no stream operation of the caller's, so it
// must not happen during a stream capture).
cudaError_t build_gelu_table() {
    static PerDevice<int> built;
    int unused = 0;
    return built.get([](int &) {
        cudaStream_t s;
        cudaError_t e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
        if (e != cudaSuccess) return e;
        gelu_table_kernel<<<65536 / 256, 256, 0, s>>>();
        e = cudaGetLastError();
        cudaError_t e2 = cudaStreamSynchronize(s);
        cudaStreamDestroy(s);
        return e != cudaSuccess ? e : e2;
    }, &unused);
}
}  // namespace

cudaError_t launch_debug_gelu(const uint16_t *H, int n, float *G, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (cudaError_t e = build_gelu_table()) return e;
    int grid = (n + 255) / 256;
    if (grid > num_sms() * 8) grid = num_sms() * 8;
    gelu_values_kernel<<<grid, 256, 0, st>>>(H, n, G);
    return cudaGetLastError();
}

cudaError_t launch_gelu_quant_act(const uint16_t *H, const float *lambda, int M, int K, int8_t *Xq,
                                  float *x_scale, cudaStream_t st) {
    if (cudaError_t e = build_gelu_table()) return e;
    if (K <= 16384) {
        ActParams p{};
        p.br[0] = ActBranch{H, lambda, Xq, x_scale, M};
        p.K = K;
        return launch_act_quant_teams<true>(p, st);
    }
    int g2 = num_sms() * 2;
    if (g2 > M) g2 = M;
    row_quant_long_kernel<uint16_t, true, true><<<g2, 512, 0, st>>>(H, lambda, M, K, Xq, x_scale);
    return cudaGetLastError();
}

}  // namespace w8a8
