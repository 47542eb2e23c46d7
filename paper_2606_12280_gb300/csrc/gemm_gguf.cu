// gemm_gguf.cu -- the GGUF weight-only linear: Y = bf16(X dequant(W)^T + b)
// with bf16 activations X and Q8_0 or Q4_K weight blocks, on pairs of SMs
// (tcgen05.mma.cta_group::2, bf16 operands, fp32 accumulation).
//
// Sec. 3, "GGUF k-quants": the DiT serialized to Q8_0 (8.5 bits per weight)
// and Q4_K (4.5 bits, the paper's memory-Pareto choice), which it ran with a
// Torch dequantization (Sec. 5).  Here the weights stay in their GGUF blocks
// in HBM and are decoded tile by tile in shared memory, next to the MMA.
//
// A cluster of two CTAs (one per SM) computes a 256 x 256 output tile.  Per
// CTA: warp 0 issues TMA loads of X tiles [128 x 64] straight into the
// 128-byte-swizzled K-major layout and of raw weight blocks [128 rows x one
// 256-weight span] into a raw ring; warp 1 allocates TMEM (both CTAs) and,
// on the leader, issues one M=256 N=256 K=16 bf16 MMA per K step; the
// converter warps decode the raw blocks of each K=64 step into the swizzled
// bf16 B tile (fp32 arithmetic as the decoder defines it, then round to
// bf16); the last four warps drain the fp32 accumulator (two TMEM buffers),
// add the bias and write bf16.  All waits are bounded in time.
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "launch.h"
#include "tc_ptx.cuh"

namespace w8a8 {
namespace {

using namespace tc;

constexpr int PAIR_M = 256, CTA_M = 128, PAIR_N = 256, CTA_N = 128;
constexpr int BK = 64;                         // bf16 per swizzle row = one MMA stage
constexpr int KR = 256;                        // weights per raw span (one Q4_K block)
#ifndef W8A8_GGUF_SUB
#define W8A8_GGUF_SUB 2
#endif
#ifndef W8A8_GGUF_STAGES
#define W8A8_GGUF_STAGES 2
#endif
constexpr int SUB = W8A8_GGUF_SUB;             // K=64 steps per pipeline stage
constexpr int SUBS = KR / BK;                  // K=64 steps per raw span
constexpr int STAGES_PER_SPAN = SUBS / SUB;
constexpr int S = W8A8_GGUF_STAGES;            // bf16 stage ring
constexpr int TILE_BYTES = CTA_M * BK * 2;     // 16 KB, A or B of one K=64 step
constexpr int STEP_BYTES = 2 * TILE_BYTES;     // A then B
constexpr int STAGE = SUB * STEP_BYTES;
static_assert(SUBS % SUB == 0, "whole stages per raw span");
#ifndef W8A8_GGUF_CONV_WARPS
#define W8A8_GGUF_CONV_WARPS 8
#endif
constexpr int NUM_CONV_WARPS = W8A8_GGUF_CONV_WARPS;
constexpr int CONV_TASKS = CTA_N * 4;          // per K=64 step: 128 rows x 4 chunk pairs
constexpr int kTasksPerThread = CONV_TASKS / (32 * NUM_CONV_WARPS);
static_assert(CONV_TASKS % (32 * NUM_CONV_WARPS) == 0, "whole tasks per converter thread");
constexpr int NUM_EPI_WARPS = 4;
constexpr int CONV_WARP0 = 2, EPI_WARP0 = CONV_WARP0 + NUM_CONV_WARPS;
constexpr int THREADS = 32 * (EPI_WARP0 + NUM_EPI_WARPS);
constexpr int TMEM_COLS = 512;
constexpr int SMEM_BARRIERS = 256;

constexpr unsigned ERR_PRODUCER = 1u, ERR_CONVERTER = 2u, ERR_MMA = 4u, ERR_EPILOGUE = 8u,
                   ERR_DRAIN = 16u, ERR_TMEM_PAIR = 64u;

// Per-format raw span: bytes per weight row per 256 weights, raw ring depth.
template <int FMT> struct Fmt;
template <> struct Fmt<0> {                    // Q8_0: 8 blocks of (fp16 d, 32 x int8)
    static constexpr int ROW = 8 * 34;         // 272 bytes
    static constexpr int SR = 2;
};
template <> struct Fmt<1> {                    // Q4_K: fp16 d, fp16 dmin, 12 B scales, 128 B quants
    static constexpr int ROW = 144;
    static constexpr int SR = 3;
};

template <int FMT> struct Layout {
    static constexpr int RAW_SLOT = CTA_N * Fmt<FMT>::ROW;
    static constexpr int SR = Fmt<FMT>::SR;
    static constexpr uint32_t OFF_ST = 0;
    static constexpr uint32_t OFF_RAW = S * STAGE;
    static constexpr uint32_t OFF_BAR = OFF_RAW + SR * RAW_SLOT;
    static constexpr uint32_t BAR_RFULL = OFF_BAR;
    static constexpr uint32_t BAR_REMPTY = BAR_RFULL + 8 * SR;
    static constexpr uint32_t BAR_AFULL = BAR_REMPTY + 8 * SR;
    static constexpr uint32_t BAR_FULL = BAR_AFULL + 8 * S;
    static constexpr uint32_t BAR_EMPTY = BAR_FULL + 8 * S;
    static constexpr uint32_t BAR_ACCFULL = BAR_EMPTY + 8 * S;
    static constexpr uint32_t BAR_ACCEMPTY = BAR_ACCFULL + 16;
    static constexpr uint32_t BAR_DRAIN = BAR_ACCEMPTY + 16;
    static constexpr uint32_t OFF_TMEM = BAR_DRAIN + 8;
    static constexpr uint32_t OFF_ABORT = OFF_TMEM + 4;
    static constexpr int SMEM_TOTAL = 1024 + OFF_BAR + SMEM_BARRIERS;
    static_assert(OFF_ABORT + 4 - OFF_BAR <= SMEM_BARRIERS, "barrier area");
    static_assert(SMEM_TOTAL <= 232448, "shared memory");
};

__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
           (static_cast<uint32_t>(M >> 4) << 24);
}

struct Params {
    const float *bias;
    uint16_t *Y;
    int M, N, K;
    int m_tiles, total_tiles, spans;           // spans = K / 256 per tile
    unsigned int *err;
    uint64_t wait_limit_ns;
};

__device__ __forceinline__ uint32_t ld_shared_u32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}

__device__ __forceinline__ uint2 ld_shared_v2(uint32_t a) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
    return v;
}

__device__ __forceinline__ uint32_t ld_shared_u16(uint32_t a) {
    uint16_t v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}

__device__ __forceinline__ float f16_bits_to_f32(uint32_t h) {
    return __half2float(__ushort_as_half(static_cast<unsigned short>(h)));
}

// The 6-bit scale and min of Q4_K sub-block j from the 12 scale bytes
// (three little-endian words w0 = bytes 0-3, w1 = 4-7, w2 = 8-11).
__device__ __forceinline__ void q4k_scale_min(uint32_t w0, uint32_t w1, uint32_t w2, int j,
                                              uint32_t &sc, uint32_t &m) {
    if (j < 4) {
        sc = (w0 >> (8 * j)) & 63u;
        m = (w1 >> (8 * j)) & 63u;
    } else {
        const int i = j - 4;
        const uint32_t b8 = (w2 >> (8 * i)) & 0xffu;
        sc = (b8 & 15u) | (((w0 >> (8 * i)) >> 6 & 3u) << 4);
        m = (b8 >> 4) | (((w1 >> (8 * i)) >> 6 & 3u) << 4);
    }
}

// Packed fp32 pairs (each packed operation rounds like its scalar form).
__device__ __forceinline__ uint64_t pk2(uint32_t a, uint32_t b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(a), "r"(b));
    return r;
}

__device__ __forceinline__ uint64_t pkf(float a) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %1};" : "=l"(r) : "f"(a));
    return r;
}

__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

// the pair as one bf16x2 word (low = first), each rounded to nearest even
__device__ __forceinline__ uint32_t pack_bf16_pair(uint64_t v) {
    uint32_t a, b, r;
    asm("mov.b64 {%0, %1}, %2;" : "=r"(a), "=r"(b) : "l"(v));
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "r"(b), "r"(a));
    return r;
}

// fp32 bit patterns 2^23 + byte_i(x) for bytes i0 and i1 of x, as a pair:
// one byte permute each (the byte lands in the low mantissa bits of 2^23).
template <int I0, int I1>
__device__ __forceinline__ uint64_t magic_pair(uint32_t x) {
    return pk2(__byte_perm(x, 0x4B000000u, 0x7440 | I0), __byte_perm(x, 0x4B000000u, 0x7440 | I1));
}

// Decode 8 Q4_K weights d1 * q - m1 (q = the low (SHIFT 0) or high (SHIFT 4)
// nibbles of the 8 quant bytes in v) into 4 bf16x2 words.  d1 * q is exact
// (17 + 4 bits), so the fused multiply-add rounds once, as the decoder does.
template <int SHIFT>
__device__ __forceinline__ uint4 q4k_chunk(uint2 v, float d1, float m1) {
    const uint32_t n0 = (v.x >> SHIFT) & 0x0f0f0f0fu, n1 = (v.y >> SHIFT) & 0x0f0f0f0fu;
    const uint64_t bias = pkf(-8388608.0f), D = pkf(d1), Mn = pkf(-m1);
    uint32_t w[4];
    w[0] = pack_bf16_pair(fma2(D, add2(magic_pair<0, 1>(n0), bias), Mn));
    w[1] = pack_bf16_pair(fma2(D, add2(magic_pair<2, 3>(n0), bias), Mn));
    w[2] = pack_bf16_pair(fma2(D, add2(magic_pair<0, 1>(n1), bias), Mn));
    w[3] = pack_bf16_pair(fma2(D, add2(magic_pair<2, 3>(n1), bias), Mn));
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// Decode 8 Q8_0 quants (bytes of lo, hi) times d into 4 bf16x2 words:
// 2^23 + (q + 128) minus 2^23 + 128 is q exactly, d * q is exact.
__device__ __forceinline__ uint4 q8_chunk(uint32_t lo, uint32_t hi, float d) {
    const uint32_t a = lo ^ 0x80808080u, b = hi ^ 0x80808080u;
    const uint64_t bias = pkf(-8388736.0f), D = pkf(d);
    uint32_t w[4];
    w[0] = pack_bf16_pair(mul2(D, add2(magic_pair<0, 1>(a), bias)));
    w[1] = pack_bf16_pair(mul2(D, add2(magic_pair<2, 3>(a), bias)));
    w[2] = pack_bf16_pair(mul2(D, add2(magic_pair<0, 1>(b), bias)));
    w[3] = pack_bf16_pair(mul2(D, add2(magic_pair<2, 3>(b), bias)));
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// Per-row constants of one 256-weight span, computed once per span and kept
// in registers: Q4_K d * sc_j and dmin * m_j for the eight sub-blocks; Q8_0
// the eight block scales d (in d1).
struct Q4kRow {
    float d1[8], m1[8];
};

__device__ __forceinline__ void q8_row_consts(uint32_t src, Q4kRow &r) {
#pragma unroll
    for (int b = 0; b < 8; ++b) r.d1[b] = f16_bits_to_f32(ld_shared_u16(src + 34 * b));
}

__device__ __forceinline__ void q4k_row_consts(uint32_t src, Q4kRow &r) {
    const uint32_t dd = ld_shared_u32(src);
    const float d = f16_bits_to_f32(dd & 0xffffu), dmin = f16_bits_to_f32(dd >> 16);
    const uint32_t w0 = ld_shared_u32(src + 4), w1 = ld_shared_u32(src + 8), w2 = ld_shared_u32(src + 12);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        uint32_t sc, m;
        q4k_scale_min(w0, w1, w2, j, sc, m);
        r.d1[j] = __fmul_rn(d, static_cast<float>(sc));     // exact: 11 x 6 bits
        r.m1[j] = __fmul_rn(dmin, static_cast<float>(m));
    }
}

// One converter task: row `row` of the CTA's 128 weight rows, output chunks c
// and c + 4 (16 bf16) of K=64 step u of the raw span.  Q4_K: chunk c holds
// the low nibbles (sub-block 2u), chunk c + 4 the high nibbles (2u + 1) of
// the same 8 quant bytes.  Q8_0: chunks c and c + 4 come from blocks 2u and
// 2u + 1, whose 8 quant bytes start 2 bytes into their 34-byte block.
template <int FMT>
__device__ __forceinline__ void convert_task(uint32_t raw, uint32_t dst, int row, int c, int u,
                                             float d1a, float m1a, float d1b, float m1b) {
    const uint32_t src = raw + static_cast<uint32_t>(row) * Fmt<FMT>::ROW;
    uint4 lo, hi;
    if (FMT == 1) {
        const uint2 v = ld_shared_v2(src + 16 + 32 * u + 8 * c);
        lo = q4k_chunk<0>(v, d1a, m1a);
        hi = q4k_chunk<4>(v, d1b, m1b);
    } else {
        // block 2u's quants start 2 mod 4 bytes into the row: three aligned
        // words and two byte permutes; block 2u + 1's are 4-byte aligned
        const uint32_t q0 = src + 34 * (2 * u) + 2 + 8 * c, q1 = q0 + 34;
        const uint32_t x0 = ld_shared_u32(q0 - 2), x1 = ld_shared_u32(q0 + 2), x2 = ld_shared_u32(q0 + 6);
        lo = q8_chunk(__byte_perm(x0, x1, 0x5432), __byte_perm(x1, x2, 0x5432), d1a);
        hi = q8_chunk(ld_shared_u32(q1), ld_shared_u32(q1 + 4), d1b);
    }
    // 128-byte swizzle: 16-byte chunk k of row r at (k ^ (r & 7))
    const uint32_t rb = dst + static_cast<uint32_t>(row) * 128;
    st_shared_v4(rb + ((static_cast<uint32_t>(c) ^ (row & 7)) << 4), lo);
    st_shared_v4(rb + ((static_cast<uint32_t>(c + 4) ^ (row & 7)) << 4), hi);
}

template <int FMT>
__device__ __forceinline__ void epilogue_role(const Params &p, uint32_t sb, uint32_t tmem,
                                              const WaitCtx &wc, int warp, int lane,
                                              uint32_t rank, int pair, int npairs) {
    using L = Layout<FMT>;
    const int q = warp & 3;                          // TMEM lane quarter of this warp
    uint32_t c = 0;
    for (int t = pair; t < p.total_tiles; t += npairs, ++c) {
        const uint32_t buf = c & 1;
        if (!mbar_wait_cluster(sb + L::BAR_ACCFULL + 8 * buf, (c >> 1) & 1, wc, ERR_EPILOGUE)) break;
        tc_fence_after();
        const int m0 = (t % p.m_tiles) * PAIR_M;
        const int n0 = (t / p.m_tiles) * PAIR_N;
        const int m = m0 + static_cast<int>(rank) * CTA_M + q * 32 + lane;
        const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * PAIR_N;
        uint16_t *out = p.Y + (size_t)m * p.N + n0;
#pragma unroll 1
        for (int cc = 0; cc < PAIR_N / 16; ++cc) {
            uint32_t v[16];
            tmem_ld_32x32b_x16(base + cc * 16, v);
            tmem_ld_wait();
            const int n = n0 + cc * 16;
            if (m < p.M) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (n + 8 * h < p.N) {
                        float b[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) b[i] = 0.0f;
                        if (p.bias != nullptr) {
                            const float4 b0 = __ldg(reinterpret_cast<const float4 *>(p.bias + n + 8 * h));
                            const float4 b1 = __ldg(reinterpret_cast<const float4 *>(p.bias + n + 8 * h + 4));
                            b[0] = b0.x; b[1] = b0.y; b[2] = b0.z; b[3] = b0.w;
                            b[4] = b1.x; b[5] = b1.y; b[6] = b1.z; b[7] = b1.w;
                        }
                        uint32_t w[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            w[i] = pack_bf16_pair(add2(pk2(v[8 * h + 2 * i], v[8 * h + 2 * i + 1]),
                                                       pk2(__float_as_uint(b[2 * i]), __float_as_uint(b[2 * i + 1]))));
                        *reinterpret_cast<uint4 *>(out + cc * 16 + 8 * h) = make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
            }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
            if (rank == 0) mbar_arrive(sb + L::BAR_ACCEMPTY + 8 * buf);
            else mbar_arrive_cluster_relaxed(mapa_shared(sb + L::BAR_ACCEMPTY + 8 * buf, 0));
        }
    }
}

template <int FMT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_gguf_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmW,
                 const Params p) {
    using L = Layout<FMT>;
    constexpr int SR = L::SR;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sb = (smem_addr(smem_raw) + 1023u) & ~1023u;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    const int npairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int i = 0; i < SR; ++i) {
            mbar_init(sb + L::BAR_RFULL + 8 * i, 1);
            mbar_init(sb + L::BAR_REMPTY + 8 * i, NUM_CONV_WARPS);
        }
        for (int i = 0; i < S; ++i) {
            mbar_init(sb + L::BAR_AFULL + 8 * i, 1);
            mbar_init(sb + L::BAR_FULL + 8 * i, 2 * NUM_CONV_WARPS);
            mbar_init(sb + L::BAR_EMPTY + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(sb + L::BAR_ACCFULL + 8 * i, 1);
            mbar_init(sb + L::BAR_ACCEMPTY + 8 * i, 2 * NUM_EPI_WARPS);
        }
        mbar_init(sb + L::BAR_DRAIN, 1);
        st_shared_s32(sb + L::OFF_ABORT, 0);
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmW);
    }
    if (warp == 1) {
        tmem_alloc_pair(sb + L::OFF_TMEM, TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(ld_shared_s32(sb + L::OFF_TMEM));
    const uint32_t peer_tmem = ld_shared_cluster_u32(mapa_shared(sb + L::OFF_TMEM, rank ^ 1u));
    const bool run_ok = (tmem == peer_tmem);
    if (!run_ok && threadIdx.x == 0) atomicOr(p.err, ERR_TMEM_PAIR);
    const WaitCtx wc{sb + L::OFF_ABORT, p.err, p.wait_limit_ns};
    // spans are numbered q = 0, 1, ... over this pair's tiles in order; span q
    // is span (q % spans) of tile pair + (q / spans) * npairs
    const int my_tiles = p.total_tiles > pair ? (p.total_tiles - pair + npairs - 1) / npairs : 0;
    const int total_spans = my_tiles * p.spans;

    if (!run_ok) {
    } else if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            int raw_issued = 0;
            auto issue_raw = [&](int qs) -> bool {
                const int t = pair + (qs / p.spans) * npairs;
                const int brow = (t / p.m_tiles) * PAIR_N + static_cast<int>(rank) * CTA_N;
                const uint32_t rs = qs % SR;
                if (!mbar_wait(sb + L::BAR_REMPTY + 8 * rs, ((qs / SR) & 1) ^ 1, wc, ERR_PRODUCER))
                    return false;
                mbar_arrive_expect_tx(sb + L::BAR_RFULL + 8 * rs, L::RAW_SLOT);
                const int x = FMT == 1 ? (qs % p.spans) * Fmt<FMT>::ROW : (qs % p.spans) * (Fmt<FMT>::ROW / 2);
                tma_load_2d(sb + L::OFF_RAW + rs * L::RAW_SLOT, &tmW, x, brow, sb + L::BAR_RFULL + 8 * rs);
                ++raw_issued;
                return true;
            };
            bool ok = total_spans == 0 || issue_raw(0);
            uint32_t j = 0;
            for (int qs = 0; ok && qs < total_spans; ++qs) {
                const int t = pair + (qs / p.spans) * npairs;
                const int arow = (t % p.m_tiles) * PAIR_M + static_cast<int>(rank) * CTA_M;
                for (int g = 0; ok && g < STAGES_PER_SPAN; ++g, ++j) {
                    const uint32_t st = j % S;
                    if (!mbar_wait_cluster(sb + L::BAR_EMPTY + 8 * st, ((j / S) & 1) ^ 1, wc, ERR_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(sb + L::BAR_AFULL + 8 * st, SUB * TILE_BYTES);
#pragma unroll
                    for (int v = 0; v < SUB; ++v)
                        tma_load_2d(sb + L::OFF_ST + st * STAGE + v * STEP_BYTES, &tmA,
                                    ((qs % p.spans) * SUBS + g * SUB + v) * BK, arow, sb + L::BAR_AFULL + 8 * st);
                    if (g == 0 && qs + 1 < total_spans) ok = issue_raw(qs + 1);
                }
            }
            // drain: every issued TMA has landed before the CTA may exit
            const uint32_t nraw = static_cast<uint32_t>(raw_issued);
            for (uint32_t i = (j > S ? j - S : 0); i < j; ++i)
                mbar_wait(sb + L::BAR_AFULL + 8 * (i % S), (i / S) & 1, wc, ERR_DRAIN, false);
            for (uint32_t i = (nraw > SR ? nraw - SR : 0); i < nraw; ++i)
                mbar_wait(sb + L::BAR_RFULL + 8 * (i % SR), (i / SR) & 1, wc, ERR_DRAIN, false);
        }
    } else if (warp == 1) {
        // ---------------------------------------------- MMA issue (leader)
        if (lane == 0 && leader) {
            constexpr uint32_t idesc = idesc_bf16_f32(PAIR_M, PAIR_N);
            uint32_t j = 0, c = 0;
            bool ok = true;
            for (int t = pair; ok && t < p.total_tiles; t += npairs, ++c) {
                const uint32_t buf = c & 1;
                if (!mbar_wait_cluster(sb + L::BAR_ACCEMPTY + 8 * buf, ((c >> 1) & 1) ^ 1, wc, ERR_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + buf * PAIR_N;
                const int nk = p.spans * STAGES_PER_SPAN;
                for (int ks = 0; ks < nk; ++ks, ++j) {
                    const uint32_t st = j % S;
                    if (!mbar_wait_cluster(sb + L::BAR_FULL + 8 * st, (j / S) & 1, wc, ERR_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll
                    for (int v = 0; v < SUB; ++v) {
                        const uint32_t a = sb + L::OFF_ST + st * STAGE + v * STEP_BYTES;
                        const uint32_t b = a + TILE_BYTES;
#pragma unroll
                        for (int kk = 0; kk < BK / 16; ++kk)
                            mma_f16_ss_pair(d, smem_desc_sw128(a + kk * 32), smem_desc_sw128(b + kk * 32), idesc,
                                            (ks > 0 || v > 0 || kk > 0) ? 1u : 0u);
                    }
                    mma_commit_pair_multicast(sb + L::BAR_EMPTY + 8 * st, 0x3);
                }
                if (ok) mma_commit_pair_multicast(sb + L::BAR_ACCFULL + 8 * buf, 0x3);
            }
            mma_commit_pair(sb + L::BAR_DRAIN);
            mbar_wait_cluster(sb + L::BAR_DRAIN, 0, wc, ERR_DRAIN, false);
        }
    } else if (warp < EPI_WARP0) {
        // ------------------------------------------------------ converters
        const int cw = warp - CONV_WARP0;
        const int tid = cw * 32 + lane;
        const uint32_t full0 = leader ? 0u : mapa_shared(sb + L::BAR_FULL, 0);
        uint32_t j = 0;
        bool ok = true;
        for (int qs = 0; ok && qs < total_spans; ++qs) {
            const uint32_t rs = qs % SR;
            // every lane waits; __all_sync keeps the warp's control flow uniform
            // if a wait gives up
            if (!__all_sync(0xffffffffu, mbar_wait(sb + L::BAR_RFULL + 8 * rs, (qs / SR) & 1, wc,
                                                    ERR_CONVERTER)))
                break;
            const uint32_t raw = sb + L::OFF_RAW + rs * L::RAW_SLOT;
            // this thread's tasks: a warp's 32 tasks are 8 consecutive rows
            // (lane & 7) x the 4 chunk pairs (lane >> 3), so that every
            // quarter-warp stores to 8 different 16-byte bank groups of the
            // swizzled tile
            Q4kRow rc[kTasksPerThread];
#pragma unroll
            for (int i = 0; i < kTasksPerThread; ++i) {
                const int task = tid + 32 * NUM_CONV_WARPS * i;
                const uint32_t rsrc = raw + static_cast<uint32_t>(8 * (task >> 5) + (task & 7)) * Fmt<FMT>::ROW;
                if (FMT == 1) q4k_row_consts(rsrc, rc[i]);
                else q8_row_consts(rsrc, rc[i]);
            }
#pragma unroll
            for (int g = 0; g < STAGES_PER_SPAN; ++g) {
                const uint32_t st = j % S;
                if (!__all_sync(0xffffffffu, mbar_wait_cluster(sb + L::BAR_EMPTY + 8 * st,
                                                               ((j / S) & 1) ^ 1, wc, ERR_CONVERTER))) {
                    ok = false;
                    break;
                }
#pragma unroll
                for (int v = 0; v < SUB; ++v) {
                    const int u = g * SUB + v;                 // K=64 step within the span
                    const uint32_t dst = sb + L::OFF_ST + st * STAGE + v * STEP_BYTES + TILE_BYTES;
#pragma unroll
                    for (int i = 0; i < kTasksPerThread; ++i) {
                        const int task = tid + 32 * NUM_CONV_WARPS * i;
                        convert_task<FMT>(raw, dst, 8 * (task >> 5) + (task & 7), (task >> 3) & 3, u,
                                          rc[i].d1[2 * u], rc[i].m1[2 * u], rc[i].d1[2 * u + 1],
                                          rc[i].m1[2 * u + 1]);
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                // the A tile of this stage must have landed too before the
                // leader may issue: converter warp 0 checks it
                bool a_ok = true;
                if (cw == 0 && lane == 0)
                    a_ok = mbar_wait(sb + L::BAR_AFULL + 8 * st, (j / S) & 1, wc, ERR_CONVERTER);
                if (!__shfl_sync(0xffffffffu, a_ok ? 1 : 0, 0)) {
                    ok = false;
                    break;
                }
                if (lane == 0) {
                    if (leader) mbar_arrive(sb + L::BAR_FULL + 8 * st);
                    else mbar_arrive_cluster_relaxed(full0 + 8 * st);
                }
                ++j;
            }
            if (!ok) break;
            if (lane == 0) mbar_arrive(sb + L::BAR_REMPTY + 8 * rs);
        }
    } else {
        epilogue_role<FMT>(p, sb, tmem, wc, warp, lane, rank, pair, npairs);
    }
    tc_fence_before();
    __syncwarp();
    __syncthreads();
    cluster_sync();
    if (warp == 1 && run_ok) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, TMEM_COLS);
    }
}

// Test export: decode raw blocks to bf16 in global memory with the same
// arithmetic as the converters; one thread per 8 consecutive weights.
template <int FMT>
__global__ void gguf_dequant_kernel(const uint8_t *__restrict__ raw, int N, int K,
                                    uint16_t *__restrict__ W) {
    const int chunks = K / 8;
    const long long total = static_cast<long long>(N) * chunks;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int n = static_cast<int>(i / chunks), k = static_cast<int>(i % chunks);
        const int span = k / 32, k8 = k % 32, u = k8 / 8, cc = k8 % 8;
        const uint8_t *src = raw + ((size_t)n * (K / KR) + span) * Fmt<FMT>::ROW;
        uint4 out;
        if (FMT == 1) {
            const uint32_t *w = reinterpret_cast<const uint32_t *>(src);
            const uint32_t dd = w[0];
            uint32_t sc, m;
            q4k_scale_min(w[1], w[2], w[3], 2 * u + (cc >= 4 ? 1 : 0), sc, m);
            const uint2 v = *reinterpret_cast<const uint2 *>(src + 16 + 32 * u + 8 * (cc & 3));
            const float d1 = __fmul_rn(f16_bits_to_f32(dd & 0xffffu), static_cast<float>(sc));
            const float m1 = __fmul_rn(f16_bits_to_f32(dd >> 16), static_cast<float>(m));
            out = cc >= 4 ? q4k_chunk<4>(v, d1, m1) : q4k_chunk<0>(v, d1, m1);
        } else {
            const uint8_t *blk = src + 34 * (2 * u + (cc >= 4 ? 1 : 0));
            const uint16_t *h = reinterpret_cast<const uint16_t *>(blk);
            const uint32_t q = 1 + 4 * (cc & 3);               // u16 index of the chunk's quants
            out = q8_chunk(h[q] | (static_cast<uint32_t>(h[q + 1]) << 16),
                           h[q + 2] | (static_cast<uint32_t>(h[q + 3]) << 16), f16_bits_to_f32(h[0]));
        }
        *reinterpret_cast<uint4 *>(W + (size_t)n * K + 8 * (size_t)k) = out;
    }
}

// ------------------------------------------------------------------ host

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

bool make_map(CUtensorMap *m, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t rows,
              uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle sw) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {inner, rows};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, dt, 2, const_cast<void *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int g_sms = 0;

template <int FMT>
cudaError_t launch_fmt(const uint16_t *X, const uint8_t *Wraw, const float *bias, int M, int N, int K,
                       uint16_t *Y, unsigned int *err, cudaStream_t st) {
    using L = Layout<FMT>;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(gemm_gguf_kernel<FMT>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_TOTAL);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    CUtensorMap mA, mW;
    if (!make_map(&mA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, X, static_cast<uint64_t>(K), M,
                  static_cast<uint64_t>(K) * 2, BK, CTA_M, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    const uint64_t spans = static_cast<uint64_t>(K) / KR;
    const uint64_t row_bytes = spans * Fmt<FMT>::ROW;
    bool okw;
    if (FMT == 1)
        okw = make_map(&mW, CU_TENSOR_MAP_DATA_TYPE_UINT8, Wraw, row_bytes, N, row_bytes, Fmt<FMT>::ROW,
                       CTA_N, CU_TENSOR_MAP_SWIZZLE_NONE);
    else
        okw = make_map(&mW, CU_TENSOR_MAP_DATA_TYPE_UINT16, Wraw, row_bytes / 2, N, row_bytes,
                       Fmt<FMT>::ROW / 2, CTA_N, CU_TENSOR_MAP_SWIZZLE_NONE);
    if (!okw) return cudaErrorInvalidValue;
    Params p{};
    p.bias = bias;
    p.Y = Y;
    p.M = M;
    p.N = N;
    p.K = K;
    p.m_tiles = (M + PAIR_M - 1) / PAIR_M;
    p.total_tiles = p.m_tiles * ((N + PAIR_N - 1) / PAIR_N);
    p.spans = static_cast<int>(spans);
    p.err = err;
    p.wait_limit_ns = 2000000000ull;
    const int pairs = p.total_tiles < g_sms / 2 ? p.total_tiles : g_sms / 2;
    gemm_gguf_kernel<FMT><<<2 * pairs, THREADS, L::SMEM_TOTAL, st>>>(mA, mW, p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_gguf(const uint16_t *X, const uint8_t *Wraw, int fmt, const float *bias, int M,
                             int N, int K, uint16_t *Y, unsigned int *err, cudaStream_t st) {
    if (g_sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
    }
    return fmt == 1 ? launch_fmt<1>(X, Wraw, bias, M, N, K, Y, err, st)
                    : launch_fmt<0>(X, Wraw, bias, M, N, K, Y, err, st);
}

cudaError_t launch_gguf_dequant(const uint8_t *Wraw, int fmt, int N, int K, uint16_t *W,
                                cudaStream_t st) {
    const long long total = static_cast<long long>(N) * (K / 8);
    const int grid = static_cast<int>(total / 256 + 1 < 4096 ? total / 256 + 1 : 4096);
    if (fmt == 1) gguf_dequant_kernel<1><<<grid, 256, 0, st>>>(Wraw, N, K, W);
    else gguf_dequant_kernel<0><<<grid, 256, 0, st>>>(Wraw, N, K, W);
    return cudaGetLastError();
}

}  // namespace w8a8
