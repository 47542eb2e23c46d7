// gemm_gguf.cu -- the GGUF weight-only linear: Y = bf16(X dequant(W)^T + b)
// with bf16 activations X and Q8_0 or Q4_K weight blocks, on pairs of SMs
// (tcgen05.mma.cta_group::2, bf16 operands, fp32 accumulation).
//
// Sec. 3, "GGUF k-quants": the DiT serialized to Q8_0 (8.5 bits per weight)
// and Q4_K (4.5 bits, the paper's memory-Pareto choice), which it ran with a
// Torch dequantization (Sec. 5).  Here the weights stay in their GGUF blocks
// in HBM and are decoded next to the MMA, straight into tensor memory: the
// decoded weights are the MMA's A operand in TMEM ("TS" form), the
// activations its B operand in shared memory, loaded by TMA unconverted, so
// no decoded operand passes through shared memory (the same placement as
// gemm_ts.cu).
//
// A cluster of two CTAs computes a 256 (output features) x 256 (tokens) tile
// of Y^T: CTA r decodes weight rows f0 + 128r .. +127 into its TMEM lanes
// (one row per converter thread) and holds tokens t0 + 128r .. +127 in its
// shared memory; the leader issues M=256 N=256 K=16 bf16 MMAs, eight per
// stage of K=128.  TMEM per CTA: one 256-column fp32 accumulator and four
// 64-column weight slots.  Per CTA: warp 0 TMA of the raw weight blocks (one
// 256-weight span per ring slot), warp 2 TMA of the activations (both CTAs
// against the leader's barrier), warp 1 TMEM allocation and MMA issue
// (leader), warps 4-7 decode (warp w owns TMEM lanes 32(w%4) .. +31), warps
// 8-15 drain the accumulator once per tile, add the bias and write bf16.
// All waits are bounded in time.
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "host_once.h"
#include "launch.h"
#include "tc_ptx.cuh"
#include "tile_order.cuh"

namespace w8a8 {
namespace {

using namespace tc;

constexpr int PAIR_F = 256, CTA_F = 128;      // output features per pair / CTA (MMA M)
constexpr int PAIR_T = 256, CTA_T = 128;      // tokens per pair / CTA (MMA N)
constexpr int BK = 64;                         // bf16 per swizzle row = one K=64 sub-block
constexpr int KR = 256;                        // weights per raw span (one Q4_K block)
constexpr int SUB = 2;                         // sub-blocks per stage (K=128)
constexpr int STAGES_PER_SPAN = KR / (SUB * BK);
constexpr int SA = 4;                          // slots: TMEM weights + smem activations
constexpr int SUBX = CTA_T * BK * 2;           // 16 KB of activations per sub-block
constexpr int STAGE_X = SUB * SUBX;
constexpr uint32_t ACC_COLS = PAIR_T;
constexpr uint32_t A_COL0 = ACC_COLS;
constexpr uint32_t A_SLOT_COLS = SUB * BK / 2; // bf16 pairs per row of a slot
constexpr int NUM_CONV_WARPS = 4;
constexpr int NUM_EPI_WARPS = 8;
constexpr int THREADS = 512;
constexpr int LAUNCH_REGS = 128;
constexpr int REGS_LOW = 72, REGS_HIGH = 184;
static_assert(256 * REGS_LOW + 256 * REGS_HIGH <= THREADS * LAUNCH_REGS, "register split");
constexpr int RUN = PAIR_T / 2;                // accumulator columns per epilogue thread
constexpr int TMEM_COLS = 512;
static_assert(A_COL0 + SA * A_SLOT_COLS <= TMEM_COLS, "tensor memory");
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
    static constexpr int RAW_SLOT = CTA_F * Fmt<FMT>::ROW;
    static constexpr int SR = Fmt<FMT>::SR;
    static constexpr uint32_t OFF_X = 0;
    static constexpr uint32_t OFF_RAW = OFF_X + SA * STAGE_X;
    static constexpr uint32_t OFF_BAR = OFF_RAW + SR * RAW_SLOT;
    static constexpr uint32_t BAR_RFULL = OFF_BAR;
    static constexpr uint32_t BAR_REMPTY = BAR_RFULL + 8 * SR;
    static constexpr uint32_t BAR_SFULL = BAR_REMPTY + 8 * SR;     // leader: slot written and landed
    static constexpr uint32_t BAR_SEMPTY = BAR_SFULL + 8 * SA;     // MMA done with the slot
    static constexpr uint32_t BAR_ACCFULL = BAR_SEMPTY + 8 * SA;
    static constexpr uint32_t BAR_ACCEMPTY = BAR_ACCFULL + 8;
    static constexpr uint32_t BAR_DRAIN = BAR_ACCEMPTY + 8;
    static constexpr uint32_t OFF_TMEM = BAR_DRAIN + 8;
    static constexpr uint32_t OFF_ABORT = OFF_TMEM + 4;
    static constexpr int SMEM_TOTAL = 1024 + OFF_BAR + SMEM_BARRIERS;
    static_assert(OFF_ABORT + 4 - OFF_BAR <= SMEM_BARRIERS, "barrier area");
    static_assert(SMEM_TOTAL <= 232448, "shared memory");
    static_assert(RAW_SLOT % 16 == 0 && STAGE_X % 1024 == 0, "TMA destinations aligned");
};

__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
           (static_cast<uint32_t>(M >> 4) << 24);
}

struct Params {
    const float *bias;
    uint16_t *Y;
    int M, N, K;
    int t_tiles, total_tiles, spans;           // spans = K / 256 per tile
    int f_tiles, group;                        // feature tiles; tile order (tile_order.cuh)
    unsigned int *err;
    uint64_t wait_limit_ns;
};

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

// Decode stage H (weights 128H .. 128H + 127 of the 256-weight span) of one
// weight row (`row`: its raw bytes in shared memory) into 64 bf16x2 columns
// of TMEM at `tcol` (this warp's lanes), two tcgen05.st of 32 columns.
//
// Q8_0: blocks 4H .. 4H + 3, two at a time: the 68 bytes of blocks b0, b0 + 1
// start 4-byte aligned (34 b0 = 136H + 68k) and are read as five 16-byte loads
// (conflict-free across a warp's rows at the 272-byte stride); block b0's
// quants start 2 bytes into it (byte permutes), block b0 + 1's are aligned.
template <int H>
__device__ __forceinline__ void q8_stage(uint32_t row, uint32_t tcol) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int s0 = 136 * H + 68 * k;
        const int a0 = s0 & ~15;
        const int w0 = (s0 - a0) / 4;
        uint32_t W[20];
#pragma unroll
        for (int i = 0; i < 5; ++i) {
            const uint4 v = ld_shared_v4(row + a0 + 16 * i);
            W[4 * i] = v.x;
            W[4 * i + 1] = v.y;
            W[4 * i + 2] = v.z;
            W[4 * i + 3] = v.w;
        }
        const float da = f16_bits_to_f32(W[w0] & 0xffffu);
        const float db = f16_bits_to_f32(W[w0 + 8] >> 16);
        uint32_t out[32];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint4 o = q8_chunk(__byte_perm(W[w0 + 2 * c], W[w0 + 2 * c + 1], 0x5432),
                                     __byte_perm(W[w0 + 2 * c + 1], W[w0 + 2 * c + 2], 0x5432), da);
            out[4 * c] = o.x;
            out[4 * c + 1] = o.y;
            out[4 * c + 2] = o.z;
            out[4 * c + 3] = o.w;
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint4 o = q8_chunk(W[w0 + 9 + 2 * c], W[w0 + 10 + 2 * c], db);
            out[16 + 4 * c] = o.x;
            out[16 + 4 * c + 1] = o.y;
            out[16 + 4 * c + 2] = o.z;
            out[16 + 4 * c + 3] = o.w;
        }
        tmem_st_32x32b_x32(tcol + 32 * k, out);
    }
}

// Q4_K: the block header (d, dmin, 12 scale bytes), then chunks c = 2H and
// 2H + 1 of 32 quant bytes: low nibbles are weights 64c .. 64c + 31
// (sub-block 2c), high nibbles 64c + 32 .. 64c + 63 (sub-block 2c + 1).
template <int H>
__device__ __forceinline__ void q4k_stage(uint32_t row, uint32_t tcol) {
    const uint4 hd = ld_shared_v4(row);
    const float d = f16_bits_to_f32(hd.x & 0xffffu), dmin = f16_bits_to_f32(hd.x >> 16);
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int c = 2 * H + k;
        const uint4 qa = ld_shared_v4(row + 16 + 32 * c), qb = ld_shared_v4(row + 32 + 32 * c);
        uint32_t sc, m;
        q4k_scale_min(hd.y, hd.z, hd.w, 2 * c, sc, m);
        const float d1a = __fmul_rn(d, static_cast<float>(sc)), m1a = __fmul_rn(dmin, static_cast<float>(m));
        q4k_scale_min(hd.y, hd.z, hd.w, 2 * c + 1, sc, m);
        const float d1b = __fmul_rn(d, static_cast<float>(sc)), m1b = __fmul_rn(dmin, static_cast<float>(m));
        const uint2 v[4] = {make_uint2(qa.x, qa.y), make_uint2(qa.z, qa.w), make_uint2(qb.x, qb.y),
                            make_uint2(qb.z, qb.w)};
        uint32_t out[32];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const uint4 lo = q4k_chunk<0>(v[e], d1a, m1a);
            const uint4 hi = q4k_chunk<4>(v[e], d1b, m1b);
            out[4 * e] = lo.x;
            out[4 * e + 1] = lo.y;
            out[4 * e + 2] = lo.z;
            out[4 * e + 3] = lo.w;
            out[16 + 4 * e] = hi.x;
            out[16 + 4 * e + 1] = hi.y;
            out[16 + 4 * e + 2] = hi.z;
            out[16 + 4 * e + 3] = hi.w;
        }
        tmem_st_32x32b_x32(tcol + 32 * k, out);
    }
}

__device__ __forceinline__ void arrive_leader(uint32_t bar, uint32_t rank) {
    if (rank == 0) mbar_arrive(bar);
    else mbar_arrive_cluster_relaxed(mapa_shared(bar, 0));
}

__device__ __forceinline__ void tile_coords(const Params &p, int t, int &t0, int &f0) {
    int ti, fi;
    grouped_tile(t, p.t_tiles, p.f_tiles, p.group, ti, fi);
    t0 = ti * PAIR_T;
    f0 = fi * PAIR_F;
}

template <int FMT>
__device__ __forceinline__ void epilogue_role(const Params &p, uint32_t sb, uint32_t tmem,
                                              const WaitCtx &wc, int warp, int lane,
                                              uint32_t rank, int pair, int npairs) {
    using L = Layout<FMT>;
    const int q = warp & 3;                          // TMEM lane quarter of this warp
    const int h = (warp - 8) >> 2;                   // token half of the tile
    uint32_t c = 0;
    for (int t = pair; t < p.total_tiles; t += npairs, ++c) {
        if (!mbar_wait_cluster(sb + L::BAR_ACCFULL, c & 1, wc, ERR_EPILOGUE)) break;
        tc_fence_after();
        const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + h * RUN;
        uint32_t acc[RUN];
#pragma unroll
        for (int jj = 0; jj < RUN / 16; jj += 4) {
            uint32_t v[4][16];
#pragma unroll
            for (int g = 0; g < 4; ++g) tmem_ld_32x32b_x16(base + (jj + g) * 16, v[g]);
            tmem_ld_wait();
#pragma unroll
            for (int g = 0; g < 4; ++g)
#pragma unroll
                for (int i = 0; i < 16; ++i) acc[(jj + g) * 16 + i] = v[g][i];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) arrive_leader(sb + L::BAR_ACCEMPTY, rank);
        int t0, f0;
        tile_coords(p, t, t0, f0);
        const int f = f0 + static_cast<int>(rank) * CTA_F + q * 32 + lane;    // output feature
        const int tok0 = t0 + h * RUN;
        const int ntok = min(RUN, p.M - tok0);
        const bool fok = f < p.N;
        if (ntok > 0) {                              // uniform across the warp
            const float b = (p.bias != nullptr && fok) ? __ldg(p.bias + f) : 0.0f;
            // lanes 2i, 2i + 1 (features f, f + 1) swap one value per pair of
            // tokens, so that each stores one 32-bit word (N % 8 == 0)
            const bool odd = lane & 1;
            uint16_t *out = p.Y + (size_t)tok0 * p.N + (f & ~1);
#pragma unroll
            for (int i = 0; i < RUN; i += 2) {
                const uint32_t y = pack_bf16_pair(add2(pk2(acc[i], acc[i + 1]),
                                                       pk2(__float_as_uint(b), __float_as_uint(b))));
                // y: low = token i, high = token i + 1 of this feature
                const uint32_t other = __shfl_xor_sync(0xffffffffu, odd ? (y & 0xffffu) : (y >> 16), 1);
                const uint32_t word = odd ? (other | (y & 0xffff0000u)) : ((y & 0xffffu) | (other << 16));
                const int tk = i + (odd ? 1 : 0);
                if (tk < ntok && fok)
                    asm volatile("st.global.cs.u32 [%0], %1;" ::"l"(out + (size_t)tk * p.N), "r"(word)
                                 : "memory");
            }
        }
        __syncwarp();
    }
}

template <int FMT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_gguf_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
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
        for (int i = 0; i < SA; ++i) {
            mbar_init(sb + L::BAR_SFULL + 8 * i, 2 * NUM_CONV_WARPS + 1);
            mbar_init(sb + L::BAR_SEMPTY + 8 * i, 1);
        }
        mbar_init(sb + L::BAR_ACCFULL, 1);
        mbar_init(sb + L::BAR_ACCEMPTY, 2 * NUM_EPI_WARPS);
        mbar_init(sb + L::BAR_DRAIN, 1);
        st_shared_s32(sb + L::OFF_ABORT, 0);
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmX);
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
    wait_prior_grid();
    const WaitCtx wc{sb + L::OFF_ABORT, p.err, p.wait_limit_ns};
    const int NS = p.spans * STAGES_PER_SPAN;          // stages per tile

    if (warp >= 8) {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(REGS_HIGH));
        if (run_ok) epilogue_role<FMT>(p, sb, tmem, wc, warp, lane, rank, pair, npairs);
    } else {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REGS_LOW));
        if (!run_ok) {
        } else if (warp == 0) {
            // ------------------------------- TMA producer: raw weight blocks
            if (lane == 0) {
                uint32_t qs = 0;                       // spans so far
                bool ok = true;
                for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                    int t0, f0;
                    tile_coords(p, t, t0, f0);
                    const int frow = f0 + static_cast<int>(rank) * CTA_F;
                    for (int sp = 0; sp < p.spans; ++sp, ++qs) {
                        const uint32_t rs = qs % SR;
                        if (!mbar_wait(sb + L::BAR_REMPTY + 8 * rs, ((qs / SR) & 1) ^ 1, wc, ERR_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(sb + L::BAR_RFULL + 8 * rs, L::RAW_SLOT);
                        const int x = FMT == 1 ? sp * Fmt<FMT>::ROW : sp * (Fmt<FMT>::ROW / 2);
                        tma_load_2d(sb + L::OFF_RAW + rs * L::RAW_SLOT, &tmW, x, frow, sb + L::BAR_RFULL + 8 * rs);
                    }
                }
                for (uint32_t i = (qs > SR ? qs - SR : 0); i < qs; ++i)
                    mbar_wait(sb + L::BAR_RFULL + 8 * (i % SR), (i / SR) & 1, wc, ERR_DRAIN, false);
            }
        } else if (warp == 2) {
            // ------------------------------- TMA producer: activations (bf16)
            // both CTAs load against the leader's barrier, which the leader
            // armed for both CTAs' bytes (every load has landed before the
            // kernel ends: the MMA waits for each)
            if (lane == 0) {
                uint32_t j = 0;
                bool ok = true;
                for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                    int t0, f0;
                    tile_coords(p, t, t0, f0);
                    const int trow = t0 + static_cast<int>(rank) * CTA_T;
                    for (int ks = 0; ks < NS; ++ks, ++j) {
                        const uint32_t s = j % SA;
                        if (!mbar_wait_cluster(sb + L::BAR_SEMPTY + 8 * s, ((j / SA) & 1) ^ 1, wc, ERR_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = mapa_shared(sb + L::BAR_SFULL + 8 * s, 0);
                        if (leader) mbar_arrive_expect_tx(sb + L::BAR_SFULL + 8 * s, 2 * STAGE_X);
#pragma unroll
                        for (int u = 0; u < SUB; ++u)
                            tma_load_2d_pair(sb + L::OFF_X + s * STAGE_X + u * SUBX, &tmX, (ks * SUB + u) * BK, trow, fb);
                    }
                }
            }
        } else if (warp == 1) {
            // ---------------------------------------- MMA issue (leader)
            if (lane == 0 && leader) {
                constexpr uint32_t idesc = idesc_bf16_f32(PAIR_F, PAIR_T);
                const uint64_t b_desc0 = smem_desc_sw128(sb + L::OFF_X);
                const uint32_t a_base = tmem + A_COL0;
                uint32_t j = 0, c = 0;
                bool ok = true;
                for (int t = pair; ok && t < p.total_tiles; t += npairs, ++c) {
                    if (!mbar_wait_cluster(sb + L::BAR_ACCEMPTY, (c & 1) ^ 1, wc, ERR_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int ks = 0; ks < NS; ++ks, ++j) {
                        const uint32_t sa = j % SA;
                        if (!mbar_wait_cluster(sb + L::BAR_SFULL + 8 * sa, (j / SA) & 1, wc, ERR_MMA)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t a = a_base + sa * A_SLOT_COLS;
                        const uint64_t bd = b_desc0 + sa * (STAGE_X >> 4);
#pragma unroll
                        for (int u = 0; u < SUB; ++u)
#pragma unroll
                            for (int kk = 0; kk < BK / 16; ++kk)
                                mma_f16_ts_pair(tmem, a + u * (BK / 2) + kk * 8, bd + u * (SUBX >> 4) + kk * 2, idesc,
                                                (ks > 0 || u > 0 || kk > 0) ? 1u : 0u);
                        mma_commit_pair_multicast(sb + L::BAR_SEMPTY + 8 * sa, 0x3);
                    }
                    if (ok) mma_commit_pair_multicast(sb + L::BAR_ACCFULL, 0x3);
                }
                mma_commit_pair(sb + L::BAR_DRAIN);
                mbar_wait_cluster(sb + L::BAR_DRAIN, 0, wc, ERR_DRAIN, false);
            }
        } else if (warp >= 4) {
            // ------------------------------------------------------ decoders
            // thread = weight row r of this CTA = TMEM lane r
            const uint32_t r = static_cast<uint32_t>((warp & 3) * 32 + lane);
            const uint32_t a_lane = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + A_COL0;
            uint32_t j = 0, qs = 0;
            bool ok = true;
            for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                for (int sp = 0; ok && sp < p.spans; ++sp, ++qs) {
                    const uint32_t rs = qs % SR;
                    // every lane waits; __all_sync keeps the warp's control flow
                    // uniform if a wait gives up
                    if (!__all_sync(0xffffffffu, mbar_wait(sb + L::BAR_RFULL + 8 * rs, (qs / SR) & 1, wc,
                                                            ERR_CONVERTER))) {
                        ok = false;
                        break;
                    }
                    const uint32_t row = sb + L::OFF_RAW + rs * L::RAW_SLOT + r * Fmt<FMT>::ROW;
#pragma unroll
                    for (int hh = 0; hh < STAGES_PER_SPAN; ++hh, ++j) {
                        const uint32_t sa = j % SA;
                        if (!__all_sync(0xffffffffu, mbar_wait_cluster(sb + L::BAR_SEMPTY + 8 * sa,
                                                                        ((j / SA) & 1) ^ 1, wc, ERR_CONVERTER))) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t tcol = a_lane + sa * A_SLOT_COLS;
                        if (FMT == 1) {
                            if (hh == 0) q4k_stage<0>(row, tcol);
                            else q4k_stage<1>(row, tcol);
                        } else {
                            if (hh == 0) q8_stage<0>(row, tcol);
                            else q8_stage<1>(row, tcol);
                        }
                        if (hh == STAGES_PER_SPAN - 1) {
                            // the span's bytes are all in registers (and TMEM)
                            __syncwarp();
                            if (lane == 0) mbar_arrive(sb + L::BAR_REMPTY + 8 * rs);
                        }
                        tmem_st_wait();
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) arrive_leader(sb + L::BAR_SFULL + 8 * sa, rank);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncwarp();
    asm volatile("bar.sync 1, %0;" ::"n"(THREADS) : "memory");
    cluster_sync();
    if (warp == 1) {
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
    // a function-local static: initialised once, thread-safe
    static const EncodeTiledFn fn = [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<EncodeTiledFn>(ptr);
        return static_cast<EncodeTiledFn>(nullptr);
    }();
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

template <int FMT>
cudaError_t launch_fmt(const uint16_t *X, const uint8_t *Wraw, const float *bias, int M, int N, int K,
                       uint16_t *Y, unsigned int *err, cudaStream_t st) {
    using L = Layout<FMT>;
    static PerDevice<int> setup;
    int regs = -1;
    cudaError_t e = setup.get([](int &v) {
        cudaFuncAttributes fa;
        cudaError_t r = cudaFuncGetAttributes(&fa, gemm_gguf_kernel<FMT>);
        if (r != cudaSuccess) return r;
        v = fa.numRegs;
        return cudaFuncSetAttribute(gemm_gguf_kernel<FMT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    L::SMEM_TOTAL);
    }, &regs);
    if (e != cudaSuccess) return e;
    // the register split above assumes the launch gets exactly this many
    if (regs != LAUNCH_REGS) return cudaErrorInvalidConfiguration;
    CUtensorMap mX, mW;
    if (!make_map(&mX, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, X, static_cast<uint64_t>(K), M,
                  static_cast<uint64_t>(K) * 2, BK, CTA_T, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    const uint64_t spans = static_cast<uint64_t>(K) / KR;
    const uint64_t row_bytes = spans * Fmt<FMT>::ROW;
    bool okw;
    if (FMT == 1)
        okw = make_map(&mW, CU_TENSOR_MAP_DATA_TYPE_UINT8, Wraw, row_bytes, N, row_bytes, Fmt<FMT>::ROW,
                       CTA_F, CU_TENSOR_MAP_SWIZZLE_NONE);
    else
        okw = make_map(&mW, CU_TENSOR_MAP_DATA_TYPE_UINT16, Wraw, row_bytes / 2, N, row_bytes,
                       Fmt<FMT>::ROW / 2, CTA_F, CU_TENSOR_MAP_SWIZZLE_NONE);
    if (!okw) return cudaErrorInvalidValue;
    Params p{};
    p.bias = bias;
    p.Y = Y;
    p.M = M;
    p.N = N;
    p.K = K;
    p.t_tiles = (M + PAIR_T - 1) / PAIR_T;
    p.f_tiles = (N + PAIR_F - 1) / PAIR_F;
    p.total_tiles = p.t_tiles * p.f_tiles;
    // tile order (tile_order.cuh): bf16 activations, raw blocks of row_bytes per row
    p.group = tile_group(2LL * K * M, static_cast<long long>(PAIR_F) * row_bytes, p.f_tiles);
    p.spans = static_cast<int>(spans);
    p.err = err;
    p.wait_limit_ns = 2000000000ull;
    const int sms = device_sms();
    const int pairs = p.total_tiles < sms / 2 ? p.total_tiles : sms / 2;
    return launch_pdl(gemm_gguf_kernel<FMT>, dim3(2 * pairs), THREADS, L::SMEM_TOTAL, st, mX, mW, p);
}

}  // namespace

cudaError_t launch_gemm_gguf(const uint16_t *X, const uint8_t *Wraw, int fmt, const float *bias, int M,
                             int N, int K, uint16_t *Y, unsigned int *err, cudaStream_t st) {
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
