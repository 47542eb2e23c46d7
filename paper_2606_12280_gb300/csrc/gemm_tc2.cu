// gemm_tc2.cu -- the W8A8 linear (a4 + a5, dual-branch a6) on pairs of SMs:
// tcgen05.mma.cta_group::2, the exact-integer scheme of gemm_tc.cu.
//
// The INT8 x INT8 -> INT32 product runs exactly on the fp16 tensor datapath
// (int8 values are fp16 values, products are exact in fp32, partial sums of
// at most 1024 products stay below 2^24); K advances in chunks of 1024 that
// are drained from TMEM into int32 running sums.
//
// A cluster of two CTAs (one per SM) computes a 256 x 256 output tile.  Each
// CTA stages its own 128 rows of Xq (A) and its own 128 rows of the 256-row
// Wq tile (B), converts them from int8 to fp16 in its shared memory, and the
// leader CTA (cluster rank 0) issues one M=256 N=256 K=16 MMA per K step that
// reads A and B from both CTAs' shared memory and writes each CTA's 128 rows
// of the accumulator into that CTA's TMEM.  Compared with one CTA per tile,
// every SM stages and feeds half of B, which is what the shared-memory
// bandwidth of the int8 -> fp16 staging needs.
//
// Per CTA: warp 0 TMA producer (int8 tiles), warp 1 TMEM allocation (both
// CTAs) and MMA issue (leader only), warps 2-7 converters (int8 -> fp16 into
// the swizzled fp16 ring), warps 8-15 epilogue (TMEM -> int32 running sums ->
// bf16 dequantized output).  Pipeline stages carry SUB K=64 sub-blocks.  The
// A16 variant takes the activation codes already as fp16 values: lane 1 of
// warp 0 loads them by TMA straight into the fp16 ring and the converters
// handle the weights only.  Cross-CTA signalling: converters and epilogue
// warps arrive on the leader's barriers through cluster addresses; the leader
// commits MMA completion to both CTAs' barriers by multicast.  All waits are
// bounded in time.
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "host_once.h"
#include "launch.h"
#include "tc_ptx.cuh"
#include "tile_order.cuh"

namespace w8a8 {
namespace {

using namespace tc;

#ifndef W8A8_TC2_SUB
#define W8A8_TC2_SUB 2
#endif
#ifndef W8A8_TC2_S8
#define W8A8_TC2_S8 2
#endif
#ifndef W8A8_TC2_S16
#define W8A8_TC2_S16 2
#endif
// One pipeline stage carries SUB sub-blocks of K = 64 (one 128-byte swizzle
// atom of fp16 per row each), so barrier hand-offs happen every 64*SUB of K.
constexpr int PAIR_M = 256, CTA_M = 128, PAIR_N = 256, CTA_N = 128, BK = 64;
constexpr int SUB = W8A8_TC2_SUB;
constexpr int KC_BLOCKS = 16;                        // K chunk = 1024 (exactness bound)
constexpr int KC_STAGES = KC_BLOCKS / SUB;           // stages per K chunk
constexpr int SUB8_A = CTA_M * BK, SUB8_B = CTA_N * BK;   // int8 bytes of A, B per sub-block
constexpr int SUB16_A = CTA_M * BK * 2, SUB16_B = CTA_N * BK * 2;
constexpr int SUB16 = SUB16_A + SUB16_B;             // 32 KB fp16 per sub-block
static_assert(KC_BLOCKS % SUB == 0, "chunk of whole stages");
constexpr int NUM_CONV_WARPS = 6;
constexpr int NUM_EPI_WARPS = 8;
constexpr int THREADS = 512;
constexpr int TMEM_COLS = 512;
constexpr int SMEM_BARRIERS = 256;
constexpr int LAUNCH_REGS = 128;
constexpr int REGS_LOW = 72, REGS_HIGH = 184;
static_assert(256 * REGS_LOW + 256 * REGS_HIGH <= THREADS * LAUNCH_REGS, "register split");
static_assert(KC_BLOCKS * BK * 127 * 127 < (1 << 24), "fp32 exactness bound");

constexpr unsigned ERR_PRODUCER = 1u, ERR_CONVERTER = 2u, ERR_MMA = 4u, ERR_EPILOGUE = 8u,
                   ERR_DRAIN = 16u, ERR_TMEM_PAIR = 64u;

#ifndef W8A8_TC2_A16_S8
#define W8A8_TC2_A16_S8 2
#endif
#ifndef W8A8_TC2_STAGE_EPI
#define W8A8_TC2_STAGE_EPI 1
#endif
#ifndef W8A8_TC2_A16_S16
#define W8A8_TC2_A16_S16 3
#endif
#ifndef W8A8_TC2_A16_SA
#define W8A8_TC2_A16_SA 3
#endif
// Shared-memory layout of one variant: fp16 stages, then int8 stages, then
// (A16) the A ring, then barriers, then (int8-A variant) the epilogue's
// staging of w_scale / bias.  In the A16 variant the fp16 and int8 stages
// carry B only and A has its own, deeper ring (TMA straight from the fp16
// codes), so that the A copy latency has SA - 1 stages of slack; its epilogue
// reads w_scale and bias through L1.
template <bool A16> struct Lay {
    static constexpr int NCONV = NUM_CONV_WARPS;              // converter warps 2 .. 7
    static constexpr int S8 = A16 ? W8A8_TC2_A16_S8 : W8A8_TC2_S8;
    static constexpr int S16 = A16 ? W8A8_TC2_A16_S16 : W8A8_TC2_S16;
    static constexpr int SUB8 = A16 ? SUB8_B : SUB8_A + SUB8_B;     // int8 bytes per sub-block
    static constexpr int B8 = A16 ? 0 : SUB8_A;                      // B's offset in it
    static constexpr int STAGE8 = SUB * SUB8;
    static constexpr int SUB16S = A16 ? SUB16_B : SUB16;            // fp16 bytes per sub-block
    static constexpr int STAGE16S = SUB * SUB16S;
    static constexpr int SA = A16 ? W8A8_TC2_A16_SA : 0;            // A ring stages
    static constexpr int SAm = SA > 0 ? SA : 1;                      // modulus (int8-A: unused)
    static constexpr int STAGEA = SUB * SUB16_A;
    static constexpr bool STAGE_EPI = !A16 && W8A8_TC2_STAGE_EPI;
    static constexpr int SMEM_EPI = STAGE_EPI ? NUM_EPI_WARPS * 1024 : 0;
    static constexpr uint32_t OFF_ST16 = 0;
    static constexpr uint32_t OFF_ST8 = OFF_ST16 + S16 * STAGE16S;
    static constexpr uint32_t OFF_A = OFF_ST8 + S8 * STAGE8;
    static constexpr uint32_t OFF_BAR = OFF_A + SA * STAGEA;
    static constexpr uint32_t BAR_FULL8 = OFF_BAR;
    static constexpr uint32_t BAR_EMPTY8 = BAR_FULL8 + 8 * S8;
    static constexpr uint32_t BAR_FULL16 = BAR_EMPTY8 + 8 * S8;
    static constexpr uint32_t BAR_EMPTY16 = BAR_FULL16 + 8 * S16;
    static constexpr uint32_t BAR_ACCFULL = BAR_EMPTY16 + 8 * S16;
    static constexpr uint32_t BAR_ACCEMPTY = BAR_ACCFULL + 16;
    static constexpr uint32_t BAR_DRAIN = BAR_ACCEMPTY + 16;
    static constexpr uint32_t BAR_AFULL = BAR_DRAIN + 8;            // A16: A slot landed
    static constexpr uint32_t BAR_AEMPTY = BAR_AFULL + 8 * SA;      // A16: MMA done with A slot
    static constexpr uint32_t OFF_TMEM = BAR_AEMPTY + 8 * SA;
    // operand addresses of sub-block u of stage (fp16 slot s16, A slot sa)
    static __device__ __forceinline__ uint32_t a_addr(uint32_t sb, uint32_t s16, uint32_t sa, int u) {
        return A16 ? sb + OFF_A + sa * STAGEA + u * SUB16_A : sb + OFF_ST16 + s16 * STAGE16S + u * SUB16;
    }
    static __device__ __forceinline__ uint32_t b_addr(uint32_t sb, uint32_t s16, int u) {
        return A16 ? sb + OFF_ST16 + s16 * STAGE16S + u * SUB16_B
                   : sb + OFF_ST16 + s16 * STAGE16S + u * SUB16 + SUB16_A;
    }
    static constexpr uint32_t OFF_ABORT = OFF_TMEM + 4;
    static constexpr uint32_t OFF_EPI = OFF_BAR + SMEM_BARRIERS;
    static constexpr int SMEM_TOTAL = 1024 + OFF_EPI + SMEM_EPI;
    static_assert(OFF_ABORT + 4 - OFF_BAR <= SMEM_BARRIERS, "barrier area");
    static_assert(SMEM_TOTAL <= 232448, "shared memory");
};

struct BranchArgs {
    const float *x_scale;
    const float *w_scale;
    const float *bias;
    void *out;
    int M;
    int m_tiles;     // pair tiles of 256 rows
    int tiles;       // m_tiles * n_tiles
};

struct Params {
    BranchArgs br[2];
    int N, K;
    int total_tiles;
    int k_blocks;
    int n_tiles, group;        // feature tiles; tile order (tile_order.cuh)
    unsigned int *err;
    uint64_t wait_limit_ns;
};

struct Tile {
    int branch, m0, n0;
};

__device__ __forceinline__ Tile tile_coords(const Params &p, int t) {
    Tile r;
    r.branch = t >= p.br[0].tiles ? 1 : 0;
    const int local = t - (r.branch ? p.br[0].tiles : 0);
    int mi, ni;
    grouped_tile(local, p.br[r.branch].m_tiles, p.n_tiles, p.group, mi, ni);
    r.m0 = mi * PAIR_M;
    r.n0 = ni * PAIR_N;
    return r;
}

__device__ __forceinline__ float4 ld_shared_f4(uint32_t a) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a));
    return v;
}

__device__ __forceinline__ void st_global_v4(void *p, uint4 v) {
    asm volatile("st.global.v4.b32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w) : "memory");
}

// int8 x4 -> two fp16x2 words, exact (bytes + 128 in the mantissa of 1024.0,
// minus 1152).
__device__ __forceinline__ void i8x4_to_f16x4(uint32_t w, uint32_t &lo, uint32_t &hi) {
    const uint32_t u = w ^ 0x80808080u;
    asm("prmt.b32 %0, %1, %2, 0x4140;" : "=r"(lo) : "r"(u), "r"(0x64646464u));
    asm("prmt.b32 %0, %1, %2, 0x4342;" : "=r"(hi) : "r"(u), "r"(0x64646464u));
    asm("sub.f16x2 %0, %0, %1;" : "+r"(lo) : "r"(0x64806480u));
    asm("sub.f16x2 %0, %0, %1;" : "+r"(hi) : "r"(0x64806480u));
}

template <bool OUT_I32, bool A16>
__device__ __forceinline__ void epilogue_role(const Params &p, uint32_t sb, uint32_t tmem,
                                              const WaitCtx &wc, int warp, int lane, int NC,
                                              uint32_t rank, int pair, int npairs) {
    using L = Lay<A16>;
    const int e = warp - 8;
    const int q = warp & 3;            // TMEM lane quarter this warp may access
    const int h = e >> 2;              // column half of the 256-wide tile
    uint32_t c = 0;
    bool ok = true;
    for (int t = pair; ok && t < p.total_tiles; t += npairs) {
        int32_t run[128];
#pragma unroll
        for (int i = 0; i < 128; ++i) run[i] = 0;
        for (int ci = 0; ci < NC; ++ci, ++c) {
            const uint32_t buf = c & 1;
            if (!mbar_wait_cluster(sb + L::BAR_ACCFULL + 8 * buf, (c >> 1) & 1, wc, ERR_EPILOGUE)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * PAIR_N + h * 128;
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                uint32_t v[16];
                tmem_ld_32x32b_x16(base + jj * 16, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 16; ++i) run[jj * 16 + i] += __float2int_rn(__uint_as_float(v[i]));
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (rank == 0) mbar_arrive(sb + L::BAR_ACCEMPTY + 8 * buf);
                else mbar_arrive_cluster_relaxed(mapa_shared(sb + L::BAR_ACCEMPTY + 8 * buf, 0));
            }
        }
        if (!ok) break;
        const Tile tl = tile_coords(p, t);
        const BranchArgs &br = p.br[tl.branch];
        const int m = tl.m0 + static_cast<int>(rank) * CTA_M + q * 32 + lane;
        const int n_base = tl.n0 + h * 128;
        const uint32_t epi = sb + L::OFF_EPI + e * 1024;
        if (!OUT_I32 && L::STAGE_EPI) {
            const int n = n_base + lane * 4;
            float4 w = make_float4(0.f, 0.f, 0.f, 0.f), b = w;
            if (n < p.N) {
                w = __ldg(reinterpret_cast<const float4 *>(br.w_scale + n));
                if (br.bias) b = __ldg(reinterpret_cast<const float4 *>(br.bias + n));
            }
            asm volatile("st.shared.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(epi + lane * 16),
                         "f"(w.x), "f"(w.y), "f"(w.z), "f"(w.w) : "memory");
            asm volatile("st.shared.v4.f32 [%0], {%1,%2,%3,%4};" ::"r"(epi + 512 + lane * 16),
                         "f"(b.x), "f"(b.y), "f"(b.z), "f"(b.w) : "memory");
            __syncwarp();
        }
        if (m < br.M) {
            if (OUT_I32) {
                int32_t *out = static_cast<int32_t *>(br.out) + (size_t)m * p.N + n_base;
#pragma unroll
                for (int g = 0; g < 16; ++g) {
                    if (n_base + g * 8 < p.N) {
                        *reinterpret_cast<int4 *>(out + g * 8) =
                            make_int4(run[g * 8], run[g * 8 + 1], run[g * 8 + 2], run[g * 8 + 3]);
                        *reinterpret_cast<int4 *>(out + g * 8 + 4) =
                            make_int4(run[g * 8 + 4], run[g * 8 + 5], run[g * 8 + 6], run[g * 8 + 7]);
                    }
                }
            } else {
                const float sx = __ldg(br.x_scale + m);
                const bool hb = br.bias != nullptr;
                uint16_t *out = static_cast<uint16_t *>(br.out) + (size_t)m * p.N + n_base;
#pragma unroll
                for (int g = 0; g < 16; ++g) {
                    if (n_base + g * 8 < p.N) {
                        float4 w0, w1, b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
                        if (L::STAGE_EPI) {
                            w0 = ld_shared_f4(epi + g * 32);
                            w1 = ld_shared_f4(epi + g * 32 + 16);
                            if (hb) {
                                b0 = ld_shared_f4(epi + 512 + g * 32);
                                b1 = ld_shared_f4(epi + 512 + g * 32 + 16);
                            }
                        } else {
                            // every lane reads the same 8 columns: L1 broadcast
                            const float4 *wp = reinterpret_cast<const float4 *>(br.w_scale + n_base + g * 8);
                            w0 = __ldg(wp);
                            w1 = __ldg(wp + 1);
                            if (hb) {
                                const float4 *bp = reinterpret_cast<const float4 *>(br.bias + n_base + g * 8);
                                b0 = __ldg(bp);
                                b1 = __ldg(bp + 1);
                            }
                        }
                        const uint32_t y0 = epilogue_value(run[g * 8 + 0], sx, w0.x, b0.x, hb);
                        const uint32_t y1 = epilogue_value(run[g * 8 + 1], sx, w0.y, b0.y, hb);
                        const uint32_t y2 = epilogue_value(run[g * 8 + 2], sx, w0.z, b0.z, hb);
                        const uint32_t y3 = epilogue_value(run[g * 8 + 3], sx, w0.w, b0.w, hb);
                        const uint32_t y4 = epilogue_value(run[g * 8 + 4], sx, w1.x, b1.x, hb);
                        const uint32_t y5 = epilogue_value(run[g * 8 + 5], sx, w1.y, b1.y, hb);
                        const uint32_t y6 = epilogue_value(run[g * 8 + 6], sx, w1.z, b1.z, hb);
                        const uint32_t y7 = epilogue_value(run[g * 8 + 7], sx, w1.w, b1.w, hb);
                        st_global_v4(out + g * 8, make_uint4(y0 | (y1 << 16), y2 | (y3 << 16),
                                                             y4 | (y5 << 16), y6 | (y7 << 16)));
                    }
                }
            }
        }
        __syncwarp();
    }
}

// A16: the activation codes arrive as fp16 values (exact: |q| <= 127), so
// TMA puts A straight into the swizzled fp16 tile and only the weights are
// converted; the int8 ring then carries B alone (in its B half).
template <bool OUT_I32, bool A16>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmB0,
                const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
                const Params p) {
    using L = Lay<A16>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sb = (smem_addr(smem_raw) + 1023u) & ~1023u;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    const int npairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int i = 0; i < L::S8; ++i) {
            mbar_init(sb + L::BAR_FULL8 + 8 * i, 1);
            mbar_init(sb + L::BAR_EMPTY8 + 8 * i, L::NCONV);
        }
        for (int i = 0; i < L::S16; ++i) {
            mbar_init(sb + L::BAR_FULL16 + 8 * i, 2 * L::NCONV);
            mbar_init(sb + L::BAR_EMPTY16 + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(sb + L::BAR_ACCFULL + 8 * i, 1);
            mbar_init(sb + L::BAR_ACCEMPTY + 8 * i, 2 * NUM_EPI_WARPS);
        }
        for (int i = 0; i < L::SA; ++i) {
            mbar_init(sb + L::BAR_AFULL + 8 * i, 1);
            mbar_init(sb + L::BAR_AEMPTY + 8 * i, 1);
        }
        mbar_init(sb + L::BAR_DRAIN, 1);
        st_shared_s32(sb + L::OFF_ABORT, 0);
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmA0);
        tma_prefetch_desc(&tmB0);
        tma_prefetch_desc(&tmA1);
        tma_prefetch_desc(&tmB1);
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
    const int KB = p.k_blocks;
    const int NS = (KB + SUB - 1) / SUB;                  // pipeline stages per tile
    const int NC = (KB + KC_BLOCKS - 1) / KC_BLOCKS;

    if (warp >= 8) {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(REGS_HIGH));
        if (run_ok) epilogue_role<OUT_I32, A16>(p, sb, tmem, wc, warp, lane, NC, rank, pair, npairs);
        tc_fence_before();
        __syncwarp();
        asm volatile("bar.sync 1, %0;" ::"n"(THREADS) : "memory");
        cluster_sync();
    } else {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REGS_LOW));
        if (!run_ok) {
        } else if (warp == 0) {
            // -------------------------------------------------- TMA producer
            // lane 0: the int8 ring (A and B, or B alone for A16); lane 1
            // (A16): A straight into the fp16 ring, as soon as the MMA frees a
            // slot, so that A's copy latency never waits behind B's ring
            if (lane == 0) {
                uint32_t j = 0;
                bool ok = true;
                for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                    const Tile tl = tile_coords(p, t);
                    const CUtensorMap *mA = tl.branch ? &tmA1 : &tmA0;
                    const CUtensorMap *mB = tl.branch ? &tmB1 : &tmB0;
                    const int arow = tl.m0 + static_cast<int>(rank) * CTA_M;
                    const int brow = tl.n0 + static_cast<int>(rank) * CTA_N;
                    for (int ks = 0; ks < NS; ++ks, ++j) {
                        const uint32_t st = j % L::S8;
                        if (!mbar_wait(sb + L::BAR_EMPTY8 + 8 * st, ((j / L::S8) & 1) ^ 1, wc, ERR_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = sb + L::BAR_FULL8 + 8 * st;
                        mbar_arrive_expect_tx(fb, L::STAGE8);
#pragma unroll
                        for (int u = 0; u < SUB; ++u) {
                            const uint32_t dst = sb + L::OFF_ST8 + st * L::STAGE8 + u * L::SUB8;
                            if (!A16) tma_load_2d(dst, mA, (ks * SUB + u) * BK, arow, fb);
                            tma_load_2d(dst + L::B8, mB, (ks * SUB + u) * BK, brow, fb);
                        }
                    }
                }
                for (uint32_t i = (j > L::S8 ? j - L::S8 : 0); i < j; ++i)
                    mbar_wait(sb + L::BAR_FULL8 + 8 * (i % L::S8), (i / L::S8) & 1, wc, ERR_DRAIN, false);
            } else if (A16 && lane == 1) {
                uint32_t j = 0;
                bool ok = true;
                for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                    const Tile tl = tile_coords(p, t);
                    const CUtensorMap *mA = tl.branch ? &tmA1 : &tmA0;
                    const int arow = tl.m0 + static_cast<int>(rank) * CTA_M;
                    for (int ks = 0; ks < NS; ++ks, ++j) {
                        const uint32_t sa = j % L::SAm;
                        if (!mbar_wait_cluster(sb + L::BAR_AEMPTY + 8 * sa, ((j / L::SAm) & 1) ^ 1, wc,
                                               ERR_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t ab = sb + L::BAR_AFULL + 8 * sa;
                        mbar_arrive_expect_tx(ab, L::STAGEA);
#pragma unroll
                        for (int u = 0; u < SUB; ++u)
                            tma_load_2d(L::a_addr(sb, 0, sa, u), mA, (ks * SUB + u) * BK, arow, ab);
                    }
                }
                for (uint32_t i = (j > L::SA ? j - L::SA : 0); i < j; ++i)
                    mbar_wait(sb + L::BAR_AFULL + 8 * (i % L::SAm), (i / L::SAm) & 1, wc, ERR_DRAIN, false);
            }
        } else if (warp == 1) {
            // ------------------------------------------- MMA issue (leader)
            if (lane == 0 && leader) {
                constexpr uint32_t idesc = idesc_f16_f32(PAIR_M, PAIR_N);
                uint32_t j = 0, c = 0;
                bool ok = true;
                for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                    for (int ci = 0; ok && ci < NC; ++ci, ++c) {
                        const uint32_t buf = c & 1;
                        if (!mbar_wait_cluster(sb + L::BAR_ACCEMPTY + 8 * buf, ((c >> 1) & 1) ^ 1, wc,
                                               ERR_MMA)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t d = tmem + buf * PAIR_N;
                        const int ks0 = ci * KC_STAGES;
                        const int ks1 = min(NS, ks0 + KC_STAGES);
                        for (int ks = ks0; ks < ks1; ++ks, ++j) {
                            const uint32_t st = j % L::S16;
                            if (!mbar_wait_cluster(sb + L::BAR_FULL16 + 8 * st, (j / L::S16) & 1, wc, ERR_MMA)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint32_t sa = A16 ? j % L::SAm : 0;
#pragma unroll
                            for (int u = 0; u < SUB; ++u) {
                                const uint32_t a = L::a_addr(sb, st, sa, u);
                                const uint32_t b = L::b_addr(sb, st, u);
#pragma unroll
                                for (int kk = 0; kk < BK / 16; ++kk) {
                                    mma_f16_ss_pair(d, smem_desc_sw128(a + kk * 32),
                                                    smem_desc_sw128(b + kk * 32), idesc,
                                                    (ks > ks0 || u > 0 || kk > 0) ? 1u : 0u);
                                }
                            }
                            mma_commit_pair_multicast(sb + L::BAR_EMPTY16 + 8 * st, 0x3);
                            if (A16) mma_commit_pair_multicast(sb + L::BAR_AEMPTY + 8 * sa, 0x3);
                        }
                        if (ok) mma_commit_pair_multicast(sb + L::BAR_ACCFULL + 8 * buf, 0x3);
                    }
                }
                mma_commit_pair(sb + L::BAR_DRAIN);
                mbar_wait_cluster(sb + L::BAR_DRAIN, 0, wc, ERR_DRAIN, false);
            }
        } else {
            // ---------------------------------------------------- converters
            const int cw = warp - 2;
            const uint32_t rr = lane >> 2;
            const uint32_t c4 = lane & 3;
            const uint32_t src_off = rr * BK + c4 * 16;
            const uint32_t dst_off0 = rr * 128 + (((2 * c4) ^ rr) << 4);
            const uint32_t dst_off1 = rr * 128 + (((2 * c4 + 1) ^ rr) << 4);
            uint32_t j = 0;
            bool ok = true;
            for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                for (int ks = 0; ks < NS; ++ks, ++j) {
                    const uint32_t s8 = j % L::S8, s16 = j % L::S16;
                    // every lane waits; __all_sync keeps the warp's control flow
                    // uniform if a wait gives up
                    if (!__all_sync(0xffffffffu, mbar_wait(sb + L::BAR_FULL8 + 8 * s8, (j / L::S8) & 1, wc,
                                                            ERR_CONVERTER) &&
                                                     mbar_wait_cluster(sb + L::BAR_EMPTY16 + 8 * s16,
                                                                       ((j / L::S16) & 1) ^ 1, wc,
                                                                       ERR_CONVERTER))) {
                        ok = false;
                        break;
                    }
                    const uint32_t src = sb + L::OFF_ST8 + s8 * L::STAGE8 + src_off;
                    const uint32_t dst = sb + L::OFF_ST16 + s16 * L::STAGE16S;
                    // all of this warp's 8-row groups of a sub-block in flight at
                    // once: every load is issued before the first conversion needs
                    // its data (group g of sub-block u sits at u * kG1 + g in both
                    // rings: a sub-block is CTA_M + CTA_N rows of 64 int8 bytes,
                    // 128 fp16 bytes; the A16 variant converts only the B groups,
                    // kG0 .. kG1 - 1, and keeps both sub-blocks' loads in flight)
                    constexpr int kG1 = (CTA_M + CTA_N) / 8;
                    constexpr int kG0 = A16 ? CTA_M / 8 : 0;
                    constexpr int kPer = (kG1 - kG0 + L::NCONV - 1) / L::NCONV;
                    constexpr int kAtOnce = A16 ? SUB : 1;
#pragma unroll
                    for (int u0 = 0; u0 < SUB; u0 += kAtOnce) {
                        uint4 v[kAtOnce][kPer];
#pragma unroll
                        for (int uu = 0; uu < kAtOnce; ++uu)
#pragma unroll
                            for (int i = 0; i < kPer; ++i) {
                                const int g = kG0 + cw + i * L::NCONV;
                                if (g < kG1) v[uu][i] = ld_shared_v4(src + (u0 + uu) * L::SUB8 + (g - kG0) * 8 * BK);
                            }
#pragma unroll
                        for (int uu = 0; uu < kAtOnce; ++uu)
#pragma unroll
                            for (int i = 0; i < kPer; ++i) {
                                const int g = kG0 + cw + i * L::NCONV;
                                const int u = u0 + uu;
                                if (g < kG1) {
                                    uint4 o0, o1;
                                    i8x4_to_f16x4(v[uu][i].x, o0.x, o0.y);
                                    i8x4_to_f16x4(v[uu][i].y, o0.z, o0.w);
                                    i8x4_to_f16x4(v[uu][i].z, o1.x, o1.y);
                                    i8x4_to_f16x4(v[uu][i].w, o1.z, o1.w);
                                    // A16: the fp16 stage holds B alone
                                    const uint32_t gd = dst + (A16 ? u * SUB16_B + (g - kG0) * 1024
                                                                   : (u * kG1 + g) * 1024);
                                    st_shared_v4(gd + dst_off0, o0);
                                    st_shared_v4(gd + dst_off1, o1);
                                }
                            }
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (A16) {
                        // this CTA's A tile must have landed too before the
                        // leader may issue: converter warp 0 checks it
                        bool a_ok = true;
                        if (cw == 0 && lane == 0)
                            a_ok = mbar_wait(sb + L::BAR_AFULL + 8 * (j % L::SAm), (j / L::SAm) & 1, wc,
                                             ERR_CONVERTER);
                        if (!__shfl_sync(0xffffffffu, a_ok ? 1 : 0, 0)) {
                            ok = false;
                            break;
                        }
                    }
                    if (lane == 0) {
                        if (leader) mbar_arrive(sb + L::BAR_FULL16 + 8 * s16);
                        else mbar_arrive_cluster_relaxed(mapa_shared(sb + L::BAR_FULL16 + 8 * s16, 0));
                        mbar_arrive(sb + L::BAR_EMPTY8 + 8 * s8);
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

// int8 row-major [rows, K] -> 2-D map with box [box_rows, 64 bytes], zero fill.
bool make_map(CUtensorMap *m, const int8_t *base, int rows, int K, int box_rows) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(K)};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t *>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp16 row-major [rows, K] -> 2-D map with box [box_rows, 64 elements] landing
// in the 128-byte swizzled layout, zero fill.
bool make_map_f16(CUtensorMap *m, const void *base, int rows, int K, int box_rows) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool OUT_I32, bool A16>
cudaError_t prepare_tc2_kernel() {
    static PerDevice<int> setup;
    int regs = -1;
    cudaError_t e = setup.get([](int &v) {
        cudaFuncAttributes fa;
        cudaError_t r = cudaFuncGetAttributes(&fa, gemm_tc2_kernel<OUT_I32, A16>);
        if (r != cudaSuccess) return r;
        v = fa.numRegs;
        return cudaFuncSetAttribute(gemm_tc2_kernel<OUT_I32, A16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    Lay<A16>::SMEM_TOTAL);
    }, &regs);
    if (e != cudaSuccess) return e;
    return regs == LAUNCH_REGS ? cudaSuccess : cudaErrorInvalidConfiguration;
}

}  // namespace

cudaError_t launch_gemm_tc2(const GemmBranch *br, int nb, int N, int K, bool out_i32, bool a16,
                            unsigned int *err, cudaStream_t st) {
    const int sms = device_sms();
    const int smem_total = a16 ? Lay<true>::SMEM_TOTAL : Lay<false>::SMEM_TOTAL;
    auto kern = a16 ? (out_i32 ? gemm_tc2_kernel<true, true> : gemm_tc2_kernel<false, true>)
                    : (out_i32 ? gemm_tc2_kernel<true, false> : gemm_tc2_kernel<false, false>);
    cudaError_t e = a16 ? (out_i32 ? prepare_tc2_kernel<true, true>() : prepare_tc2_kernel<false, true>())
                        : (out_i32 ? prepare_tc2_kernel<true, false>() : prepare_tc2_kernel<false, false>());
    if (e != cudaSuccess) return e;

    Params p{};
    CUtensorMap maps[4];
    int first = -1;
    for (int i = 0; i < 2; ++i) {
        const GemmBranch *b = (i < nb) ? &br[i] : nullptr;
        BranchArgs &a = p.br[i];
        a = BranchArgs{nullptr, nullptr, nullptr, nullptr, 0, 0, 0};
        if (b && b->M > 0) {
            a.x_scale = b->x_scale;
            a.w_scale = b->w_scale;
            a.bias = b->bias;
            a.out = b->out;
            a.M = b->M;
            a.m_tiles = (b->M + PAIR_M - 1) / PAIR_M;
            a.tiles = a.m_tiles * ((N + PAIR_N - 1) / PAIR_N);
            const bool okA = a16 ? make_map_f16(&maps[2 * i], b->Xq, b->M, K, CTA_M)
                                 : make_map(&maps[2 * i], b->Xq, b->M, K, CTA_M);
            if (!okA || !make_map(&maps[2 * i + 1], b->Wq, N, K, CTA_N))
                return cudaErrorInvalidValue;
            if (first < 0) first = i;
        }
    }
    if (first < 0) return cudaSuccess;
    for (int i = 0; i < 2; ++i)
        if (p.br[i].M == 0) {
            maps[2 * i] = maps[2 * first];
            maps[2 * i + 1] = maps[2 * first + 1];
        }
    p.N = N;
    p.K = K;
    p.total_tiles = p.br[0].tiles + p.br[1].tiles;
    p.k_blocks = (K + BK - 1) / BK;
    // tile order (tile_order.cuh): activation codes of 1 or 2 bytes, int8 weights
    p.n_tiles = (N + PAIR_N - 1) / PAIR_N;
    p.group = tile_group((a16 ? 2LL : 1LL) * K * (p.br[0].M > p.br[1].M ? p.br[0].M : p.br[1].M),
                         static_cast<long long>(PAIR_N) * K, p.n_tiles);
    p.err = err;
    p.wait_limit_ns = 2000000000ull;
    const int pairs = p.total_tiles < sms / 2 ? p.total_tiles : sms / 2;
    return launch_pdl(kern, dim3(2 * pairs), THREADS, smem_total, st, maps[0], maps[1], maps[2], maps[3], p);
}

}  // namespace w8a8
