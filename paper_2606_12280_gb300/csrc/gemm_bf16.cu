// gemm_bf16.cu -- the protected (unquantized) linear: Y = bf16(X W^T + b) with
// bf16 X and W, fp32 accumulation, on pairs of SMs (tcgen05.mma.cta_group::2).
//
// Sec. 3, "Activation-fragility profiling and protection": the most fragile
// layers keep their bf16 weights and skip activation quantization.  This is
// that layer's GEMM; the W8A8 layers run gemm_tc2.cu.
//
// A cluster of two CTAs (one per SM) computes a 256 x 256 output tile.  Each
// CTA loads its own 128 rows of X (A) and its own 128 rows of the 256-row W
// tile (B) with TMA straight into the 128-byte-swizzled K-major layout the
// tensor core reads (no staging copy, no conversion), and the leader CTA
// issues one M=256 N=256 K=16 bf16 MMA per K step over both CTAs' shared
// memory.  Per CTA: warp 0 TMA producer (both CTAs' loads complete on the
// leader's stage barrier, which the leader's producer arms for both CTAs'
// bytes), warp 1 TMEM allocation (both CTAs) and MMA issue (leader only),
// warps 4-7 drain the fp32 accumulator (double-buffered in TMEM, 2 x 256
// columns), add the bias and write bf16.  All waits are bounded in time.
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

#ifndef W8A8_BF16_SUB
#define W8A8_BF16_SUB 2
#endif
#ifndef W8A8_BF16_STAGES
#define W8A8_BF16_STAGES 3
#endif

constexpr int PAIR_M = 256, CTA_M = 128, PAIR_N = 256, CTA_N = 128;
constexpr int BK = 64;                                // bf16 per 128-byte swizzle row
constexpr int SUB = W8A8_BF16_SUB;                    // K = 64 boxes per stage
constexpr int S = W8A8_BF16_STAGES;
constexpr int BOX_A = CTA_M * BK * 2, BOX_B = CTA_N * BK * 2;   // 16 KB each
constexpr int SUB_BYTES = BOX_A + BOX_B;
constexpr int STAGE = SUB * SUB_BYTES;
constexpr int THREADS = 256;
constexpr int TMEM_COLS = 512;
constexpr int SMEM_BARRIERS = 256;
constexpr int SMEM_TOTAL = 1024 + S * STAGE + SMEM_BARRIERS;
static_assert(SMEM_TOTAL <= 232448, "shared memory");

constexpr unsigned ERR_PRODUCER = 1u, ERR_MMA = 4u, ERR_EPILOGUE = 8u, ERR_DRAIN = 16u,
                   ERR_TMEM_PAIR = 64u;

constexpr uint32_t OFF_ST = 0;
constexpr uint32_t OFF_BAR = OFF_ST + S * STAGE;
constexpr uint32_t BAR_PFULL = OFF_BAR;               // leader: both CTAs' bytes landed
constexpr uint32_t BAR_EMPTY = BAR_PFULL + 8 * S;     // local: MMA done with the stage
constexpr uint32_t BAR_ACCFULL = BAR_EMPTY + 8 * S;
constexpr uint32_t BAR_ACCEMPTY = BAR_ACCFULL + 16;
constexpr uint32_t BAR_DRAIN = BAR_ACCEMPTY + 16;
constexpr uint32_t OFF_TMEM = BAR_DRAIN + 8;
constexpr uint32_t OFF_ABORT = OFF_TMEM + 4;
static_assert(OFF_ABORT + 4 - OFF_BAR <= SMEM_BARRIERS, "barrier area");

constexpr int NUM_EPI_WARPS = 4;

// kind::f16 instruction descriptor with bf16 A and B (K-major), fp32 D.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4)                                    // D format: f32
           | (1u << 7) | (1u << 10)                     // A, B format: bf16
           | (static_cast<uint32_t>(N >> 3) << 17)
           | (static_cast<uint32_t>(M >> 4) << 24);
}

struct Params {
    const float *bias;
    uint16_t *Y;
    int M, N, K;
    int m_tiles, total_tiles, k_blocks;
    int n_tiles, group;        // feature tiles; tile order (tile_order.cuh)
    unsigned int *err;
    uint64_t wait_limit_ns;
};

// Row offsets of tile t's tokens (m0) and features (n0).
__device__ __forceinline__ void tile_mn(const Params &p, int t, int &m0, int &n0) {
    int mi, ni;
    grouped_tile(t, p.m_tiles, p.n_tiles, p.group, mi, ni);
    m0 = mi * PAIR_M;
    n0 = ni * PAIR_N;
}


__device__ __forceinline__ void epilogue_role(const Params &p, uint32_t sb, uint32_t tmem,
                                              const WaitCtx &wc, int warp, int lane,
                                              uint32_t rank, int pair, int npairs) {
    const int q = warp & 3;                          // TMEM lane quarter of this warp
    uint32_t c = 0;
    for (int t = pair; t < p.total_tiles; t += npairs, ++c) {
        const uint32_t buf = c & 1;
        if (!mbar_wait_cluster(sb + BAR_ACCFULL + 8 * buf, (c >> 1) & 1, wc, ERR_EPILOGUE)) break;
        tc_fence_after();
        int m0, n0;
        tile_mn(p, t, m0, n0);
        const int m = m0 + static_cast<int>(rank) * CTA_M + q * 32 + lane;
        const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * PAIR_N;
        uint16_t *out = p.Y + (size_t)m * p.N + n0;
#pragma unroll 1
        for (int cc = 0; cc < PAIR_N / 16; ++cc) {
            uint32_t v[16];
            tmem_ld_32x32b_x16(base + cc * 16, v);
            tmem_ld_wait();
            const int n = n0 + cc * 16;
            float b[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) b[i] = 0.0f;
            if (p.bias != nullptr) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (n + 8 * h < p.N) {
                        const float4 b0 = __ldg(reinterpret_cast<const float4 *>(p.bias + n + 8 * h));
                        const float4 b1 = __ldg(reinterpret_cast<const float4 *>(p.bias + n + 8 * h + 4));
                        b[8 * h + 0] = b0.x; b[8 * h + 1] = b0.y; b[8 * h + 2] = b0.z; b[8 * h + 3] = b0.w;
                        b[8 * h + 4] = b1.x; b[8 * h + 5] = b1.y; b[8 * h + 6] = b1.z; b[8 * h + 7] = b1.w;
                    }
                }
            }
            if (m < p.M) {
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (n + 8 * h < p.N) {
                        uint32_t w[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float y0 = __fadd_rn(__uint_as_float(v[8 * h + 2 * i]), b[8 * h + 2 * i]);
                            const float y1 = __fadd_rn(__uint_as_float(v[8 * h + 2 * i + 1]), b[8 * h + 2 * i + 1]);
                            // one conversion instruction per pair (round to
                            // nearest even; a NaN becomes the canonical one)
                            w[i] = pack_bf16x2_cvt(y0, y1);
                        }
                        *reinterpret_cast<uint4 *>(out + cc * 16 + 8 * h) = make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
            }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
            if (rank == 0) mbar_arrive(sb + BAR_ACCEMPTY + 8 * buf);
            else mbar_arrive_cluster_relaxed(mapa_shared(sb + BAR_ACCEMPTY + 8 * buf, 0));
        }
    }
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_bf16_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const Params p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sb = (smem_addr(smem_raw) + 1023u) & ~1023u;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    const int npairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int i = 0; i < S; ++i) {
            mbar_init(sb + BAR_PFULL + 8 * i, 1);
            mbar_init(sb + BAR_EMPTY + 8 * i, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(sb + BAR_ACCFULL + 8 * i, 1);
            mbar_init(sb + BAR_ACCEMPTY + 8 * i, 2 * NUM_EPI_WARPS);
        }
        mbar_init(sb + BAR_DRAIN, 1);
        st_shared_s32(sb + OFF_ABORT, 0);
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) {
        tmem_alloc_pair(sb + OFF_TMEM, TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(ld_shared_s32(sb + OFF_TMEM));
    const uint32_t peer_tmem = ld_shared_cluster_u32(mapa_shared(sb + OFF_TMEM, rank ^ 1u));
    const bool run_ok = (tmem == peer_tmem);
    if (!run_ok && threadIdx.x == 0) atomicOr(p.err, ERR_TMEM_PAIR);
    wait_prior_grid();
    const WaitCtx wc{sb + OFF_ABORT, p.err, p.wait_limit_ns};
    const int NS = (p.k_blocks + SUB - 1) / SUB;           // stages per tile

    if (!run_ok) {
    } else if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            uint32_t j = 0;
            bool ok = true;
            for (int t = pair; ok && t < p.total_tiles; t += npairs) {
                int m0, n0;
                tile_mn(p, t, m0, n0);
                const int arow = m0 + static_cast<int>(rank) * CTA_M;
                const int brow = n0 + static_cast<int>(rank) * CTA_N;
                for (int ks = 0; ks < NS; ++ks, ++j) {
                    const uint32_t st = j % S;
                    if (!mbar_wait_cluster(sb + BAR_EMPTY + 8 * st, ((j / S) & 1) ^ 1, wc, ERR_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    // both CTAs' loads complete on the leader's barrier (the
                    // MMA waits for every stage, so each load has landed
                    // before the kernel ends)
                    const uint32_t fb = mapa_shared(sb + BAR_PFULL + 8 * st, 0);
                    if (leader) mbar_arrive_expect_tx(sb + BAR_PFULL + 8 * st, 2 * STAGE);
#pragma unroll
                    for (int u = 0; u < SUB; ++u) {
                        const uint32_t dst = sb + OFF_ST + st * STAGE + u * SUB_BYTES;
                        tma_load_2d_pair(dst, &tmA, (ks * SUB + u) * BK, arow, fb);
                        tma_load_2d_pair(dst + BOX_A, &tmB, (ks * SUB + u) * BK, brow, fb);
                    }
                }
            }
        }
    } else if (warp == 1) {
        // --------------------------------------------- MMA issue (leader)
        if (lane == 0 && leader) {
            constexpr uint32_t idesc = idesc_bf16_f32(PAIR_M, PAIR_N);
            uint32_t j = 0, c = 0;
            bool ok = true;
            for (int t = pair; ok && t < p.total_tiles; t += npairs, ++c) {
                const uint32_t buf = c & 1;
                if (!mbar_wait_cluster(sb + BAR_ACCEMPTY + 8 * buf, ((c >> 1) & 1) ^ 1, wc, ERR_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + buf * PAIR_N;
                for (int ks = 0; ks < NS; ++ks, ++j) {
                    const uint32_t st = j % S;
                    if (!mbar_wait_cluster(sb + BAR_PFULL + 8 * st, (j / S) & 1, wc, ERR_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll
                    for (int u = 0; u < SUB; ++u) {
                        const uint32_t a = sb + OFF_ST + st * STAGE + u * SUB_BYTES;
                        const uint32_t b = a + BOX_A;
#pragma unroll
                        for (int kk = 0; kk < BK / 16; ++kk)
                            mma_f16_ss_pair(d, smem_desc_sw128(a + kk * 32), smem_desc_sw128(b + kk * 32),
                                            idesc, (ks > 0 || u > 0 || kk > 0) ? 1u : 0u);
                    }
                    mma_commit_pair_multicast(sb + BAR_EMPTY + 8 * st, 0x3);
                }
                if (ok) mma_commit_pair_multicast(sb + BAR_ACCFULL + 8 * buf, 0x3);
            }
            mma_commit_pair(sb + BAR_DRAIN);
            mbar_wait_cluster(sb + BAR_DRAIN, 0, wc, ERR_DRAIN, false);
        }
    } else if (warp >= 4) {
        epilogue_role(p, sb, tmem, wc, warp, lane, rank, pair, npairs);
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

// bf16 row-major [rows, K] -> 2-D map, box [128 rows, 64 elements] landing in
// the 128-byte swizzled layout, zero fill outside the matrix.
bool make_map_bf16(CUtensorMap *m, const uint16_t *base, int rows, int K) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(CTA_M)};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_gemm_bf16(const uint16_t *X, const uint16_t *W, const float *bias, int M,
                             int N, int K, uint16_t *Y, unsigned int *err, cudaStream_t st) {
    const int sms = device_sms();
    static PerDevice<int> attr;
    int unused = 0;
    cudaError_t e = attr.get([](int &) {
        return cudaFuncSetAttribute(gemm_bf16_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_TOTAL);
    }, &unused);
    if (e != cudaSuccess) return e;
    CUtensorMap mA, mB;
    if (!make_map_bf16(&mA, X, M, K) || !make_map_bf16(&mB, W, N, K)) return cudaErrorInvalidValue;
    Params p{};
    p.bias = bias;
    p.Y = Y;
    p.M = M;
    p.N = N;
    p.K = K;
    p.m_tiles = (M + PAIR_M - 1) / PAIR_M;
    p.n_tiles = (N + PAIR_N - 1) / PAIR_N;
    p.total_tiles = p.m_tiles * p.n_tiles;
    p.k_blocks = (K + BK - 1) / BK;
    // tile order (tile_order.cuh): bf16 activations and weights
    p.group = tile_group(2LL * K * M, 2LL * PAIR_N * K, p.n_tiles);
    p.err = err;
    p.wait_limit_ns = 2000000000ull;
    const int pairs = p.total_tiles < sms / 2 ? p.total_tiles : sms / 2;
    return launch_pdl(gemm_bf16_kernel, dim3(2 * pairs), THREADS, SMEM_TOTAL, st, mA, mB, p);
}

}  // namespace w8a8
