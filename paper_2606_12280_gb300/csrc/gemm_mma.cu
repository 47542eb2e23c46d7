// gemm_mma.cu -- INT8 x INT8 -> INT32 GEMM on the legacy warp-level tensor
// path (mma.sync.m16n8k32 s8, native int32 accumulation) with the
// dequantizing epilogue fused (a4 + a5 of the W8A8 layer, Sec. 3 "INT8 W8A8";
// the fused kernel the paper lists as missing, Sec. 7 Limitations).
//
// It is the exact-integer anchor of the library and the measured "native
// INT8" engine of this GPU.  128x128 output tile per CTA, K step 64, 8 warps
// (2 x 4, 64x32 per warp), 3-stage cp.async pipeline into padded shared
// memory (80-byte rows, so ldmatrix phases touch 8 distinct 16-byte bank
// groups).  Rows beyond M, N and K are zero-filled by cp.async.
#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"
#include "host_once.h"
#include "launch.h"

namespace w8a8 {
namespace {

constexpr int BM = 128, BN = 128, BK = 64, STAGES = 3, PITCH = 80;
constexpr int TILE_BYTES = BM * PITCH;                 // one operand, one stage
constexpr int SMEM_BYTES = STAGES * 2 * TILE_BYTES;    // 61440

struct Branches {
    GemmBranch b[2];
};

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, bool valid) {
    const int n = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                        uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma_s8(int32_t (&d)[4], const uint32_t (&a)[4],
                                       uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, "
        "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <bool OUT_I32>
__global__ void __launch_bounds__(256)
gemm_mma_kernel(Branches brs, int N, int K) {
    extern __shared__ __align__(128) uint8_t smem[];
    const GemmBranch &br = brs.b[blockIdx.z];
    const int M = br.M;
    const int m0 = blockIdx.y * BM;
    const int n0 = blockIdx.x * BN;
    if (m0 >= M) return;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int wm = warp >> 2, wn = warp & 3;
    const int8_t *__restrict__ A = br.Xq;
    const int8_t *__restrict__ B = br.Wq;
    const int KT = (K + BK - 1) / BK;

    auto stage_a = [&](int s) { return smem + s * 2 * TILE_BYTES; };
    auto stage_b = [&](int s) { return smem + s * 2 * TILE_BYTES + TILE_BYTES; };

    auto load_stage = [&](int s, int kt) {
        const int k0 = kt * BK;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int c = tid + i * 256;           // 512 chunks of 16 bytes
            const int r = c >> 2, kc = (c & 3) * 16;
            const bool kin = (k0 + kc) < K;
            const int ar = m0 + r, bn = n0 + r;
            const bool av = kin && ar < M, bv = kin && bn < N;
            cp_async16(smem_u32(stage_a(s) + r * PITCH + kc),
                       av ? (const void *)(A + (size_t)ar * K + k0 + kc) : (const void *)A, av);
            cp_async16(smem_u32(stage_b(s) + r * PITCH + kc),
                       bv ? (const void *)(B + (size_t)bn * K + k0 + kc) : (const void *)B, bv);
        }
    };

    int32_t acc[4][4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[i][j][e] = 0;

#pragma unroll
    for (int s = 0; s < STAGES - 1; ++s) {
        if (s < KT) load_stage(s, s);
        asm volatile("cp.async.commit_group;\n" ::);
    }

    for (int kt = 0; kt < KT; ++kt) {
        asm volatile("cp.async.wait_group %0;\n" ::"n"(STAGES - 2));
        __syncthreads();
        const int nk = kt + STAGES - 1;
        if (nk < KT) load_stage(nk % STAGES, nk);
        asm volatile("cp.async.commit_group;\n" ::);

        const uint8_t *sa = stage_a(kt % STAGES);
        const uint8_t *sb = stage_b(kt % STAGES);
#pragma unroll
        for (int ks = 0; ks < BK; ks += 32) {
            uint32_t af[4][4];
#pragma unroll
            for (int mi = 0; mi < 4; ++mi) {
                const int j = lane >> 3;
                const int r = wm * 64 + mi * 16 + (j & 1) * 8 + (lane & 7);
                const int kb = ks + (j >> 1) * 16;
                ldsm_x4(smem_u32(sa + r * PITCH + kb), af[mi][0], af[mi][1], af[mi][2], af[mi][3]);
            }
            uint32_t bf[4][2];
#pragma unroll
            for (int np = 0; np < 2; ++np) {
                const int j = lane >> 3;
                const int n = wn * 32 + (np * 2 + (j >> 1)) * 8 + (lane & 7);
                const int kb = ks + (j & 1) * 16;
                ldsm_x4(smem_u32(sb + n * PITCH + kb), bf[np * 2][0], bf[np * 2][1],
                        bf[np * 2 + 1][0], bf[np * 2 + 1][1]);
            }
#pragma unroll
            for (int mi = 0; mi < 4; ++mi)
#pragma unroll
                for (int ni = 0; ni < 4; ++ni) mma_s8(acc[mi][ni], af[mi], bf[ni][0], bf[ni][1]);
        }
    }
    asm volatile("cp.async.wait_group 0;\n" ::);

    // epilogue
    const int g = lane >> 2, t4 = lane & 3;
#pragma unroll
    for (int mi = 0; mi < 4; ++mi) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int r = m0 + wm * 64 + mi * 16 + g + h * 8;
            if (r >= M) continue;
            float sx = 0.0f;
            if (!OUT_I32) sx = __ldg(br.x_scale + r);
#pragma unroll
            for (int ni = 0; ni < 4; ++ni) {
                const int c = n0 + wn * 32 + ni * 8 + t4 * 2;
                if (c >= N) continue;
                const int32_t v0 = acc[mi][ni][h * 2], v1 = acc[mi][ni][h * 2 + 1];
                if (OUT_I32) {
                    *reinterpret_cast<int2 *>(static_cast<int32_t *>(br.out) + (size_t)r * N + c) =
                        make_int2(v0, v1);
                } else {
                    const bool hb = br.bias != nullptr;
                    const float b0 = hb ? __ldg(br.bias + c) : 0.0f;
                    const float b1 = hb ? __ldg(br.bias + c + 1) : 0.0f;
                    const uint32_t y0 = epilogue_value(v0, sx, __ldg(br.w_scale + c), b0, hb);
                    const uint32_t y1 = epilogue_value(v1, sx, __ldg(br.w_scale + c + 1), b1, hb);
                    *reinterpret_cast<uint32_t *>(static_cast<uint16_t *>(br.out) + (size_t)r * N + c) =
                        y0 | (y1 << 16);
                }
            }
        }
    }
}

}  // namespace

cudaError_t launch_gemm_mma(const GemmBranch *br, int nb, int N, int K, bool out_i32,
                            cudaStream_t st) {
    Branches bs{};
    int maxM = 0;
    for (int i = 0; i < nb; ++i) {
        bs.b[i] = br[i];
        if (br[i].M > maxM) maxM = br[i].M;
    }
    if (maxM == 0) return cudaSuccess;
    dim3 grid((N + BN - 1) / BN, (maxM + BM - 1) / BM, nb);
    static PerDevice<int> attr[2];
    int unused = 0;
    cudaError_t e = attr[out_i32 ? 1 : 0].get([&](int &) {
        return cudaFuncSetAttribute(out_i32 ? gemm_mma_kernel<true> : gemm_mma_kernel<false>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    }, &unused);
    if (e != cudaSuccess) return e;
    if (out_i32) gemm_mma_kernel<true><<<grid, 256, SMEM_BYTES, st>>>(bs, N, K);
    else gemm_mma_kernel<false><<<grid, 256, SMEM_BYTES, st>>>(bs, N, K);
    return cudaGetLastError();
}

}  // namespace w8a8
