// stats.cu -- activation statistics for fragility profiling, and the
// per-tensor activation quantization of the ablation.
//
//   stats_update_kernel    per input channel j, accumulates max_t |x_tj| and
//                          the power sums sum_t (x_tj - c_j)^p, p = 1..4
//                          (Sec. 3, "Activation-fragility profiling and
//                          protection": max-abs, standard deviation and
//                          kurtosis of every linear's input, recorded over
//                          the denoising trajectory, so the sums accumulate
//                          over any number of calls)
//   stats_finalize_kernel  per-channel and whole-tensor max-abs, mean,
//                          population std and Pearson kurtosis from the sums
//   tensor_absmax_kernel   max over the whole tensor of |x_mj / lambda_j|
//   tensor_quant_kernel    INT8 codes of x_mj / lambda_j with that one scale
//                          (the naive per-tensor arm of the activation-quant
//                          ablation, Sec. 5, "What drives INT8 recovery")
//
// Layout of the streaming passes: a block is WR warps; lane l of every warp
// owns the same few columns (fixed per thread, so per-column factors stay in
// registers) and warp w takes rows w, w + WR, ... of the block's row slab, so
// a warp reads one contiguous run of the row per instruction and consecutive
// warps read consecutive rows.
#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"
#include "host_once.h"
#include "launch.h"

namespace w8a8 {
namespace {

int num_sms() { return device_sms(); }

// ----------------------------------------------------- packed fp32 helpers
// Two fp32 lanes per instruction (sm_100 family).  Used only in the
// statistics pass, whose result is compared within an error bound, so
// contraction of these operations does not matter.
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 r;
    asm("{\n.reg .b64 ra, rb, rr;\nmov.b64 ra, {%2, %3};\nmov.b64 rb, {%4, %5};\n"
        "add.rn.f32x2 rr, ra, rb;\nmov.b64 {%0, %1}, rr;\n}"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
    float2 r;
    asm("{\n.reg .b64 ra, rb, rr;\nmov.b64 ra, {%2, %3};\nmov.b64 rb, {%4, %5};\n"
        "mul.rn.f32x2 rr, ra, rb;\nmov.b64 {%0, %1}, rr;\n}"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    float2 r;
    asm("{\n.reg .b64 ra, rb, rc, rr;\nmov.b64 ra, {%2, %3};\nmov.b64 rb, {%4, %5};\n"
        "mov.b64 rc, {%6, %7};\nfma.rn.f32x2 rr, ra, rb, rc;\nmov.b64 {%0, %1}, rr;\n}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return r;
}

// ------------------------------------------------------------ statistics
//
// Lane l owns 4 consecutive channels of the block's 128 (one 8-byte load per
// row) and the 8 warps of a block split the block's row slab.  Each thread
// sums (x - c)^p in fp32 over groups of at most kGroup of its rows, adds the
// group sums into fp32 level-2 sums (at most kGroup groups), and only those
// into fp64 (at the end of the slab, or every kGroup groups); the block then
// combines its warps in fp64 through shared memory and adds into the global
// fp64 sums with atomics.  Rounding: every returned sum is within
// (2 kGroup + 4) * 2^-24 of sum |x - c|^p of its exact value.
constexpr int kStatsWarps = 8;
constexpr int kGroup = 64;
constexpr int kUnroll = 16;
static_assert(kGroup % kUnroll == 0, "whole unrolled batches per group");

struct Acc4 {                   // one moment for the thread's 4 channels
    float2 a, b;
};

__global__ void __launch_bounds__(32 * kStatsWarps, 2)
stats_update_kernel(const uint2 *__restrict__ X4, int T, int K, const float *__restrict__ shift,
                    int rows_per_slab, double *__restrict__ sums, float *__restrict__ absmax) {
    __shared__ double red_s[kStatsWarps][16][32];     // per-thread fp64 sums [p][e]
    __shared__ float lvl2[kStatsWarps][16][32];       // per-thread level-2 fp32 sums,
                                                      // then the maxima [e] (48 KB total)
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int quad = blockIdx.x * 32 + lane;            // 4-channel group index
    const int kq = K / 4;
    const bool active = quad < kq;
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(T, r0 + rows_per_slab);
    constexpr int kStep = kStatsWarps * kUnroll;

    float2 c0 = make_float2(0.0f, 0.0f), c1 = c0;     // -shift
    if (active && shift) {
        const float4 sh = __ldg(reinterpret_cast<const float4 *>(shift) + quad);
        c0 = make_float2(-sh.x, -sh.y);
        c1 = make_float2(-sh.z, -sh.w);
    }
    const float2 z = make_float2(0.f, 0.f);
    Acc4 g[4] = {{z, z}, {z, z}, {z, z}, {z, z}};      // level 1, p = 1..4
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        red_s[w][i][lane] = 0.0;
        lvl2[w][i][lane] = 0.0f;
    }
    float mx[4] = {0.f, 0.f, 0.f, 0.f};
    int rows_in_group = 0, groups = 0;

    // level 1 -> level 2 (every kGroup rows), level 2 -> fp64 (every kGroup
    // groups); both live in this thread's slots of shared memory
    auto fold_group = [&]() {
#pragma unroll
        for (int p = 0; p < 4; ++p) {
            lvl2[w][4 * p + 0][lane] += g[p].a.x;
            lvl2[w][4 * p + 1][lane] += g[p].a.y;
            lvl2[w][4 * p + 2][lane] += g[p].b.x;
            lvl2[w][4 * p + 3][lane] += g[p].b.y;
            g[p].a = z;
            g[p].b = z;
        }
        rows_in_group = 0;
        ++groups;
    };
    auto fold_level2 = [&]() {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            red_s[w][i][lane] += lvl2[w][i][lane];
            lvl2[w][i][lane] = 0.0f;
        }
        groups = 0;
    };
    auto load_batch = [&](int rb, uint2 (&v)[kUnroll]) {
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int r = rb + u * kStatsWarps;
            v[u] = (active && r < r1) ? __ldcs(X4 + (size_t)r * kq + quad) : make_uint2(0u, 0u);
        }
    };

    // two batches of kUnroll rows in flight: the next one loads while this
    // one is summed
    uint2 v[kUnroll];
    load_batch(r0 + w, v);
    for (int rb = r0 + w; rb < r1; rb += kStep) {
        uint2 vn[kUnroll];
        load_batch(rb + kStep, vn);
        // rows of this batch inside the slab
        const int valid = min(kUnroll, (r1 - rb + kStatsWarps - 1) / kStatsWarps);
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            if (u < valid) {
                const float2 xa = make_float2(__uint_as_float(v[u].x << 16), __uint_as_float(v[u].x & 0xffff0000u));
                const float2 xb = make_float2(__uint_as_float(v[u].y << 16), __uint_as_float(v[u].y & 0xffff0000u));
                mx[0] = fmaxf(mx[0], fabsf(xa.x));
                mx[1] = fmaxf(mx[1], fabsf(xa.y));
                mx[2] = fmaxf(mx[2], fabsf(xb.x));
                mx[3] = fmaxf(mx[3], fabsf(xb.y));
                const float2 da = add2(xa, c0), db = add2(xb, c1);
                const float2 da2 = mul2(da, da), db2 = mul2(db, db);
                g[0].a = add2(g[0].a, da);
                g[0].b = add2(g[0].b, db);
                g[1].a = add2(g[1].a, da2);
                g[1].b = add2(g[1].b, db2);
                g[2].a = fma2(da2, da, g[2].a);
                g[2].b = fma2(db2, db, g[2].b);
                g[3].a = fma2(da2, da2, g[3].a);
                g[3].b = fma2(db2, db2, g[3].b);
            }
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) v[u] = vn[u];
        rows_in_group += kUnroll;
        if (rows_in_group >= kGroup) {
            fold_group();
            if (groups >= kGroup) fold_level2();
        }
    }
    fold_group();
    fold_level2();
#pragma unroll
    for (int e = 0; e < 4; ++e) lvl2[w][e][lane] = mx[e];   // own slots: no other thread reads them yet
    __syncthreads();
    // warp p (p < 4) reduces moment p, warp 4 the maxima: 4 channels per lane
    if (active && r0 < r1 && w < 5) {
        if (w < 4) {
            double tot[4] = {0, 0, 0, 0};
            for (int ww = 0; ww < kStatsWarps; ++ww)
#pragma unroll
                for (int e = 0; e < 4; ++e) tot[e] += red_s[ww][4 * w + e][lane];
#pragma unroll
            for (int e = 0; e < 4; ++e) atomicAdd(sums + (size_t)w * K + 4 * quad + e, tot[e]);
        } else {
            float a[4] = {0.f, 0.f, 0.f, 0.f};
            for (int ww = 0; ww < kStatsWarps; ++ww)
#pragma unroll
                for (int e = 0; e < 4; ++e) a[e] = fmaxf(a[e], lvl2[ww][e][lane]);
            // non-negative floats order like their bit patterns
#pragma unroll
            for (int e = 0; e < 4; ++e)
                atomicMax(reinterpret_cast<unsigned int *>(absmax) + 4 * quad + e, __float_as_uint(a[e]));
        }
    }
}

// Central moments of channel j about its own mean from the sums about c_j:
// with n rows and e = S1/n (the mean minus c_j),
//   M2 = S2 - n e^2,  M3 = S3 - 3 e S2 + 2 n e^3,
//   M4 = S4 - 4 e S3 + 6 e^2 S2 - 3 n e^4   (binomial expansion of (d - e)^p).
// A computed M2 within the accumulation error of zero (1e-5 of S2) is a
// constant channel: variance 0, kurtosis 0.
struct Central {
    double mean, m2, m3, m4;
};

__device__ __forceinline__ Central central(const double *sums, const float *shift, int K, int j,
                                           double n) {
    const double S1 = sums[j], S2 = sums[(size_t)K + j], S3 = sums[2 * (size_t)K + j],
                 S4 = sums[3 * (size_t)K + j];
    const double e = S1 / n;
    Central r;
    r.mean = (shift ? (double)shift[j] : 0.0) + e;
    r.m2 = S2 - n * e * e;
    r.m3 = S3 - 3.0 * e * S2 + 2.0 * n * e * e * e;
    r.m4 = S4 - 4.0 * e * S3 + 6.0 * e * e * S2 - 3.0 * n * e * e * e * e;
    if (!(r.m2 > 1e-5 * S2)) {
        r.m2 = 0.0;
        r.m3 = 0.0;
        r.m4 = 0.0;
    }
    return r;
}

constexpr int kFinThreads = 1024;

__device__ __forceinline__ double block_sum(double v, double *red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    double t = 0.0;
    for (int i = 0; i < kFinThreads / 32; ++i) t += red[i];
    return t;
}

__global__ void __launch_bounds__(kFinThreads)
stats_finalize_kernel(const double *__restrict__ sums, const float *__restrict__ absmax,
                      const float *__restrict__ shift, double n, int K, float *__restrict__ chan,
                      float *__restrict__ tensor) {
    __shared__ double red[kFinThreads / 32];
    double mean_sum = 0.0, amax = 0.0;
    for (int j = threadIdx.x; j < K; j += kFinThreads) {
        const Central c = central(sums, shift, K, j, n);
        const double var = c.m2 / n;
        chan[j] = absmax[j];
        chan[(size_t)K + j] = static_cast<float>(c.mean);
        chan[2 * (size_t)K + j] = static_cast<float>(sqrt(var));
        chan[3 * (size_t)K + j] = static_cast<float>(var > 0.0 ? (c.m4 / n) / (var * var) : 0.0);
        mean_sum += c.mean;
        amax = fmax(amax, (double)absmax[j]);
    }
    // whole tensor: pool the channels about the grand mean mu (all channels
    // have n rows), with delta_j = mean_j - mu:
    //   M2 = sum_j M2_j + n delta_j^2,
    //   M4 = sum_j M4_j + 4 delta_j M3_j + 6 delta_j^2 M2_j + n delta_j^4
    const double mu = block_sum(mean_sum, red) / K;
    double t2 = 0.0, t4 = 0.0, ss = 0.0;
    for (int j = threadIdx.x; j < K; j += kFinThreads) {
        const Central c = central(sums, shift, K, j, n);
        const double dl = c.mean - mu;
        t2 += c.m2 + n * dl * dl;
        t4 += c.m4 + 4.0 * dl * c.m3 + 6.0 * dl * dl * c.m2 + n * dl * dl * dl * dl;
        // size of the pooled second moment's terms about mu, for the
        // constant-tensor test (same criterion as per channel)
        ss += sums[(size_t)K + j] + n * dl * dl;
    }
    const double T2 = block_sum(t2, red), T4 = block_sum(t4, red), SS = block_sum(ss, red);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) amax = fmax(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
    __syncthreads();
    if (threadIdx.x == 0) {
        double am = 0.0;
        for (int i = 0; i < kFinThreads / 32; ++i) am = fmax(am, red[i]);
        const double nt = n * K;
        const double var = (T2 > 1e-5 * SS) ? T2 / nt : 0.0;
        tensor[0] = static_cast<float>(am);
        tensor[1] = static_cast<float>(mu);
        tensor[2] = static_cast<float>(sqrt(var));
        tensor[3] = static_cast<float>(var > 0.0 ? (T4 / nt) / (var * var) : 0.0);
    }
}

// ------------------------------------------------- per-tensor quantization
//
// Lane l owns 8 consecutive columns of the block's 256 (16-byte loads, 1/lambda
// of its columns in registers).
constexpr int kQWarps = 8;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ void load_recip(const float *lam, int col0, bool active, float (&r)[8]) {
#pragma unroll
    for (int e = 0; e < 8; ++e) r[e] = (lam != nullptr && active) ? __frcp_rn(__ldg(lam + col0 + e)) : 1.0f;
}

__global__ void __launch_bounds__(32 * kQWarps)
tensor_absmax_kernel(const uint16_t *__restrict__ X, const float *__restrict__ lam, int M, int K,
                     int rows_per_slab, float *__restrict__ amax) {
    __shared__ float red[kQWarps];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int col0 = (blockIdx.x * 32 + lane) * 8;
    const bool active = col0 < K;
    float r[8];
    load_recip(lam, col0, active, r);
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(M, r0 + rows_per_slab);
    float a = 0.0f;
    for (int rb = r0 + w; rb < r1; rb += kQWarps * 4) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int row = rb + u * kQWarps;
            v[u] = (active && row < r1) ? __ldcs(reinterpret_cast<const uint4 *>(X + (size_t)row * K + col0))
                                        : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                a = fmaxf(a, fabsf(__fmul_rn(__uint_as_float(wd[e] << 16), r[2 * e])));
                a = fmaxf(a, fabsf(__fmul_rn(__uint_as_float(wd[e] & 0xffff0000u), r[2 * e + 1])));
            }
        }
    }
    a = warp_max(a);
    if (lane == 0) red[w] = a;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.0f;
        for (int i = 0; i < kQWarps; ++i) t = fmaxf(t, red[i]);
        atomicMax(reinterpret_cast<unsigned int *>(amax), __float_as_uint(t));
    }
}

constexpr float kRoundMagic = 12582912.0f;   // 1.5 * 2^23: low byte of the sum = rne(y)

__device__ __forceinline__ uint32_t pack4_low_bytes(float a, float b, float c, float d) {
    const uint32_t ab = __byte_perm(__float_as_uint(a), __float_as_uint(b), 0x0040);
    const uint32_t cd = __byte_perm(__float_as_uint(c), __float_as_uint(d), 0x0040);
    return __byte_perm(ab, cd, 0x5410);
}

__global__ void __launch_bounds__(32 * kQWarps)
tensor_quant_kernel(const uint16_t *__restrict__ X, const float *__restrict__ lam, int M, int K,
                    int rows_per_slab, const float *__restrict__ amax, int8_t *__restrict__ Xq,
                    float *__restrict__ x_scale) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int col0 = (blockIdx.x * 32 + lane) * 8;
    const bool active = col0 < K;
    float r[8];
    load_recip(lam, col0, active, r);
    const float a = *amax;                       // written by the previous kernel
    const bool zero = (a == 0.0f);
    const float inv = zero ? 0.0f : __fdiv_rn(127.0f, a);
    const float scale = zero ? 0.0f : __fdiv_rn(a, 127.0f);
    // a and 127/a finite: |x' * inv| <= 127 (1 + 2^-23), no clamp needed
    const bool fast = (a <= 3.402823466e38f) && (inv <= 3.402823466e38f);
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(M, r0 + rows_per_slab);
    for (int rb = r0 + w; rb < r1; rb += kQWarps * 4) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int row = rb + u * kQWarps;
            v[u] = (active && row < r1) ? __ldcs(reinterpret_cast<const uint4 *>(X + (size_t)row * K + col0))
                                        : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int row = rb + u * kQWarps;
            if (row >= r1) continue;
            if (blockIdx.x == 0 && lane == 0) x_scale[row] = scale;
            if (!active) continue;
            const uint32_t wd[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
            float xs[8];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                xs[2 * e] = __fmul_rn(__uint_as_float(wd[e] << 16), r[2 * e]);
                xs[2 * e + 1] = __fmul_rn(__uint_as_float(wd[e] & 0xffff0000u), r[2 * e + 1]);
            }
            uint32_t word[2] = {0u, 0u};
            if (zero) {
            } else if (fast) {
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    word[h] = pack4_low_bytes(__fadd_rn(__fmul_rn(xs[4 * h], inv), kRoundMagic),
                                              __fadd_rn(__fmul_rn(xs[4 * h + 1], inv), kRoundMagic),
                                              __fadd_rn(__fmul_rn(xs[4 * h + 2], inv), kRoundMagic),
                                              __fadd_rn(__fmul_rn(xs[4 * h + 3], inv), kRoundMagic));
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const uint32_t b = static_cast<uint32_t>(quantize_rne_clamp(__fmul_rn(xs[e], inv))) & 0xffu;
                    word[e >> 2] |= b << (8 * (e & 3));
                }
            }
            *reinterpret_cast<uint2 *>(Xq + (size_t)row * K + col0) = make_uint2(word[0], word[1]);
        }
    }
}

// Resident blocks per SM of `kern` (no dynamic shared memory), looked up once
// per device.
template <typename Kern>
int blocks_per_sm(PerDevice<int> &cache, Kern kern, int threads) {
    int v = 1;
    if (cache.get([&](int &n) {
            cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, 0);
            if (n < 1) n = 1;
            return e;
        }, &v) != cudaSuccess)
        return 1;
    return v;
}

// Row slabs so that a (gx x gy) grid fills the GPU once: gy = the resident
// blocks on all SMs divided by gx, at most one slab per row.
int slabs_for(int per_sm, int rows, int gx) {
    int gy = (num_sms() * per_sm) / gx;
    if (gy > rows) gy = rows;
    if (gy < 1) gy = 1;
    return gy;
}

// One-shot statistics without caller accumulators: a file-scope scratch of
// power sums (4 x max K doubles) then max-abs (max K floats), cleared at the
// start of every call.  Calls that overlap in time share it.
constexpr int kNoAllocMaxK = W8A8_NOALLOC_STATS_MAX_K;
static __device__ __align__(256) unsigned char g_stats_scratch[kNoAllocMaxK * (4 * sizeof(double) + sizeof(float))];

// Device address of the scratch on the current device, looked up once per
// device (the lookup is not a stream operation: do it before any capture).
void *stats_scratch_address() {
    static PerDevice<void *> addr;
    void *p = nullptr;
    if (addr.get([](void *&v) { return cudaGetSymbolAddress(&v, g_stats_scratch); }, &p) != cudaSuccess)
        return nullptr;
    return p;
}

}  // namespace

cudaError_t launch_act_stats_update(const uint16_t *X, int T, int K, const float *shift,
                                    double *sums, float *absmax, cudaStream_t st) {
    const int gx = (K / 4 + 31) / 32;
    static PerDevice<int> occ;
    int gy = slabs_for(blocks_per_sm(occ, stats_update_kernel, 32 * kStatsWarps), T, gx);
    const int rows_per_slab = (T + gy - 1) / gy;
    gy = (T + rows_per_slab - 1) / rows_per_slab;
    stats_update_kernel<<<dim3(gx, gy), 32 * kStatsWarps, 0, st>>>(
        reinterpret_cast<const uint2 *>(X), T, K, shift, rows_per_slab, sums, absmax);
    return cudaGetLastError();
}

cudaError_t launch_act_stats_finalize(const double *sums, const float *absmax, const float *shift,
                                      long long count, int K, float *chan, float *tensor,
                                      cudaStream_t st) {
    stats_finalize_kernel<<<1, kFinThreads, 0, st>>>(sums, absmax, shift, (double)count, K, chan,
                                                     tensor);
    return cudaGetLastError();
}

cudaError_t launch_quant_act_per_tensor(const uint16_t *X, const float *lambda, int M, int K,
                                        int8_t *Xq, float *x_scale, float *amax, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(amax, 0, sizeof(float), st);
    if (e != cudaSuccess) return e;
    const int gx = (K / 8 + 31) / 32;
    static PerDevice<int> occ1, occ2;
    const int gy1 = slabs_for(blocks_per_sm(occ1, tensor_absmax_kernel, 32 * kQWarps), M, gx);
    const int gy2 = slabs_for(blocks_per_sm(occ2, tensor_quant_kernel, 32 * kQWarps), M, gx);
    const int rps1 = (M + gy1 - 1) / gy1, rps2 = (M + gy2 - 1) / gy2;
    tensor_absmax_kernel<<<dim3(gx, (M + rps1 - 1) / rps1), 32 * kQWarps, 0, st>>>(X, lambda, M, K,
                                                                                   rps1, amax);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    tensor_quant_kernel<<<dim3(gx, (M + rps2 - 1) / rps2), 32 * kQWarps, 0, st>>>(
        X, lambda, M, K, rps2, amax, Xq, x_scale);
    return cudaGetLastError();
}

}  // namespace w8a8

namespace w8a8 {

cudaError_t launch_act_stats_noalloc(const uint16_t *X, int T, int K, const float *shift, float *chan,
                                     float *tensor, cudaStream_t st) {
    void *base = stats_scratch_address();
    if (!base) return cudaErrorInvalidSymbol;
    double *sums = static_cast<double *>(base);
    float *absmax = reinterpret_cast<float *>(sums + 4 * static_cast<size_t>(kNoAllocMaxK));
    cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(double) * 4 * static_cast<size_t>(K), st);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(absmax, 0, sizeof(float) * static_cast<size_t>(K), st);
    if (e != cudaSuccess) return e;
    e = launch_act_stats_update(X, T, K, shift, sums, absmax, st);
    if (e != cudaSuccess) return e;
    return launch_act_stats_finalize(sums, absmax, shift, T, K, chan, tensor, st);
}

}  // namespace w8a8
