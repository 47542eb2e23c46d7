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
#include "launch.h"

namespace w8a8 {
namespace {

int g_sms = 0;

int num_sms() {
    if (g_sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_sms <= 0) g_sms = 148;
    }
    return g_sms;
}

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
// Lane l owns the channel pair (2l, 2l+1) of the block's 64 channels.  Each
// thread sums (x - c)^p in fp32 over at most kGroup of its rows, then adds
// the group sums into fp64 registers; the block combines its warps in fp64
// through shared memory and adds into the global fp64 sums with atomics.
// Rounding: every fp32 group sum is within (kGroup + 4) * 2^-24 of
// sum |x - c|^p over the group, fp64 adds are exact to ~2^-53.
constexpr int kStatsWarps = 16;
constexpr int kGroup = 64;
constexpr int kUnroll = 16;

__global__ void __launch_bounds__(32 * kStatsWarps, 2)
stats_update_kernel(const uint32_t *__restrict__ X2, int T, int K, const float *__restrict__ shift,
                    int rows_per_slab, double *__restrict__ sums, float *__restrict__ absmax) {
    __shared__ double red_s[kStatsWarps][8][32];
    __shared__ float red_m[kStatsWarps][2][32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int pair = blockIdx.x * 32 + lane;            // channel pair index
    const int kp = K / 2;
    const bool active = pair < kp;
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(T, r0 + rows_per_slab);

    float2 c = make_float2(0.0f, 0.0f);
    if (active && shift) c = make_float2(-__ldg(shift + 2 * pair), -__ldg(shift + 2 * pair + 1));
    float2 s1 = make_float2(0.f, 0.f), s2 = s1, s3 = s1, s4 = s1;
    double S[8] = {0, 0, 0, 0, 0, 0, 0, 0};          // p-major: S[2(p-1) + e]
    float m0 = 0.0f, m1 = 0.0f;
    int in_group = 0;

    for (int rb = r0 + w; rb < r1; rb += kStatsWarps * kUnroll) {
        uint32_t v[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int r = rb + u * kStatsWarps;
            v[u] = (active && r < r1) ? __ldcs(X2 + (size_t)r * kp + pair) : 0u;
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int r = rb + u * kStatsWarps;
            if (r < r1) {
                const float2 x = make_float2(__uint_as_float(v[u] << 16), __uint_as_float(v[u] & 0xffff0000u));
                m0 = fmaxf(m0, fabsf(x.x));
                m1 = fmaxf(m1, fabsf(x.y));
                const float2 d = add2(x, c);
                const float2 d2 = mul2(d, d);
                s1 = add2(s1, d);
                s2 = add2(s2, d2);
                s3 = fma2(d2, d, s3);
                s4 = fma2(d2, d2, s4);
                ++in_group;
            }
        }
        if (in_group >= kGroup - kUnroll) {            // fold before kGroup rows pile up
            S[0] += s1.x; S[1] += s1.y; S[2] += s2.x; S[3] += s2.y;
            S[4] += s3.x; S[5] += s3.y; S[6] += s4.x; S[7] += s4.y;
            s1 = make_float2(0.f, 0.f); s2 = s1; s3 = s1; s4 = s1;
            in_group = 0;
        }
    }
    S[0] += s1.x; S[1] += s1.y; S[2] += s2.x; S[3] += s2.y;
    S[4] += s3.x; S[5] += s3.y; S[6] += s4.x; S[7] += s4.y;

#pragma unroll
    for (int i = 0; i < 8; ++i) red_s[w][i][lane] = S[i];
    red_m[w][0][lane] = m0;
    red_m[w][1][lane] = m1;
    __syncthreads();
    if (w == 0 && active && r0 < r1) {
        double tot[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        float a0 = 0.0f, a1 = 0.0f;
        for (int ww = 0; ww < kStatsWarps; ++ww) {
#pragma unroll
            for (int i = 0; i < 8; ++i) tot[i] += red_s[ww][i][lane];
            a0 = fmaxf(a0, red_m[ww][0][lane]);
            a1 = fmaxf(a1, red_m[ww][1][lane]);
        }
#pragma unroll
        for (int p = 0; p < 4; ++p) {
            atomicAdd(sums + (size_t)p * K + 2 * pair, tot[2 * p]);
            atomicAdd(sums + (size_t)p * K + 2 * pair + 1, tot[2 * p + 1]);
        }
        // non-negative floats order like their bit patterns
        atomicMax(reinterpret_cast<unsigned int *>(absmax) + 2 * pair, __float_as_uint(a0));
        atomicMax(reinterpret_cast<unsigned int *>(absmax) + 2 * pair + 1, __float_as_uint(a1));
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

// Row slabs so that the grid fills the GPU about `waves` times over.
int slabs_for(int rows, int gx, int blocks_per_sm) {
    int gy = (num_sms() * blocks_per_sm + gx - 1) / gx;
    if (gy > rows) gy = rows;
    if (gy < 1) gy = 1;
    return gy;
}

}  // namespace

cudaError_t launch_act_stats_update(const uint16_t *X, int T, int K, const float *shift,
                                    double *sums, float *absmax, cudaStream_t st) {
    const int gx = (K / 2 + 31) / 32;
    int gy = slabs_for(T, gx, 2);
    const int rows_per_slab = (T + gy - 1) / gy;
    gy = (T + rows_per_slab - 1) / rows_per_slab;
    stats_update_kernel<<<dim3(gx, gy), 32 * kStatsWarps, 0, st>>>(
        reinterpret_cast<const uint32_t *>(X), T, K, shift, rows_per_slab, sums, absmax);
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
    int gy = slabs_for(M, gx, 8);
    const int rows_per_slab = (M + gy - 1) / gy;
    gy = (M + rows_per_slab - 1) / rows_per_slab;
    tensor_absmax_kernel<<<dim3(gx, gy), 32 * kQWarps, 0, st>>>(X, lambda, M, K, rows_per_slab, amax);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    tensor_quant_kernel<<<dim3(gx, gy), 32 * kQWarps, 0, st>>>(X, lambda, M, K, rows_per_slab, amax,
                                                                Xq, x_scale);
    return cudaGetLastError();
}

}  // namespace w8a8
