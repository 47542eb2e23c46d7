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
//   stats_channels_kernel  per-channel max-abs, mean, population std and
//   stats_tensor_kernel    Pearson kurtosis from the sums, then the same four
//                          over the whole tensor
//   tensor_absmax_kernel   max over the whole tensor of |x_mj / lambda_j|
//   tensor_quant_kernel    INT8 codes of x_mj / lambda_j with that one scale
//                          (the naive per-tensor arm of the activation-quant
//                          ablation, Sec. 5, "What drives INT8 recovery")
//
// Layout of the streaming passes: a block is 8 warps; lane l of every warp
// owns the same 8 columns (fixed per thread, so per-column factors and sums
// stay in registers) and warp w takes rows w, w + 8, ... of the block's row
// slab, so a warp reads 512 contiguous bytes of a row per copy and
// consecutive warps read consecutive rows.  Rows reach the threads through
// per-thread cp.async rings in shared memory; the grids fill the GPU once.
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

// ------------------------------------------------- streaming through rings
//
// The passes below stream rows through a per-thread ring of 16-byte slots in
// shared memory filled with cp.async: a thread copies its own chunks and reads
// back only those, so no barrier is needed, and the bytes in flight take no
// registers.  One commit group per row: waiting until at most S - 1 groups
// are pending makes the oldest row of an S-deep ring visible.
__device__ __forceinline__ void ring_cp16(uint32_t dst, const void *src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(valid ? 16 : 0) : "memory");
}

__device__ __forceinline__ void ring_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

template <int S>
__device__ __forceinline__ void ring_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(S - 1) : "memory");
}

__device__ __forceinline__ void ring_drain() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ uint4 ring_lds(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

// max(|a|, |b|) of each bf16 half (max.xorsign.abs keeps the larger
// magnitude; the sign bit of the result is meaningless and is dropped by the
// caller).  Exact.
__device__ __forceinline__ uint32_t absmax_bf16x2(uint32_t m, uint32_t x) {
    uint32_t r;
    asm("max.xorsign.abs.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(m), "r"(x));
    return r;
}

// Magnitudes of the two halves of a packed bf16 max-abs, as floats.
__device__ __forceinline__ float absmax_lo(uint32_t m) { return __uint_as_float((m << 16) & 0x7fffffffu); }
__device__ __forceinline__ float absmax_hi(uint32_t m) { return __uint_as_float(m & 0x7fff0000u); }

// Programmatic dependent launch: a kernel launched with the
// programmatic-serialization attribute may start while the previous kernel of
// the stream still runs; grid_dependency_wait() returns once that kernel has
// completed and its writes are visible (at once when launched without the
// attribute).  allow_dependents() lets the next such kernel start.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void allow_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ------------------------------------------------------------ statistics
//
// Lane l owns 8 consecutive channels of the block's 256 (one 16-byte chunk per
// row) and the 8 warps of a block split the block's row slab (warp w takes
// rows w, w + 8, ...).  Each thread streams its rows through a kStatsRing-deep
// ring; the row loop is unrolled over the ring, so every slot address is a
// constant, and only a warp's last (< 2 kStatsRing) rows test whether a row or
// a refill exists.  Max-abs is kept as packed bf16 (one instruction per two
// channels and row).
//
// Precision of the power sums: every sum is kept in fp32 on the SM.  A thread
// sums (x - c)^p over groups of at most kGroup of its rows (level 1), adds the
// group sums into level-2 sums (at most kGroup groups: the launch keeps a
// thread's rows at or below kGroup^2), the block adds its 8 warps' sums, and
// only the block's total is widened to fp64 and added into the caller's fp64
// accumulators with atomics.  The error of every returned sum is at most
// (63 + 63 + 7 + 4) * 2^-24 < (2 kGroup + 12) * 2^-24 of sum |x - c|^p (the
// three fp32 summation levels, and the rounding of the terms (x - c)^p);
// widening fp32 to fp64 is exact.  FP64 arithmetic runs at a small fraction
// of the fp32 rate on this part, so none happens per element.
constexpr int kStatsWarps = 8;
constexpr int kStatsThreads = 32 * kStatsWarps;
constexpr int kGroup = 64;
constexpr int kStatsRing = 6;                             // rows in flight per thread
constexpr int kL2Pitch = 36;     // [q][lane] pitch: conflict-free both by lane and by channel
constexpr int kMaxRowsPerThread = kGroup * kGroup;
static_assert(kGroup >= 4 * kStatsRing, "a level-1 group absorbs the drain");

struct StatsRed {
    float lvl[kStatsWarps][32][kL2Pitch];  // per-thread sums [q = 8 p + e][lane]
    float mx[kStatsWarps][32][8];           // per-thread maxima [lane][e]
};
constexpr int kStatsRingBytes = kStatsRing * kStatsThreads * 16;
constexpr int kStatsSmem =
    kStatsRingBytes > (int)sizeof(StatsRed) ? kStatsRingBytes : (int)sizeof(StatsRed);

struct StatsAcc {
    float2 g[4][4];         // level 1 [p][channel pair]
    float2 l2[4][4];        // level 2
    uint32_t mx[4];         // packed bf16 max-abs
    float2 c[4];            // -shift
    int in_group;

    __device__ __forceinline__ void row(const uint4 v) {
        const uint32_t wd[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            mx[h] = absmax_bf16x2(mx[h], wd[h]);
            const float2 x = make_float2(__uint_as_float(wd[h] << 16), __uint_as_float(wd[h] & 0xffff0000u));
            const float2 d = add2(x, c[h]);
            const float2 d2 = mul2(d, d);
            g[0][h] = add2(g[0][h], d);
            g[1][h] = add2(g[1][h], d2);
            g[2][h] = fma2(d2, d, g[2][h]);
            g[3][h] = fma2(d2, d2, g[3][h]);
        }
    }
    __device__ __forceinline__ void fold() {
#pragma unroll
        for (int p = 0; p < 4; ++p)
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                l2[p][h] = add2(l2[p][h], g[p][h]);
                g[p][h] = make_float2(0.f, 0.f);
            }
        in_group = 0;
    }
};

__global__ void __launch_bounds__(kStatsThreads, 2)
stats_update_kernel(const uint4 *__restrict__ X8, int T, int K, const float *__restrict__ shift,
                    int rows_per_slab, double *__restrict__ sums, float *__restrict__ absmax) {
    extern __shared__ __align__(16) unsigned char stats_smem[];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int ko = K / 8;                                 // 8-channel groups per row
    const int oct = blockIdx.x * 32 + lane;
    const bool active = oct < ko;
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(T, r0 + rows_per_slab);
    // rows of this warp: r0 + w + 8 i, i < n
    const int n = r1 - r0 > w ? (r1 - r0 - w + kStatsWarps - 1) / kStatsWarps : 0;
    const size_t step = (size_t)kStatsWarps * ko;
    const uint4 *nxt = X8 + (size_t)(r0 + w) * ko + (active ? oct : 0);   // next row to fetch
    const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(stats_smem)) + threadIdx.x * 16;
    constexpr uint32_t kSlot = kStatsThreads * 16;

#pragma unroll
    for (int u = 0; u < kStatsRing; ++u) {
        if (u < n) ring_cp16(ring + u * kSlot, nxt, active);
        nxt += step;
        ring_commit();
    }

    StatsAcc acc;
#pragma unroll
    for (int h = 0; h < 4; ++h) {
        acc.c[h] = make_float2(0.f, 0.f);
        acc.mx[h] = 0u;
#pragma unroll
        for (int p = 0; p < 4; ++p) acc.g[p][h] = acc.l2[p][h] = make_float2(0.f, 0.f);
    }
    acc.in_group = 0;
    if (active && shift) {
        const float4 s0 = __ldg(reinterpret_cast<const float4 *>(shift) + 2 * oct);
        const float4 s1 = __ldg(reinterpret_cast<const float4 *>(shift) + 2 * oct + 1);
        acc.c[0] = make_float2(-s0.x, -s0.y);
        acc.c[1] = make_float2(-s0.z, -s0.w);
        acc.c[2] = make_float2(-s1.x, -s1.y);
        acc.c[3] = make_float2(-s1.z, -s1.w);
    }

    // steady state: every row's slot is refilled with the row kStatsRing on
    int i = 0;
    for (; i + 2 * kStatsRing <= n; i += kStatsRing) {
#pragma unroll
        for (int u = 0; u < kStatsRing; ++u) {
            ring_wait<kStatsRing>();
            acc.row(ring_lds(ring + u * kSlot));
            ring_cp16(ring + u * kSlot, nxt, active);
            nxt += step;
            ring_commit();
        }
        acc.in_group += kStatsRing;
        if (acc.in_group > kGroup - 2 * kStatsRing) acc.fold();
    }
    // drain: the last n - i < 2 kStatsRing rows (in_group <= kGroup -
    // 2 kStatsRing here, so they stay within one level-1 group)
#pragma unroll
    for (int u = 0; u < kStatsRing; ++u) {
        if (i + u < n) {
            ring_wait<kStatsRing>();
            acc.row(ring_lds(ring + u * kSlot));
            if (i + u + kStatsRing < n) ring_cp16(ring + u * kSlot, nxt, active);
            nxt += step;
            ring_commit();
        }
    }
#pragma unroll
    for (int u = 0; u < kStatsRing; ++u) {
        if (i + kStatsRing + u < n) {
            ring_wait<kStatsRing>();
            acc.row(ring_lds(ring + u * kSlot));
            ring_commit();
        }
    }
    ring_drain();
    __syncthreads();                                      // the ring becomes the reduction area
    StatsRed &sm = *reinterpret_cast<StatsRed *>(stats_smem);
#pragma unroll
    for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            const float2 s = add2(acc.l2[p][h], acc.g[p][h]);
            sm.lvl[w][8 * p + 2 * h][lane] = s.x;
            sm.lvl[w][8 * p + 2 * h + 1][lane] = s.y;
        }
    reinterpret_cast<float4 *>(&sm.mx[w][lane][0])[0] =
        make_float4(absmax_lo(acc.mx[0]), absmax_hi(acc.mx[0]), absmax_lo(acc.mx[1]), absmax_hi(acc.mx[1]));
    reinterpret_cast<float4 *>(&sm.mx[w][lane][0])[1] =
        make_float4(absmax_lo(acc.mx[2]), absmax_hi(acc.mx[2]), absmax_lo(acc.mx[3]), absmax_hi(acc.mx[3]));
    __syncthreads();

    // block totals: thread t combines channel t of the block (source lane t/8,
    // entry e = t%8) over the 8 warps, for the 4 moments, and the maxima
    const int t = threadIdx.x, sl = t >> 3, e = t & 7;
    if (blockIdx.x * 256 + t < K && r0 < r1) {
        float a = 0.f;
#pragma unroll
        for (int ww = 0; ww < kStatsWarps; ++ww) a = fmaxf(a, sm.mx[ww][sl][e]);
        const size_t j = (size_t)blockIdx.x * 256 + t;
        // non-negative floats order like their bit patterns
        atomicMax(reinterpret_cast<unsigned int *>(absmax) + j, __float_as_uint(a));
#pragma unroll
        for (int p = 0; p < 4; ++p) {
            float s = 0.f;
#pragma unroll
            for (int ww = 0; ww < kStatsWarps; ++ww) s += sm.lvl[ww][8 * p + e][sl];
            atomicAdd(sums + (size_t)p * K + j, (double)s);
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

// Finalize in two launches, with the work spread over the GPU (fp64 runs at a
// small fraction of the fp32 rate here, so one block doing all K channels
// takes far longer than the data movement):
//   stats_channels_kernel  one warp per 32 channels: per-channel mean, std
//                          and kurtosis into chan; and the warp's channels
//                          pooled about their own mean mu_b (count 32 n):
//                          M2_b = sum_j M2_j + n d_j^2,
//                          M3_b = sum_j M3_j + 3 d_j M2_j + n d_j^3,
//                          M4_b = sum_j M4_j + 4 d_j M3_j + 6 d_j^2 M2_j + n d_j^4
//                          (d_j = mean_j - mu_b), with sum_j S2_j + n d_j^2 and
//                          the max-abs.  These six fp64 numbers per warp are
//                          kept in the first 12 floats per warp of chan's
//                          max-abs plane, whose own values are written last.
//   stats_tensor_kernel    one warp: pools the warps' summaries the same way
//                          about the grand mean, writes tensor[4], then the
//                          max-abs plane entries that held the summaries.
constexpr int kFinWarpCh = 32;
constexpr int kFinSummary = 6;                 // doubles per warp

__device__ __forceinline__ double warp_sum_f64(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int fin_stash_floats(int K) {
    return kFinSummary * 2 * ((K + kFinWarpCh - 1) / kFinWarpCh);
}

__global__ void __launch_bounds__(32)
stats_channels_kernel(const double *__restrict__ sums, const float *__restrict__ absmax,
                      const float *__restrict__ shift, double n, int K, float *__restrict__ chan) {
    const int lane = threadIdx.x;
    const int j = blockIdx.x * kFinWarpCh + lane;
    const bool valid = j < K;
    const int kb = min(kFinWarpCh, K - (int)blockIdx.x * kFinWarpCh);
    Central c = {0.0, 0.0, 0.0, 0.0};
    double s2 = 0.0;
    float am = 0.0f;
    if (valid) {
        c = central(sums, shift, K, j, n);
        s2 = sums[(size_t)K + j];
        am = absmax[j];
        const double var = c.m2 / n;
        if (j >= fin_stash_floats(K)) chan[j] = am;
        chan[(size_t)K + j] = static_cast<float>(c.mean);
        chan[2 * (size_t)K + j] = static_cast<float>(sqrt(var));
        chan[3 * (size_t)K + j] = static_cast<float>(var > 0.0 ? (c.m4 / n) / (var * var) : 0.0);
    }
    const double mu_b = warp_sum_f64(valid ? c.mean : 0.0) / kb;
    const double d = valid ? c.mean - mu_b : 0.0;
    const double M2 = warp_sum_f64(valid ? c.m2 + n * d * d : 0.0);
    const double M3 = warp_sum_f64(valid ? c.m3 + 3.0 * d * c.m2 + n * d * d * d : 0.0);
    const double M4 = warp_sum_f64(valid ? c.m4 + 4.0 * d * c.m3 + 6.0 * d * d * c.m2 + n * d * d * d * d : 0.0);
    const double SS = warp_sum_f64(valid ? s2 + n * d * d : 0.0);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
    if (lane == 0) {
        double *st = reinterpret_cast<double *>(chan) + (size_t)kFinSummary * blockIdx.x;
        st[0] = mu_b;
        st[1] = M2;
        st[2] = M3;
        st[3] = M4;
        st[4] = SS;
        st[5] = am;
    }
}

__global__ void __launch_bounds__(32)
stats_tensor_kernel(const float *__restrict__ absmax, double n, int K, float *__restrict__ chan,
                    float *__restrict__ tensor) {
    const int lane = threadIdx.x;
    const int G = (K + kFinWarpCh - 1) / kFinWarpCh;
    const double *st = reinterpret_cast<const double *>(chan);
    // grand mean: the warps' means weighted by their channel counts
    double ms = 0.0;
    for (int b = lane; b < G; b += 32) ms += st[kFinSummary * b] * min(kFinWarpCh, K - b * kFinWarpCh);
    const double mu = warp_sum_f64(ms) / K;
    double t2 = 0.0, t4 = 0.0, ss = 0.0, am = 0.0;
    for (int b = lane; b < G; b += 32) {
        const double *s = st + kFinSummary * b;
        const double nb = n * min(kFinWarpCh, K - b * kFinWarpCh);
        const double d = s[0] - mu;
        t2 += s[1] + nb * d * d;
        t4 += s[3] + 4.0 * d * s[2] + 6.0 * d * d * s[1] + nb * d * d * d * d;
        ss += s[4] + nb * d * d;
        am = fmax(am, s[5]);
    }
    const double T2 = warp_sum_f64(t2), T4 = warp_sum_f64(t4), SS = warp_sum_f64(ss);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) am = fmax(am, __shfl_xor_sync(0xffffffffu, am, o));
    __syncwarp();                                         // every summary has been read
    if (lane == 0) {
        const double nt = n * K;
        const double var = (T2 > 1e-5 * SS) ? T2 / nt : 0.0;
        tensor[0] = static_cast<float>(am);
        tensor[1] = static_cast<float>(mu);
        tensor[2] = static_cast<float>(sqrt(var));
        tensor[3] = static_cast<float>(var > 0.0 ? (T4 / nt) / (var * var) : 0.0);
    }
    // the max-abs plane entries that held the summaries (R is a multiple of 4)
    const int R4 = min(K, fin_stash_floats(K)) / 4;
    for (int q = lane; q < R4; q += 32)
        reinterpret_cast<float4 *>(chan)[q] = reinterpret_cast<const float4 *>(absmax)[q];
}

// ------------------------------------------------- per-tensor quantization
//
// Lane l owns 8 consecutive columns of the block's 256 (one 16-byte chunk per
// row) and warp w takes rows w, w + 8, ... of the block's slab; rows stream
// through a kPtRing-deep ring per thread.  The three launches (zero the
// maximum, pass 1, pass 2) use programmatic dependent launch: pass 1 streams
// X while the zeroing kernel finishes and waits only before its atomic; pass 2
// starts its first copies and 1/lambda while pass 1 finishes and waits before
// it reads the maximum.  X itself was complete before the first of them ran.
constexpr int kQWarps = 8;
constexpr int kPtRing = 8;
constexpr int kPtSmem = kPtRing * 32 * kQWarps * 16;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ void load_recip(const float *lam, int col0, bool active, float (&r)[8]) {
#pragma unroll
    for (int e = 0; e < 8; ++e) r[e] = (lam != nullptr && active) ? __frcp_rn(__ldg(lam + col0 + e)) : 1.0f;
}

// Runs `one(slot address)` for each of a warp's n rows in order, streaming
// them through the thread's ring (rows step `step` chunks apart, the first at
// `nxt`; the ring's first kPtRing copies are already issued).
template <typename F>
__device__ __forceinline__ void pt_stream(int n, const uint4 *nxt, size_t step, uint32_t ring,
                                          bool active, F &&one) {
    constexpr uint32_t kSlot = 32 * kQWarps * 16;
    nxt += kPtRing * step;
    int i = 0;
    for (; i + 2 * kPtRing <= n; i += kPtRing) {
#pragma unroll
        for (int u = 0; u < kPtRing; ++u) {
            ring_wait<kPtRing>();
            one(ring + u * kSlot);
            ring_cp16(ring + u * kSlot, nxt, active);
            nxt += step;
            ring_commit();
        }
    }
#pragma unroll
    for (int u = 0; u < kPtRing; ++u) {
        if (i + u < n) {
            ring_wait<kPtRing>();
            one(ring + u * kSlot);
            if (i + u + kPtRing < n) ring_cp16(ring + u * kSlot, nxt, active);
            nxt += step;
            ring_commit();
        }
    }
#pragma unroll
    for (int u = 0; u < kPtRing; ++u) {
        if (i + kPtRing + u < n) {
            ring_wait<kPtRing>();
            one(ring + u * kSlot);
            ring_commit();
        }
    }
    ring_drain();
}

__device__ __forceinline__ void pt_prologue(int n, const uint4 *nxt, size_t step, uint32_t ring, bool active) {
    constexpr uint32_t kSlot = 32 * kQWarps * 16;
#pragma unroll
    for (int u = 0; u < kPtRing; ++u) {
        if (u < n) ring_cp16(ring + u * kSlot, nxt, active);
        nxt += step;
        ring_commit();
    }
}

__global__ void zero_max_kernel(float *amax) {
    allow_dependents();
    *amax = 0.0f;
}

// Pass 1: max over the whole tensor of |x_mj / lambda_j| = |x_mj * r_j| with
// r_j = rn(1 / lambda_j).  Rounding is monotone, so for each column
// max_m fl(|x_mj| * r_j) = fl(r_j * max_m |x_mj|): a lane keeps the packed
// bf16 max-abs of its 8 columns over its rows and multiplies by r_j once.
__global__ void __launch_bounds__(32 * kQWarps)
tensor_absmax_kernel(const uint16_t *__restrict__ X, const float *__restrict__ lam, int M, int K,
                     int rows_per_slab, float *__restrict__ amax) {
    extern __shared__ __align__(16) unsigned char pt_smem[];
    __shared__ float red[kQWarps];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int ko = K / 8;
    const int oct = blockIdx.x * 32 + lane;
    const bool active = oct < ko;
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(M, r0 + rows_per_slab);
    const int n = r1 - r0 > w ? (r1 - r0 - w + kQWarps - 1) / kQWarps : 0;
    const size_t step = (size_t)kQWarps * ko;
    const uint4 *first = reinterpret_cast<const uint4 *>(X) + (size_t)(r0 + w) * ko + (active ? oct : 0);
    const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(pt_smem)) + threadIdx.x * 16;
    pt_prologue(n, first, step, ring, active);
    allow_dependents();
    uint32_t m[4] = {0u, 0u, 0u, 0u};
    pt_stream(n, first, step, ring, active, [&](uint32_t slot) {
        const uint4 v = ring_lds(slot);
        m[0] = absmax_bf16x2(m[0], v.x);
        m[1] = absmax_bf16x2(m[1], v.y);
        m[2] = absmax_bf16x2(m[2], v.z);
        m[3] = absmax_bf16x2(m[3], v.w);
    });
    float a = 0.0f;
    if (active) {
        float r[8];
        load_recip(lam, oct * 8, true, r);
#pragma unroll
        for (int h = 0; h < 4; ++h) {
            a = fmaxf(a, __fmul_rn(absmax_lo(m[h]), r[2 * h]));
            a = fmaxf(a, __fmul_rn(absmax_hi(m[h]), r[2 * h + 1]));
        }
    }
    a = warp_max(a);
    if (lane == 0) red[w] = a;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.0f;
        for (int k = 0; k < kQWarps; ++k) t = fmaxf(t, red[k]);
        grid_dependency_wait();                  // the zeroing kernel has completed
        // non-negative floats order like their bit patterns
        atomicMax(reinterpret_cast<unsigned int *>(amax), __float_as_uint(t));
    }
}

constexpr float kRoundMagic = 12582912.0f;   // 1.5 * 2^23: low byte of the sum = rne(y)

__device__ __forceinline__ uint32_t pack4_low_bytes(float a, float b, float c, float d) {
    const uint32_t ab = __byte_perm(__float_as_uint(a), __float_as_uint(b), 0x0040);
    const uint32_t cd = __byte_perm(__float_as_uint(c), __float_as_uint(d), 0x0040);
    return __byte_perm(ab, cd, 0x5410);
}

// The 8 codes of one lane's chunk: q = rne(fl(x * r) * inv), clamped.
template <bool FAST>
__device__ __forceinline__ uint2 quant8(const uint4 v, const float (&r)[8], float inv) {
    const uint32_t wd[4] = {v.x, v.y, v.z, v.w};
    float xs[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        xs[2 * e] = __fmul_rn(__uint_as_float(wd[e] << 16), r[2 * e]);
        xs[2 * e + 1] = __fmul_rn(__uint_as_float(wd[e] & 0xffff0000u), r[2 * e + 1]);
    }
    uint32_t word[2] = {0u, 0u};
    if (FAST) {
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
    return make_uint2(word[0], word[1]);
}

template <bool FAST>
__device__ __forceinline__ void quant_rows(int n, const uint4 *first, size_t step, uint32_t ring,
                                           bool active, const float (&r)[8], float inv, float scale,
                                           bool zero, uint2 *dst, size_t dstep, float *xs_out,
                                           bool write_scale) {
    pt_stream(n, first, step, ring, active, [&](uint32_t slot) {
        const uint4 v = ring_lds(slot);
        if (write_scale) *xs_out = scale;
        if (active) *dst = zero ? make_uint2(0u, 0u) : quant8<FAST>(v, r, inv);
        dst += dstep;
        xs_out += kQWarps;
    });
}

// Pass 2: INT8 codes of x_mj / lambda_j with the one scale a / 127 (each lane
// writes its 8 codes of a row as one 8-byte store; block column 0 writes the
// row scales).
__global__ void __launch_bounds__(32 * kQWarps)
tensor_quant_kernel(const uint16_t *__restrict__ X, const float *__restrict__ lam, int M, int K,
                    int rows_per_slab, const float *__restrict__ amax, int8_t *__restrict__ Xq,
                    float *__restrict__ x_scale) {
    extern __shared__ __align__(16) unsigned char pt_smem[];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int ko = K / 8;
    const int oct = blockIdx.x * 32 + lane;
    const bool active = oct < ko;
    const int r0 = blockIdx.y * rows_per_slab;
    const int r1 = min(M, r0 + rows_per_slab);
    const int n = r1 - r0 > w ? (r1 - r0 - w + kQWarps - 1) / kQWarps : 0;
    const size_t step = (size_t)kQWarps * ko;
    const uint4 *first = reinterpret_cast<const uint4 *>(X) + (size_t)(r0 + w) * ko + (active ? oct : 0);
    const uint32_t ring = static_cast<uint32_t>(__cvta_generic_to_shared(pt_smem)) + threadIdx.x * 16;
    pt_prologue(n, first, step, ring, active);
    float r[8];
    load_recip(lam, oct * 8, active, r);
    grid_dependency_wait();                      // pass 1 has completed: the maximum is final
    const float a = *amax;
    const bool zero = (a == 0.0f);
    const float inv = zero ? 0.0f : __fdiv_rn(127.0f, a);
    const float scale = zero ? 0.0f : __fdiv_rn(a, 127.0f);
    // a and 127/a finite: |x' * inv| <= 127 (1 + 2^-23), no clamp needed
    const bool fast = (a <= 3.402823466e38f) && (inv <= 3.402823466e38f);
    uint2 *dst = reinterpret_cast<uint2 *>(Xq + (size_t)(r0 + w) * K) + (active ? oct : 0);
    const size_t dstep = (size_t)kQWarps * ko;   // 8-byte units between a warp's rows
    float *xs_out = x_scale + r0 + w;
    const bool write_scale = blockIdx.x == 0 && lane == 0;
    if (fast)
        quant_rows<true>(n, first, step, ring, active, r, inv, scale, zero, dst, dstep, xs_out, write_scale);
    else
        quant_rows<false>(n, first, step, ring, active, r, inv, scale, zero, dst, dstep, xs_out, write_scale);
}

// Zeroes n 4-byte words (the one-shot statistics' accumulators).
__global__ void zero_words_kernel(uint32_t *p, size_t n) {
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
        p[i] = 0u;
}

// Sets the dynamic shared memory of `kern` and looks up its resident blocks
// per SM with that much, once per device.
template <typename Kern>
cudaError_t kernel_setup(PerDevice<int> &cache, Kern kern, int threads, int smem, int *per_sm) {
    return cache.get([&](int &n) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, smem);
        if (n < 1) n = 1;
        return e;
    }, per_sm);
}

// Row slabs so that a (gx x gy) grid fills the GPU once: gy = the resident
// blocks on all SMs divided by gx, at most one slab per row.
int slabs_for(int per_sm, int rows, int gx) {
    int gy = (num_sms() * per_sm) / gx;
    if (gy > rows) gy = rows;
    if (gy < 1) gy = 1;
    return gy;
}


// One-shot statistics without caller accumulators: a file-scope scratch that
// holds, for a call with K channels, the power sums (4 x K doubles) followed
// by the max-abs (K floats), cleared at the start of every call.  Calls that
// overlap in time share it.
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
    static PerDevice<int> occ;
    int per_sm = 1;
    cudaError_t e = kernel_setup(occ, stats_update_kernel, kStatsThreads, kStatsSmem, &per_sm);
    if (e != cudaSuccess) return e;
    const int gx = (K / 8 + 31) / 32;
    int gy = slabs_for(per_sm, T, gx);
    // at least 8 rows per warp; at most kGroup^2 rows per thread
    int rows_per_slab = (T + gy - 1) / gy;
    if (rows_per_slab < 8 * kStatsWarps) rows_per_slab = 8 * kStatsWarps;
    if (rows_per_slab > kStatsWarps * kMaxRowsPerThread) rows_per_slab = kStatsWarps * kMaxRowsPerThread;
    // at most 65535 slabs per launch (a grid's y extent)
    const long long rows_per_launch = 65535LL * rows_per_slab;
    for (long long t0 = 0; t0 < T; t0 += rows_per_launch) {
        const int rows = static_cast<int>(T - t0 < rows_per_launch ? T - t0 : rows_per_launch);
        stats_update_kernel<<<dim3(gx, (rows + rows_per_slab - 1) / rows_per_slab), kStatsThreads,
                              kStatsSmem, st>>>(reinterpret_cast<const uint4 *>(X + t0 * K), rows, K,
                                                shift, rows_per_slab, sums, absmax);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_act_stats_finalize(const double *sums, const float *absmax, const float *shift,
                                      long long count, int K, float *chan, float *tensor,
                                      cudaStream_t st) {
    stats_channels_kernel<<<(K + kFinWarpCh - 1) / kFinWarpCh, 32, 0, st>>>(sums, absmax, shift,
                                                                           (double)count, K, chan);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    stats_tensor_kernel<<<1, 32, 0, st>>>(absmax, (double)count, K, chan, tensor);
    return cudaGetLastError();
}

cudaError_t launch_quant_act_per_tensor(const uint16_t *X, const float *lambda, int M, int K,
                                        int8_t *Xq, float *x_scale, float *amax, cudaStream_t st) {
    static PerDevice<int> occ1, occ2;
    int per1 = 1, per2 = 1;
    cudaError_t e = kernel_setup(occ1, tensor_absmax_kernel, 32 * kQWarps, kPtSmem, &per1);
    if (e != cudaSuccess) return e;
    e = kernel_setup(occ2, tensor_quant_kernel, 32 * kQWarps, kPtSmem, &per2);
    if (e != cudaSuccess) return e;
    zero_max_kernel<<<1, 1, 0, st>>>(amax);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // pass 1 at two blocks per SM: pass 2's blocks start beside them
    const int gx = (K / 8 + 31) / 32;
    const int gy1 = slabs_for(per1 < 2 ? per1 : 2, M, gx);
    const int gy2 = slabs_for(per2 < 2 ? per2 : 2, M, gx);
    const int rps1 = (M + gy1 - 1) / gy1, rps2 = (M + gy2 - 1) / gy2;
    e = launch_pdl(tensor_absmax_kernel, dim3(gx, (M + rps1 - 1) / rps1), 32 * kQWarps, kPtSmem, st,
                   X, lambda, M, K, rps1, amax);
    if (e != cudaSuccess) return e;
    return launch_pdl(tensor_quant_kernel, dim3(gx, (M + rps2 - 1) / rps2), 32 * kQWarps, kPtSmem, st,
                      X, lambda, M, K, rps2, static_cast<const float *>(amax), Xq, x_scale);
}

cudaError_t launch_act_stats_noalloc(const uint16_t *X, int T, int K, const float *shift, float *chan,
                                     float *tensor, cudaStream_t st) {
    void *base = stats_scratch_address();
    if (!base) return cudaErrorInvalidSymbol;
    double *sums = static_cast<double *>(base);
    float *absmax = reinterpret_cast<float *>(sums + 4 * static_cast<size_t>(K));
    const size_t words = 9 * static_cast<size_t>(K);      // 4K doubles and K floats
    zero_words_kernel<<<(unsigned)((words + 1023) / 1024 < 256 ? (words + 1023) / 1024 : 256), 1024, 0, st>>>(
        static_cast<uint32_t *>(base), words);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    e = launch_act_stats_update(X, T, K, shift, sums, absmax, st);
    if (e != cudaSuccess) return e;
    return launch_act_stats_finalize(sums, absmax, shift, T, K, chan, tensor, st);
}

}  // namespace w8a8
