// api.cu -- the C ABI (include/w8a8.h): argument checks, then stream-ordered
// launches.  No allocation, no synchronisation (except w8a8_device_status).
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <numeric>
#include <vector>
#include <cuda_runtime.h>

#include "../../include/w8a8.h"
#include "host_once.h"
#include "launch.h"

namespace {

// The library's single device-side error word: kernels with bounded waits
// record a nonzero code here instead of spinning forever.
__device__ unsigned int g_w8a8_device_error = 0;

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Whether byte ranges [a, a + na) and [b, b + nb) overlap.
bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return x < y + nb && y < x + na;
}

w8a8_status check_mk(int M, int K) {
    if (M < 0 || K <= 0 || (K % 16) != 0 || K > W8A8_MAX_K) return W8A8_ERR_UNSUPPORTED_SHAPE;
    return W8A8_OK;
}

w8a8_status check_nk(int N, int K) {
    if (N <= 0 || (N % 8) != 0 || K <= 0 || (K % 16) != 0 || K > W8A8_MAX_K)
        return W8A8_ERR_UNSUPPORTED_SHAPE;
    return W8A8_OK;
}

w8a8_status from_cuda(cudaError_t e) { return e == cudaSuccess ? W8A8_OK : W8A8_ERR_CUDA; }

cudaStream_t as_stream(void *s) { return static_cast<cudaStream_t>(s); }

// Address of the error word on the current device, looked up once per device
// (under std::call_once: host threads may launch concurrently).
unsigned int *device_error_word() {
    static w8a8::PerDevice<unsigned int *> addr;
    unsigned int *p = nullptr;
    if (addr.get([](unsigned int *&v) {
            void *q = nullptr;
            cudaError_t e = cudaGetSymbolAddress(&q, g_w8a8_device_error);
            v = static_cast<unsigned int *>(q);
            return e;
        }, &p) != cudaSuccess)
        return nullptr;
    return p;
}

// Validation shared by the single- and dual-branch linears.
w8a8_status check_branch(const w8a8::GemmBranch &b, bool need_scales, int N, int K) {
    if (b.M < 0) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (b.M == 0) return W8A8_OK;
    if (!b.Xq || !b.Wq || !b.out) return W8A8_ERR_INVALID_ARG;
    if (need_scales && (!b.x_scale || !b.w_scale)) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(b.Xq) || !aligned16(b.Wq) || !aligned16(b.out)) return W8A8_ERR_MISALIGNED;
    if (need_scales && (!aligned16(b.x_scale) || !aligned16(b.w_scale) ||
                        (b.bias && !aligned16(b.bias))))
        return W8A8_ERR_MISALIGNED;
    (void)N;
    (void)K;
    return W8A8_OK;
}

// a4 + a5 on int8 codes: the tcgen05 GEMM on CTA pairs (both operands
// converted to fp16 in shared memory, two accumulators in tensor memory).
w8a8_status run_gemm(const w8a8::GemmBranch *br, int nb, int N, int K, bool out_i32,
                     cudaStream_t st) {
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_gemm_tc2(br, nb, N, K, out_i32, false, err, st));
}

// The same with a workspace: the codes expanded to fp16 values (with token
// sums) by a streaming pass, then the GEMM with the weights in tensor memory.
w8a8_status run_gemm_ws(const w8a8::GemmBranch *br, int nb, int N, int K, bool out_i32, void *workspace,
                        cudaStream_t st) {
    if (!workspace) return run_gemm(br, nb, N, K, out_i32, st);
    if (!aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    for (int i = 0; i < nb; ++i)
        if (br[i].M > 0 && br[i].plan && !aligned16(br[i].plan)) return W8A8_ERR_MISALIGNED;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_linear_codes8(br, nb, N, K, out_i32, workspace, err, st));
}

// The same product on the earlier engines, kept as test anchors and never on
// a product call: 1 = tcgen05 on single SMs, 0 = mma.sync s8; 2 is the
// product engine.
w8a8_status run_gemm_engine(int engine, const w8a8::GemmBranch *br, int nb, int N, int K, bool out_i32,
                            cudaStream_t st) {
    if (engine == 2) return run_gemm(br, nb, N, K, out_i32, st);
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    if (engine == 1) return from_cuda(w8a8::launch_gemm_tc(br, nb, N, K, out_i32, err, st));
    return from_cuda(w8a8::launch_gemm_mma(br, nb, N, K, out_i32, st));
}

}  // namespace

extern "C" {

const char *w8a8_status_string(w8a8_status status) {
    switch (status) {
        case W8A8_OK: return "W8A8_OK";
        case W8A8_ERR_INVALID_ARG: return "W8A8_ERR_INVALID_ARG";
        case W8A8_ERR_UNSUPPORTED_SHAPE: return "W8A8_ERR_UNSUPPORTED_SHAPE";
        case W8A8_ERR_MISALIGNED: return "W8A8_ERR_MISALIGNED";
        case W8A8_ERR_CUDA: return "W8A8_ERR_CUDA";
        case W8A8_ERR_TIMEOUT: return "W8A8_ERR_TIMEOUT";
    }
    return "W8A8_ERR_UNKNOWN";
}

w8a8_status w8a8_channel_absmax(const uint16_t *X, int T, int K, float *s, void *stream) {
    if (T < 0 || K <= 0 || (K % 16) != 0 || K > W8A8_MAX_K) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (!s || (T > 0 && !X)) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(s) || (T > 0 && !aligned16(X))) return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_channel_absmax(X, T, K, s, as_stream(stream)));
}

w8a8_status w8a8_smooth_scales(const float *act_absmax, const float *W, int N, int K,
                               float alpha, float *smooth, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (!act_absmax || !W || !smooth) return W8A8_ERR_INVALID_ARG;
    if (!(alpha >= 0.0f && alpha <= 1.0f)) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(act_absmax) || !aligned16(W) || !aligned16(smooth)) return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_smooth_scales(act_absmax, W, N, K, alpha, smooth,
                                                as_stream(stream)));
}

w8a8_status w8a8_quantize_weights(const float *W, const float *smooth, int N, int K,
                                  int8_t *Wq, float *w_scale, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (!W || !Wq || !w_scale) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(W) || !aligned16(Wq) || !aligned16(w_scale) || (smooth && !aligned16(smooth)))
        return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_quantize_weights(W, smooth, N, K, Wq, w_scale,
                                                   as_stream(stream)));
}

w8a8_status w8a8_quant_act(const uint16_t *X, const float *smooth, int M, int K,
                           int8_t *Xq, float *x_scale, void *stream) {
    if (w8a8_status e = check_mk(M, K)) return e;
    if (M == 0) return W8A8_OK;
    if (!X || !Xq || !x_scale) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(Xq) || !aligned16(x_scale) || (smooth && !aligned16(smooth)))
        return W8A8_ERR_MISALIGNED;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_quant_act(X, smooth, M, K, Xq, x_scale, err, as_stream(stream)));
}

w8a8_status w8a8_linear(const int8_t *Xq, const float *x_scale, const int8_t *Wq,
                        const float *w_scale, const float *bias, int M, int N, int K,
                        uint16_t *Y, const uint32_t *chunk_plan, void *workspace, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (w8a8_status e = check_mk(M, K)) return e;
    w8a8::GemmBranch b{Xq, x_scale, Wq, w_scale, bias, Y, M, nullptr, chunk_plan};
    if (w8a8_status e = check_branch(b, true, N, K)) return e;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    if (M == 0) return W8A8_OK;
    return run_gemm_ws(&b, 1, N, K, false, workspace, as_stream(stream));
}

long long w8a8_linear_workspace_size(long long tokens, int K) {
    return w8a8::linear_codes8_workspace_bytes(tokens, K);
}

w8a8_status w8a8_linear_dual(const w8a8_branch *br, int N, int K, void *workspace, void *stream) {
    if (!br) return W8A8_ERR_INVALID_ARG;
    if (w8a8_status e = check_nk(N, K)) return e;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    w8a8::GemmBranch b[2];
    for (int i = 0; i < 2; ++i) {
        b[i] = w8a8::GemmBranch{br[i].Xq, br[i].x_scale, br[i].Wq, br[i].w_scale,
                                br[i].bias, br[i].Y, br[i].M, nullptr, br[i].chunk_plan};
        if (w8a8_status e = check_mk(br[i].M, K)) return e;
        if (w8a8_status e = check_branch(b[i], true, N, K)) return e;
    }
    if (b[0].M == 0 && b[1].M == 0) return W8A8_OK;
    return run_gemm_ws(b, 2, N, K, false, workspace, as_stream(stream));
}

w8a8_status w8a8_debug_gemm_i32(const int8_t *Xq, const int8_t *Wq, int M, int N, int K,
                                int32_t *acc, const uint32_t *chunk_plan, void *workspace, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (w8a8_status e = check_mk(M, K)) return e;
    w8a8::GemmBranch b{Xq, nullptr, Wq, nullptr, nullptr, acc, M, nullptr, chunk_plan};
    if (w8a8_status e = check_branch(b, false, N, K)) return e;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    if (M == 0) return W8A8_OK;
    return run_gemm_ws(&b, 1, N, K, true, workspace, as_stream(stream));
}

w8a8_status w8a8_debug_linear_engine(int engine, const w8a8_branch *br, int nb, int N, int K, int out_i32,
                                     void *stream) {
    if (engine < 0 || engine > 2 || !br || nb < 1 || nb > 2) return W8A8_ERR_INVALID_ARG;
    if (w8a8_status e = check_nk(N, K)) return e;
    w8a8::GemmBranch b[2];
    for (int i = 0; i < nb; ++i) {
        b[i] = w8a8::GemmBranch{br[i].Xq, br[i].x_scale, br[i].Wq, br[i].w_scale, br[i].bias, br[i].Y, br[i].M,
                                nullptr, nullptr};
        if (w8a8_status e = check_mk(br[i].M, K)) return e;
        if (w8a8_status e = check_branch(b[i], out_i32 == 0, N, K)) return e;
    }
    if (b[0].M == 0 && (nb == 1 || b[1].M == 0)) return W8A8_OK;
    return run_gemm_engine(engine, b, nb, N, K, out_i32 != 0, as_stream(stream));
}

w8a8_status w8a8_quant_act_dual(const w8a8_act_branch *br, int K, void *stream) {
    if (!br) return W8A8_ERR_INVALID_ARG;
    w8a8::QuantActBranch b[2];
    for (int i = 0; i < 2; ++i) {
        if (w8a8_status e = check_mk(br[i].M, K)) return e;
        b[i] = w8a8::QuantActBranch{br[i].X, br[i].smooth, br[i].M, br[i].Xq, br[i].x_scale};
        if (br[i].M == 0) continue;
        if (!br[i].X || !br[i].Xq || !br[i].x_scale) return W8A8_ERR_INVALID_ARG;
        if (!aligned16(br[i].X) || !aligned16(br[i].Xq) || !aligned16(br[i].x_scale) ||
            (br[i].smooth && !aligned16(br[i].smooth)))
            return W8A8_ERR_MISALIGNED;
    }
    if (br[0].M == 0 && br[1].M == 0) return W8A8_OK;
    return from_cuda(w8a8::launch_quant_act_dual(b, K, as_stream(stream)));
}

w8a8_status w8a8_quant_act_dual_f16codes(const w8a8_act_branch16 *br, int K, void *stream) {
    if (!br) return W8A8_ERR_INVALID_ARG;
    if (K > 16384) return W8A8_ERR_UNSUPPORTED_SHAPE;
    w8a8::QuantActBranch16 b[2];
    for (int i = 0; i < 2; ++i) {
        if (w8a8_status e = check_mk(br[i].M, K)) return e;
        b[i] = w8a8::QuantActBranch16{br[i].X, br[i].smooth, br[i].M, br[i].Xq16, br[i].x_scale, br[i].x_sumsq};
        if (br[i].M == 0) continue;
        if (!br[i].X || !br[i].Xq16 || !br[i].x_scale) return W8A8_ERR_INVALID_ARG;
        if (!aligned16(br[i].X) || !aligned16(br[i].Xq16) || !aligned16(br[i].x_scale) ||
            (br[i].smooth && !aligned16(br[i].smooth)) || (br[i].x_sumsq && !aligned16(br[i].x_sumsq)))
            return W8A8_ERR_MISALIGNED;
    }
    if (br[0].M == 0 && br[1].M == 0) return W8A8_OK;
    return from_cuda(w8a8::launch_quant_act_dual_f16codes(b, K, as_stream(stream)));
}

w8a8_status w8a8_linear_dual_f16codes(const w8a8_branch16 *br, int N, int K, void *workspace,
                                      void *stream) {
    if (!br) return W8A8_ERR_INVALID_ARG;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    if (w8a8_status e = check_nk(N, K)) return e;
    w8a8::GemmBranch b[2];
    for (int i = 0; i < 2; ++i) {
        b[i] = w8a8::GemmBranch{reinterpret_cast<const int8_t *>(br[i].Xq16), br[i].x_scale, br[i].Wq,
                                br[i].w_scale, br[i].bias, br[i].Y, br[i].M, br[i].x_sumsq, br[i].chunk_plan};
        if (w8a8_status e = check_mk(br[i].M, K)) return e;
        if (w8a8_status e = check_branch(b[i], true, N, K)) return e;
        if (br[i].M > 0 && ((br[i].chunk_plan && !aligned16(br[i].chunk_plan)) ||
                            (br[i].x_sumsq && !aligned16(br[i].x_sumsq))))
            return W8A8_ERR_MISALIGNED;
    }
    if (b[0].M == 0 && b[1].M == 0) return W8A8_OK;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_gemm_ts(b, 2, N, K, false, workspace, err, as_stream(stream)));
}

w8a8_status w8a8_gelu_quant_act(const uint16_t *H, const float *smooth, int M, int K, int8_t *Xq,
                                float *x_scale, void *stream) {
    if (w8a8_status e = check_mk(M, K)) return e;
    if (M == 0) return W8A8_OK;
    if (!H || !Xq || !x_scale) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(H) || !aligned16(Xq) || !aligned16(x_scale) || (smooth && !aligned16(smooth)))
        return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_gelu_quant_act(H, smooth, M, K, Xq, x_scale, as_stream(stream)));
}

w8a8_status w8a8_debug_gelu(const uint16_t *H, int n, float *G, void *stream) {
    if (n < 0) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (n == 0) return W8A8_OK;
    if (!H || !G) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(H) || !aligned16(G)) return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_debug_gelu(H, n, G, as_stream(stream)));
}

w8a8_status w8a8_quant_act_f16codes(const uint16_t *X, const float *smooth, int M, int K,
                                    uint16_t *Xq16, float *x_scale, uint32_t *x_sumsq, int gelu,
                                    void *stream) {
    if (w8a8_status e = check_mk(M, K)) return e;
    if (K > 16384) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (M == 0) return W8A8_OK;
    if (!X || !Xq16 || !x_scale) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(Xq16) || !aligned16(x_scale) || (smooth && !aligned16(smooth)) ||
        (x_sumsq && !aligned16(x_sumsq)))
        return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_quant_act_f16codes(X, smooth, M, K, Xq16, x_scale, x_sumsq, gelu != 0,
                                                     as_stream(stream)));
}

w8a8_status w8a8_linear_f16codes(const uint16_t *Xq16, const float *x_scale, const int8_t *Wq,
                                 const float *w_scale, const float *bias, int M, int N, int K,
                                 const uint32_t *chunk_plan, const uint32_t *x_sumsq, uint16_t *Y,
                                 void *workspace, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    if (w8a8_status e = check_mk(M, K)) return e;
    w8a8::GemmBranch b{reinterpret_cast<const int8_t *>(Xq16), x_scale, Wq, w_scale, bias, Y, M, x_sumsq,
                       chunk_plan};
    if (w8a8_status e = check_branch(b, true, N, K)) return e;
    if ((chunk_plan && !aligned16(chunk_plan)) || (x_sumsq && !aligned16(x_sumsq))) return W8A8_ERR_MISALIGNED;
    if (M == 0) return W8A8_OK;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_gemm_ts(&b, 1, N, K, false, workspace, err, as_stream(stream)));
}

w8a8_status w8a8_debug_gemm_f16codes_i32(const uint16_t *Xq16, const int8_t *Wq, int M, int N, int K,
                                         const uint32_t *chunk_plan, const uint32_t *x_sumsq, int32_t *acc,
                                         void *workspace, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    if (w8a8_status e = check_mk(M, K)) return e;
    w8a8::GemmBranch b{reinterpret_cast<const int8_t *>(Xq16), nullptr, Wq, nullptr, nullptr, acc, M, x_sumsq,
                       chunk_plan};
    if (w8a8_status e = check_branch(b, false, N, K)) return e;
    if ((chunk_plan && !aligned16(chunk_plan)) || (x_sumsq && !aligned16(x_sumsq))) return W8A8_ERR_MISALIGNED;
    if (M == 0) return W8A8_OK;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_gemm_ts(&b, 1, N, K, true, workspace, err, as_stream(stream)));
}

long long w8a8_gemm_workspace_size(void) { return w8a8::gemm_ts_workspace_bytes(); }

long long w8a8_chunk_plan_size(int N, int K) {
    if (N <= 0 || K <= 0) return 1;
    return static_cast<long long>((N + 255) / 256) * w8a8::chunk_plan_words(K);
}

w8a8_status w8a8_chunk_plan(const int8_t *Wq, int N, int K, uint32_t *plan, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (!Wq || !plan) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(Wq) || !aligned16(plan)) return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_chunk_plan(Wq, N, K, plan, as_stream(stream)));
}

w8a8_status w8a8_quant_act_per_tensor(const uint16_t *X, const float *smooth, int M, int K,
                                      int8_t *Xq, float *x_scale, float *amax, void *stream) {
    if (w8a8_status e = check_mk(M, K)) return e;
    if (M == 0) return W8A8_OK;
    if (!X || !Xq || !x_scale || !amax) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(Xq) || !aligned16(x_scale) || !aligned16(amax) ||
        (smooth && !aligned16(smooth)))
        return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_quant_act_per_tensor(X, smooth, M, K, Xq, x_scale, amax,
                                                       as_stream(stream)));
}

w8a8_status w8a8_act_stats_update(const uint16_t *X, int T, int K, const float *shift,
                                  double *sums, float *absmax, void *stream) {
    if (w8a8_status e = check_mk(T, K)) return e;
    if (!sums || !absmax) return W8A8_ERR_INVALID_ARG;
    if (T == 0) return W8A8_OK;
    if (!X) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(sums) || !aligned16(absmax) || (shift && !aligned16(shift)))
        return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_act_stats_update(X, T, K, shift, sums, absmax,
                                                   as_stream(stream)));
}

w8a8_status w8a8_act_stats_finalize(const double *sums, const float *absmax, const float *shift,
                                    long long count, int K, float *chan, float *tensor,
                                    void *stream) {
    if (K <= 0 || (K % 16) != 0 || K > W8A8_MAX_K) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (count <= 0 || !sums || !absmax || !chan || !tensor) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(sums) || !aligned16(absmax) || !aligned16(chan) || !aligned16(tensor) ||
        (shift && !aligned16(shift)))
        return W8A8_ERR_MISALIGNED;
    const size_t k = static_cast<size_t>(K);
    if (overlaps(chan, 4 * k * sizeof(float), sums, 4 * k * sizeof(double)) ||
        overlaps(chan, 4 * k * sizeof(float), absmax, k * sizeof(float)) ||
        (shift && overlaps(chan, 4 * k * sizeof(float), shift, k * sizeof(float))))
        return W8A8_ERR_INVALID_ARG;
    return from_cuda(w8a8::launch_act_stats_finalize(sums, absmax, shift, count, K, chan, tensor,
                                                     as_stream(stream)));
}

w8a8_status w8a8_act_stats_noalloc(const uint16_t *X, int T, int K, const float *shift, float *chan,
                                   float *tensor, void *stream) {
    if (K <= 0 || (K % 16) != 0 || K > W8A8_NOALLOC_STATS_MAX_K) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (T <= 0 || !X || !chan || !tensor) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(chan) || !aligned16(tensor) || (shift && !aligned16(shift)))
        return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_act_stats_noalloc(X, T, K, shift, chan, tensor, as_stream(stream)));
}

w8a8_status w8a8_linear_bf16(const uint16_t *X, const uint16_t *W, const float *bias, int M,
                             int N, int K, uint16_t *Y, void *stream) {
    if (w8a8_status e = check_nk(N, K)) return e;
    if (w8a8_status e = check_mk(M, K)) return e;
    if (M == 0) return W8A8_OK;
    if (!X || !W || !Y) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(W) || !aligned16(Y) || (bias && !aligned16(bias)))
        return W8A8_ERR_MISALIGNED;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_gemm_bf16(X, W, bias, M, N, K, Y, err, as_stream(stream)));
}

static w8a8_status check_gguf(const void *Wraw, int fmt, int N, int K) {
    if (fmt != W8A8_GGUF_Q8_0 && fmt != W8A8_GGUF_Q4_K) return W8A8_ERR_INVALID_ARG;
    if (N <= 0 || (N % 8) != 0 || K <= 0 || (K % 256) != 0) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (!Wraw) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(Wraw)) return W8A8_ERR_MISALIGNED;
    return W8A8_OK;
}

w8a8_status w8a8_linear_gguf(const uint16_t *X, const uint8_t *Wraw, int fmt, const float *bias,
                             int M, int N, int K, uint16_t *Y, void *stream) {
    if (w8a8_status e = check_gguf(Wraw, fmt, N, K)) return e;
    if (M < 0) return W8A8_ERR_UNSUPPORTED_SHAPE;
    if (M == 0) return W8A8_OK;
    if (!X || !Y) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(Y) || (bias && !aligned16(bias))) return W8A8_ERR_MISALIGNED;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_gemm_gguf(X, Wraw, fmt, bias, M, N, K, Y, err, as_stream(stream)));
}

w8a8_status w8a8_debug_gguf_dequant(const uint8_t *Wraw, int fmt, int N, int K, uint16_t *W,
                                    void *stream) {
    if (w8a8_status e = check_gguf(Wraw, fmt, N, K)) return e;
    if (!W) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(W)) return W8A8_ERR_MISALIGNED;
    return from_cuda(w8a8::launch_gguf_dequant(Wraw, fmt, N, K, W, as_stream(stream)));
}

w8a8_status w8a8_layer_forward(const w8a8_layer *layer, const uint16_t *X, int M, int8_t *Xq_work,
                               float *x_scale_work, uint16_t *Y, void *workspace, void *stream) {
    if (!layer) return W8A8_ERR_INVALID_ARG;
    const int N = layer->N, K = layer->K;
    if (w8a8_status e = check_nk(N, K)) return e;
    if (w8a8_status e = check_mk(M, K)) return e;
    if (layer->protect) {
        if (!layer->W_bf16) return W8A8_ERR_INVALID_ARG;
        return w8a8_linear_bf16(X, layer->W_bf16, layer->bias, M, N, K, Y, stream);
    }
    if (!layer->Wq || !layer->w_scale) return W8A8_ERR_INVALID_ARG;
    if (workspace && !aligned16(workspace)) return W8A8_ERR_MISALIGNED;
    if (M == 0) return W8A8_OK;
    const bool direct16 = workspace != nullptr && K <= 16384;   // a3 writes fp16 codes into the workspace
    if (!x_scale_work || (!direct16 && !Xq_work)) return W8A8_ERR_INVALID_ARG;
    if (layer->chunk_plan && !aligned16(layer->chunk_plan)) return W8A8_ERR_MISALIGNED;
    // validate the GEMM's arguments before anything is enqueued
    w8a8::GemmBranch b{direct16 ? reinterpret_cast<const int8_t *>(workspace) : Xq_work, x_scale_work,
                       layer->Wq, layer->w_scale, layer->bias, Y, M, nullptr, layer->chunk_plan};
    if (w8a8_status e = check_branch(b, true, N, K)) return e;
    if (!X) return W8A8_ERR_INVALID_ARG;
    if (!aligned16(X) || (layer->smooth && !aligned16(layer->smooth))) return W8A8_ERR_MISALIGNED;
    cudaStream_t st = as_stream(stream);
    if (direct16) {
        unsigned int *err = device_error_word();
        if (!err) return W8A8_ERR_CUDA;
        uint16_t *q16 = nullptr;
        uint32_t *ss = nullptr;
        w8a8::linear_workspace_views(workspace, M, K, &q16, &ss);
        cudaError_t e = w8a8::launch_quant_act_f16codes(X, layer->smooth, M, K, q16, x_scale_work, ss, false, st);
        if (e != cudaSuccess) return W8A8_ERR_CUDA;
        b.Xq = reinterpret_cast<const int8_t *>(q16);
        b.x_sumsq = ss;
        return from_cuda(w8a8::launch_gemm_ts(&b, 1, N, K, false, workspace, err, st));
    }
    if (w8a8_status e = w8a8_quant_act(X, layer->smooth, M, K, Xq_work, x_scale_work, stream))
        return e;
    return run_gemm_ws(&b, 1, N, K, false, workspace, st);
}

w8a8_status w8a8_select_protected(const float *score, int L, int n_protect, int *protect_flags) {
    if (L < 0 || n_protect < 0 || n_protect > L) return W8A8_ERR_INVALID_ARG;
    if (L > 0 && (!score || !protect_flags)) return W8A8_ERR_INVALID_ARG;
    std::vector<int> order(static_cast<size_t>(L));
    std::iota(order.begin(), order.end(), 0);
    // most fragile first: NaN above every number, then larger scores; equal
    // scores keep the lower layer index first
    auto key_greater = [&](int a, int b) {
        const float sa = score[a], sb = score[b];
        const bool na = std::isnan(sa), nb = std::isnan(sb);
        if (na != nb) return na;
        if (!na && sa != sb) return sa > sb;
        return a < b;
    };
    std::stable_sort(order.begin(), order.end(), key_greater);
    for (int i = 0; i < L; ++i) protect_flags[i] = 0;
    for (int i = 0; i < n_protect; ++i) protect_flags[order[static_cast<size_t>(i)]] = 1;
    return W8A8_OK;
}

w8a8_status w8a8_debug_wait_timeout(uint32_t limit_us, void *stream) {
    if (limit_us == 0 || limit_us > 2000000u) return W8A8_ERR_INVALID_ARG;
    unsigned int *err = device_error_word();
    if (!err) return W8A8_ERR_CUDA;
    return from_cuda(w8a8::launch_wait_probe(err, 1000ull * limit_us, as_stream(stream)));
}

w8a8_status w8a8_device_status(void *stream, uint32_t *detail) {
    cudaStream_t st = as_stream(stream);
    if (cudaStreamSynchronize(st) != cudaSuccess) return W8A8_ERR_CUDA;
    unsigned int word = 0;
    if (cudaMemcpyFromSymbol(&word, g_w8a8_device_error, sizeof word) != cudaSuccess)
        return W8A8_ERR_CUDA;
    if (word != 0) {
        const unsigned int zero = 0;
        if (cudaMemcpyToSymbol(g_w8a8_device_error, &zero, sizeof zero) != cudaSuccess)
            return W8A8_ERR_CUDA;
    }
    if (detail) *detail = word;
    return word ? W8A8_ERR_TIMEOUT : W8A8_OK;
}

}  // extern "C"
