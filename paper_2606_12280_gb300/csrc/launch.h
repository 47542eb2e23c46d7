// launch.h -- host-side launchers of the library's kernels (internal).
// Arguments are validated by the C-ABI layer before any of these is called.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace w8a8 {

// Launch `kern` with programmatic stream serialization: it may start while
// the previous kernel in `st` finishes, and must wait for it
// (griddepcontrol.wait) before touching anything that kernel could write.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, int threads, size_t smem, cudaStream_t st,
                       Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

struct GemmBranch {
    const int8_t *Xq;
    const float *x_scale;
    const int8_t *Wq;
    const float *w_scale;
    const float *bias;
    void *out;        // uint16_t* bf16 Y, or int32_t* acc for the debug export
    int M;
    const uint32_t *x_sumsq;   // fp16-code GEMM: per token sum of squared codes, or null
    const uint32_t *plan;      // fp16-code GEMM: the weights' drain plan, or null
};

cudaError_t launch_channel_absmax(const uint16_t *X, int T, int K, float *s,
                                  cudaStream_t st);
cudaError_t launch_smooth_scales(const float *s, const float *W, int N, int K,
                                 float alpha, float *lambda, cudaStream_t st);
cudaError_t launch_quantize_weights(const float *W, const float *lambda, int N,
                                    int K, int8_t *Wq, float *w_scale,
                                    cudaStream_t st);
cudaError_t launch_quant_act(const uint16_t *X, const float *lambda, int M,
                             int K, int8_t *Xq, float *x_scale, unsigned int *err,
                             cudaStream_t st);

// One branch of the dual-branch activation quantization.
struct QuantActBranch {
    const uint16_t *X;
    const float *lambda;
    int M;
    int8_t *Xq;
    float *x_scale;
};

// a3 for both branches in one launch (two launches for K > 16384).
cudaError_t launch_quant_act_dual(const QuantActBranch *br, int K, cudaStream_t st);

// a3 with fp16 codes for both branches in one launch, K <= 16384.
struct QuantActBranch16 {
    const uint16_t *X;
    const float *lambda;
    int M;
    uint16_t *Xq16;
    float *x_scale;
    uint32_t *sumsq;
};
cudaError_t launch_quant_act_dual_f16codes(const QuantActBranch16 *br, int K, cudaStream_t st);

// a3 of GELU(H): the GELU evaluated in fp32 and quantized without rounding
// to bf16 in between.
cudaError_t launch_gelu_quant_act(const uint16_t *H, const float *lambda, int M, int K, int8_t *Xq,
                                  float *x_scale, cudaStream_t st);

// Test export: the fp32 GELU values the fused pass uses.
cudaError_t launch_debug_gelu(const uint16_t *H, int n, float *G, cudaStream_t st);

// Legacy warp-level mma.sync s8 GEMM (exact int32), nb = 1 or 2 branches.
// out_i32: write the int32 product instead of the bf16 epilogue.
cudaError_t launch_gemm_mma(const GemmBranch *br, int nb, int N, int K,
                            bool out_i32, cudaStream_t st);

// tcgen05 GEMM on pairs of SMs (cta_group::2), same exact scheme.  a16: Xq
// holds the codes as fp16 values (2 bytes each) and is not converted.
cudaError_t launch_gemm_tc2(const GemmBranch *br, int nb, int N, int K,
                            bool out_i32, bool a16, unsigned int *err, cudaStream_t st);

// tcgen05 GEMM on CTA pairs with the weights in tensor memory: Xq holds the
// activation codes as fp16 values (2 bytes each), Wq the int8 weights.  A
// branch's plan (from launch_chunk_plan on its Wq) and x_sumsq (from a3) let
// the accumulation skip drains where they bound the partial sums.
// workspace: NULL, or gemm_ts_workspace_bytes() bytes whose counters are
// zero (the kernel leaves them zero): the last, partial round of tiles is
// then split over K between the idle CTA pairs.
cudaError_t launch_gemm_ts(const GemmBranch *br, int nb, int N, int K, bool out_i32, void *workspace,
                           unsigned int *err, cudaStream_t st);
long long gemm_ts_workspace_bytes();
// The same engine on int8 codes: one streaming pass writes each branch's
// codes as fp16 values and its token sums of squares into the workspace
// (linear_codes8_workspace_bytes(M0 + M1, K) bytes, the split-K counters
// zeroed once), then the GEMM above runs on them with the branch's plan.
long long linear_codes8_workspace_bytes(long long tokens, int K);
cudaError_t launch_linear_codes8(const GemmBranch *br, int nb, int N, int K, bool out_i32, void *workspace,
                                 unsigned int *err, cudaStream_t st);
// The single-branch layout of that workspace: where the fp16 codes and the
// token sums of M tokens go (a3 may write them there directly).
void linear_workspace_views(void *workspace, int M, int K, uint16_t **codes16, uint32_t **sumsq);
int chunk_plan_words(int K);    // per block of 256 weight rows
cudaError_t launch_chunk_plan(const int8_t *Wq, int N, int K, uint32_t *plan, cudaStream_t st);

// a3 (optionally of GELU(X)) writing the codes as fp16 values, K <= 16384.
cudaError_t launch_quant_act_f16codes(const uint16_t *X, const float *lambda, int M, int K,
                                     uint16_t *Xq16, float *x_scale, uint32_t *sumsq, bool gelu,
                                     cudaStream_t st);

// tcgen05 GEMM (exact integer products on the fp16 tensor datapath).
cudaError_t launch_gemm_tc(const GemmBranch *br, int nb, int N, int K,
                           bool out_i32, unsigned int *err, cudaStream_t st);

// Protected (bf16) linear on tcgen05 CTA pairs: Y = bf16(X W^T + b).
cudaError_t launch_gemm_bf16(const uint16_t *X, const uint16_t *W, const float *bias, int M,
                             int N, int K, uint16_t *Y, unsigned int *err, cudaStream_t st);

// GGUF weight-only linear (fmt 0 = Q8_0, 1 = Q4_K) on tcgen05 CTA pairs.
cudaError_t launch_gemm_gguf(const uint16_t *X, const uint8_t *Wraw, int fmt, const float *bias, int M,
                             int N, int K, uint16_t *Y, unsigned int *err, cudaStream_t st);
// Test export: the decoded bf16 weights.
cudaError_t launch_gguf_dequant(const uint8_t *Wraw, int fmt, int N, int K, uint16_t *W,
                                cudaStream_t st);

// Activation statistics: accumulate sums / absmax, then finalize.
cudaError_t launch_act_stats_update(const uint16_t *X, int T, int K, const float *shift,
                                    double *sums, float *absmax, cudaStream_t st);
cudaError_t launch_act_stats_finalize(const double *sums, const float *absmax, const float *shift,
                                      long long count, int K, float *chan, float *tensor,
                                      cudaStream_t st);

// One-shot statistics of one batch into chan / tensor, with the sums in the
// library's static device scratch (K <= W8A8_NOALLOC_STATS_MAX_K).
cudaError_t launch_act_stats_noalloc(const uint16_t *X, int T, int K, const float *shift, float *chan,
                                     float *tensor, cudaStream_t st);

// Per-tensor activation quantization (two passes: tensor max, then codes).
cudaError_t launch_quant_act_per_tensor(const uint16_t *X, const float *lambda, int M, int K,
                                        int8_t *Xq, float *x_scale, float *amax, cudaStream_t st);

// Test hook: one bounded wait that is never satisfied (failure detection).
cudaError_t launch_wait_probe(unsigned int *err, uint64_t limit_ns, cudaStream_t st);

}  // namespace w8a8
