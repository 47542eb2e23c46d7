/*
 * w8a8.h -- C ABI of the GB300 (sm_103a) W8A8 quantized linear layer.
 *
 * The layer is the INT8 W8A8 recipe of "Quantizing a Dual-Branch Flow-Matching
 * Diffusion Transformer for Consumer GPUs" (Sec. 3, Method, paragraph
 * "INT8 W8A8"): per-output-channel symmetric INT8 weights, per-token dynamic
 * symmetric INT8 activations, SmoothQuant outlier migration with
 *     lambda_j = s_j^alpha / max_i |W_ij|^(1 - alpha),
 * activations divided by lambda and weights multiplied by it before
 * quantization.  The INT8 x INT8 -> INT32 product with a fused dequantizing
 * epilogue is the kernel the paper reports as missing (Sec. 5, Efficiency;
 * Sec. 7, Limitations), and the two separate-weight branches (conditional and
 * unconditional) of its classifier-free-guidance DiT (Sec. 1; Sec. 3,
 * Setting) run as one grouped launch.
 *
 * Conventions shared by every entry point
 *   - Every pointer is a DEVICE pointer owned by the caller (for example the
 *     data_ptr() of a CUDA tensor).  The library allocates nothing and never
 *     frees anything.  Every base pointer must be 16-byte aligned.
 *   - Every buffer must hold the elements that the call's shapes imply (for
 *     example M * N for Y): the library receives plain pointers and cannot
 *     check their extent.
 *   - Matrices are row-major and dense (row stride = number of columns).
 *     X [M,K] activations (tokens x input channels), W / Wq [N,K] weights
 *     (output channels x input channels, the nn.Linear layout), Y [M,N].
 *   - bf16 values travel as their 16-bit patterns (uint16_t).
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Every
 *     call only enqueues work on that stream and returns at once; results are
 *     ready when the stream reaches them.  Calls on one stream are ordered.
 *   - Shapes: M >= 0 (M == 0 is a no-op that returns W8A8_OK), N > 0 and a
 *     multiple of 8, K > 0 and a multiple of 16, K <= 133143 (so that
 *     K * 127^2 fits in int32).
 *   - Arithmetic is IEEE binary32 with round-to-nearest-even on every step and
 *     no fused multiply-add, so INT8 codes and FP32 scales are reproducible
 *     bit for bit; rounding to INT8 is half-to-even with a symmetric clamp
 *     to [-127, 127]; the INT32 product is exact.
 *   - Errors: argument checks run on the host before anything is enqueued.
 *     W8A8_ERR_INVALID_ARG (null pointer, alpha outside [0,1]),
 *     W8A8_ERR_UNSUPPORTED_SHAPE, W8A8_ERR_MISALIGNED (a pointer not 16-byte
 *     aligned) leave the stream untouched.  W8A8_ERR_CUDA reports a launch
 *     failure.  The library keeps one device-side error word (see
 *     w8a8_device_status), the fixed scratch of w8a8_act_stats_noalloc and
 *     the constant GELU table of w8a8_gelu_quant_act; it holds no other
 *     state (per-device kernel attributes are set once,
 *     thread-safely), and calls on different streams or host threads do not
 *     affect one another.
 *   - Every pointer refers to memory of the CURRENT device (cudaSetDevice),
 *     on which the call launches its work.
 */
#ifndef W8A8_H
#define W8A8_H

#include <stdint.h>

#if defined(__GNUC__)
#define W8A8_API __attribute__((visibility("default")))
#else
#define W8A8_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    W8A8_OK = 0,
    W8A8_ERR_INVALID_ARG = 1,
    W8A8_ERR_UNSUPPORTED_SHAPE = 2,
    W8A8_ERR_MISALIGNED = 3,
    W8A8_ERR_CUDA = 4,
    W8A8_ERR_TIMEOUT = 5
} w8a8_status;

/* A bound on K under which K * 127 * 127 < 2^31 (every |acc| of codes in
 * [-127, 127] fits int32); with K a multiple of 16 the largest accepted K is
 * 133136. */
#define W8A8_MAX_K 133143

/* Human-readable name of a status code (static storage, never NULL). */
W8A8_API const char *w8a8_status_string(w8a8_status status);

/*
 * Calibration statistic s_j = max_t |X_tj| over a batch of T tokens: the
 * per-channel activation scale that feeds the smoothing vector (Sec. 3,
 * "INT8 W8A8", where s is measured by a calibration pass over held-out
 * prompts).
 *   X      [T,K] bf16, read.
 *   s      [K] fp32, written (overwritten, not accumulated).
 */
W8A8_API w8a8_status w8a8_channel_absmax(const uint16_t *X, int T, int K, float *s,
                                void *stream);

/*
 * a1. Smoothing vector (Sec. 3, "INT8 W8A8"):
 *     lambda_j = s_j^alpha / m_j^(1-alpha),  m_j = max_i |W_ij| (over output
 *     rows i of input channel j).  s_j == 0 or m_j == 0 gives lambda_j = 1.
 *     alpha in {0, 1/2, 1} is evaluated with correctly rounded fp32
 *     operations (sqrt(s)/sqrt(m), 1/m, s); any other alpha in binary64 and
 *     rounded once.
 *   act_absmax [K] fp32 (s), read.   W [N,K] fp32, read.
 *   smooth     [K] fp32 (lambda), written; also used as working storage for
 *              m_j during the call.
 *   alpha      in [0, 1], else W8A8_ERR_INVALID_ARG.
 */
W8A8_API w8a8_status w8a8_smooth_scales(const float *act_absmax, const float *W, int N,
                               int K, float alpha, float *smooth, void *stream);

/*
 * a2. Per-output-channel symmetric INT8 weights of W' = W diag(lambda)
 * (Sec. 3, "INT8 W8A8", per-channel weights; weights multiplied by lambda):
 *     w'_ij = W_ij * lambda_j;  a_i = max_j |w'_ij|;
 *     w_scale_i = a_i / 127;  Wq_ij = clamp(rne(w'_ij * (127 / a_i)), +-127);
 *     an all-zero row gives w_scale_i = 0 and codes 0.
 *   W       [N,K] fp32, read.   smooth [K] fp32 or NULL (lambda = 1).
 *   Wq      [N,K] int8, written.   w_scale [N] fp32, written.
 */
W8A8_API w8a8_status w8a8_quantize_weights(const float *W, const float *smooth, int N,
                                  int K, int8_t *Wq, float *w_scale,
                                  void *stream);

/*
 * a3. Per-token dynamic INT8 activations of X' = X diag(lambda)^-1
 * (Sec. 3, "INT8 W8A8", per-token dynamic activations; activations divided
 * by lambda, implemented as a multiply by the correctly rounded 1/lambda_j):
 *     x'_mj = X_mj * (1/lambda_j);  a_m = max_j |x'_mj|;
 *     x_scale_m = a_m / 127;  Xq_mj = clamp(rne(x'_mj * (127 / a_m)), +-127);
 *     an all-zero token gives x_scale_m = 0 and codes 0.
 *   X       [M,K] bf16, read.   smooth [K] fp32 or NULL (lambda = 1).
 *   Xq      [M,K] int8, written.   x_scale [M] fp32, written.
 * One pass over X: reads 2MK bytes, writes MK + 4M.
 */
W8A8_API w8a8_status w8a8_quant_act(const uint16_t *X, const float *smooth, int M,
                           int K, int8_t *Xq, float *x_scale, void *stream);

/*
 * a4 + a5. Quantized linear with the dequantizing epilogue fused:
 *     acc_mn = sum_k Xq_mk * Wq_nk          (exact int32)
 *     Y_mn   = bf16_rne(((float)acc_mn * x_scale_m) * w_scale_n + bias_n)
 *   Xq [M,K] int8, x_scale [M] fp32, Wq [N,K] int8, w_scale [N] fp32,
 *   bias [N] fp32 or NULL (no bias), all read.   Y [M,N] bf16, written.
 * The product runs exactly on the fp16 tensor datapath (every int8 is an
 * fp16 value, products are exact in fp32; partial sums of at most 1024
 * products stay below 2^24 and are drained into int32).
 *   chunk_plan: NULL, or the plan that w8a8_chunk_plan wrote for this Wq
 *     (same N, K); used with a workspace (see w8a8_linear_f16codes).  A
 *     plan of other weights voids the exactness guarantee.
 *   workspace: NULL, or w8a8_linear_workspace_size(M, K) bytes of device
 *     memory (16-byte aligned) that the caller zeroed once before its first
 *     use.  Without one, both operands are converted to fp16 in shared
 *     memory inside the GEMM.  With one, a streaming pass first writes the
 *     codes as fp16 values and each token's sum of squared codes into it
 *     (3MK + 4M bytes moved, the fp16 codes left in L2), and the GEMM of
 *     w8a8_linear_f16codes runs on them (the weights converted into tensor
 *     memory, the split-K area of the same workspace).  Same bits either
 *     way.  Calls that overlap in time need workspaces of their own.
 */
W8A8_API w8a8_status w8a8_linear(const int8_t *Xq, const float *x_scale,
                        const int8_t *Wq, const float *w_scale,
                        const float *bias, int M, int N, int K, uint16_t *Y,
                        const uint32_t *chunk_plan, void *workspace, void *stream);

/* Bytes of the workspace of w8a8_linear (tokens = M) and w8a8_linear_dual
 * (tokens = M0 + M1) for K on the current device: 2 * tokens * K for the
 * fp16 codes, 4 * tokens for the token sums, w8a8_gemm_workspace_size() for
 * the split-K area, and 1024 bytes of alignment.  0 for tokens < 0 or
 * K <= 0. */
W8A8_API long long w8a8_linear_workspace_size(long long tokens, int K);

/* One branch of the dual-branch (classifier-free guidance) layer. */
typedef struct {
    const int8_t *Xq;      /* [M,K] int8 */
    const float *x_scale;  /* [M] fp32 */
    const int8_t *Wq;      /* [N,K] int8 */
    const float *w_scale;  /* [N] fp32 */
    const float *bias;     /* [N] fp32 or NULL */
    uint16_t *Y;           /* [M,N] bf16, written */
    int M;                 /* tokens of this branch, >= 0 */
    const uint32_t *chunk_plan;  /* this branch's weights' plan or NULL */
} w8a8_branch;

/*
 * a6. The same linear layer for both separate-weight branches (conditional
 * br[0], unconditional br[1]; Sec. 1 and Sec. 3 "Setting": two
 * separate-weight copies of the backbone, 211 linears each) in ONE launch
 * whose tile space covers both.  The branches share N and K; each has its
 * own M, activations, weights, scales, bias and output.  Results are
 * bitwise identical to two w8a8_linear calls.
 *   br  host pointer to an array of 2 w8a8_branch (read during the call only).
 *   workspace: NULL, or w8a8_linear_workspace_size(M0 + M1, K) bytes, as
 *     for w8a8_linear (one streaming pass for both branches' codes).
 */
W8A8_API w8a8_status w8a8_linear_dual(const w8a8_branch *br, int N, int K,
                             void *workspace, void *stream);

/*
 * Test export of a4 alone: acc = Xq Wq^T as int32 [M,N], written, so that the
 * exact integer product can be compared bit for bit.  Same shape rules,
 * chunk_plan and workspace as w8a8_linear.
 */
W8A8_API w8a8_status w8a8_debug_gemm_i32(const int8_t *Xq, const int8_t *Wq, int M,
                                int N, int K, int32_t *acc, const uint32_t *chunk_plan,
                                void *workspace, void *stream);

/*
 * Test anchors (no counterpart in the paper): the same exact-integer product
 * on the earlier int8-code GEMM engines, selected per call (nothing
 * process-wide).  engine 2 = the engine of w8a8_linear (tcgen05 on pairs of
 * SMs), 1 = tcgen05 on single SMs, 0 = warp-level mma.sync s8 (the legacy
 * INT8 tensor path); other values give W8A8_ERR_INVALID_ARG.  nb = 1 or 2
 * branches (br[0..nb-1]).  out_i32 nonzero: each branch's Y receives the
 * int32 product [M,N] instead (x_scale, w_scale and bias unused).
 */
W8A8_API w8a8_status w8a8_debug_linear_engine(int engine, const w8a8_branch *br, int nb, int N, int K,
                                              int out_i32, void *stream);

/* ------------------------------------------------------------------------
 * The same layer with the activation codes in a 16-bit container.
 * ---------------------------------------------------------------------- */

/*
 * a3 with the codes written as fp16 values: Xq16_mj is the fp16 bit pattern
 * of the same integer code w8a8_quant_act writes as int8 (every integer in
 * [-127, 127] is exactly an fp16 value), x_scale as w8a8_quant_act.  gelu
 * nonzero: quantize GELU(X) as w8a8_gelu_quant_act does.  The GEMM below then
 * takes A without converting it.  K <= 16384, else
 * W8A8_ERR_UNSUPPORTED_SHAPE.  Writes 2MK + 4M bytes (one MK more than a3).
 *   X [M,K] bf16, smooth [K] fp32 or NULL, read.
 *   Xq16 [M,K] fp16 codes (uint16 bit patterns), x_scale [M] fp32, written.
 *   x_sumsq [M] uint32 or NULL: if given, sum_j Xq_mj^2 per token, written
 *     (exact; no counterpart in the paper: w8a8_linear_f16codes uses it to
 *     bound its partial sums).
 */
W8A8_API w8a8_status w8a8_quant_act_f16codes(const uint16_t *X, const float *smooth, int M,
                                             int K, uint16_t *Xq16, float *x_scale,
                                             uint32_t *x_sumsq, int gelu, void *stream);

/*
 * a4 + a5 with the activation codes as fp16 values (from
 * w8a8_quant_act_f16codes): the same exact INT32 product and epilogue as
 * w8a8_linear, bitwise equal outputs.  The codes go to the tensor cores by
 * TMA without a conversion and the int8 weights are converted into tensor
 * memory, so no converted operand passes through shared memory.
 *   Xq16 [M,K] fp16 codes (|code| <= 128), otherwise as w8a8_linear.
 *   chunk_plan: NULL, or the plan that w8a8_chunk_plan wrote for this Wq
 *     (same N, K); with it the integer sums are drained from the fp32
 *     accumulator only where the weights require it (see w8a8_chunk_plan).
 *     A plan of other weights voids the exactness guarantee.
 *   x_sumsq: NULL, or the per-token sums of squared codes that
 *     w8a8_quant_act_f16codes wrote with these Xq16 (used with a plan): an
 *     output tile (256 tokens x 256 features) whose largest token sum times
 *     its largest weight-row sum of squares is at most 2^48 has every partial
 *     sum within 2^24 (Cauchy-Schwarz) and is accumulated without a drain.
 *     Sums of other codes void the exactness guarantee.
 *   workspace: NULL, or w8a8_gemm_workspace_size() bytes of device memory
 *     (16-byte aligned) that the caller zeroed once before its first use.
 *     The output tiles (256 x 256) fill the GPU's CTA pairs in rounds; with a
 *     workspace and at most 12 full rounds, as many tiles as a last,
 *     partial round would hold (all tiles, when there are fewer tiles than
 *     pairs) are split over K between pairs in the first round, their int32
 *     partial sums meet in the workspace, and the part that finishes last
 *     adds them (integer sums: the result is the same bits as without a
 *     workspace).  The kernel leaves the workspace's
 *     counters zero; after a call that returned an error, zero it again.
 *     Calls that overlap in time need workspaces of their own.
 */
W8A8_API w8a8_status w8a8_linear_f16codes(const uint16_t *Xq16, const float *x_scale,
                                          const int8_t *Wq, const float *w_scale,
                                          const float *bias, int M, int N, int K,
                                          const uint32_t *chunk_plan, const uint32_t *x_sumsq,
                                          uint16_t *Y, void *workspace, void *stream);

/* Bytes of the workspace of w8a8_linear_f16codes on the current device (one
 * int32 256 x 256 tile per CTA pair, and counters). */
W8A8_API long long w8a8_gemm_workspace_size(void);

/*
 * Test export of the product above alone: acc = Xq16 Wq^T as int32 [M,N],
 * written.  Same shape rules, plan, token sums and workspace.
 */
W8A8_API w8a8_status w8a8_debug_gemm_f16codes_i32(const uint16_t *Xq16, const int8_t *Wq, int M,
                                                  int N, int K, const uint32_t *chunk_plan,
                                                  const uint32_t *x_sumsq, int32_t *acc,
                                                  void *workspace, void *stream);

/* One branch of the dual-branch layer with fp16 codes (a6 on this path). */
typedef struct {
    const uint16_t *X;     /* [M,K] bf16 */
    const float *smooth;   /* [K] fp32 (this branch's lambda) or NULL */
    int M;                 /* tokens of this branch, >= 0 */
    uint16_t *Xq16;        /* [M,K] fp16 codes, written */
    float *x_scale;        /* [M] fp32, written */
    uint32_t *x_sumsq;     /* [M] uint32 or NULL, written */
} w8a8_act_branch16;

typedef struct {
    const uint16_t *Xq16;        /* [M,K] fp16 codes */
    const float *x_scale;        /* [M] fp32 */
    const int8_t *Wq;            /* [N,K] int8 */
    const float *w_scale;        /* [N] fp32 */
    const float *bias;           /* [N] fp32 or NULL */
    uint16_t *Y;                 /* [M,N] bf16, written */
    int M;                       /* tokens of this branch, >= 0 */
    const uint32_t *chunk_plan;  /* this branch's weights' plan or NULL */
    const uint32_t *x_sumsq;     /* this branch's token sums or NULL */
} w8a8_branch16;

/*
 * a3 of both separate-weight branches (Sec. 1 and 3: the conditional br[0]
 * and unconditional br[1] backbones) with fp16 codes, in one launch, as
 * w8a8_quant_act_dual does for int8 codes; each branch as
 * w8a8_quant_act_f16codes.  K <= 16384.
 */
W8A8_API w8a8_status w8a8_quant_act_dual_f16codes(const w8a8_act_branch16 *br, int K, void *stream);

/*
 * a4 + a5 of both branches in one grouped launch (a6) with fp16 codes: the
 * tile space covers both branches, each tile with its own branch's operands,
 * plan and token sums; results as two w8a8_linear_f16codes calls, bitwise.
 * The branches share N and K.  workspace as w8a8_linear_f16codes (the last
 * round's tiles of both branches are split).
 */
W8A8_API w8a8_status w8a8_linear_dual_f16codes(const w8a8_branch16 *br, int N, int K,
                                               void *workspace, void *stream);

/*
 * Drain plan of an int8 weight matrix for w8a8_linear_f16codes (no
 * counterpart in the paper: a property of the exact-integer scheme on fp32
 * accumulators).  The GEMM accumulates integer products in fp32 tensor
 * memory, exact while every partial sum stays within 2^24; with codes
 * |a| <= 128 a partial sum over a K range is at most 128 * sum |w_k| over
 * it, so a run of K chunks (1024 each) can accumulate without a drain while
 * every weight row of a 256-row block has sum |w_k| <= 2^17 over the run.
 * The plan records, per 256-row block, after which chunks the run ends (the
 * worst case, |w| = 127 everywhere, ends it after every chunk), and the
 * block's largest row sum of squares (for the x_sumsq bound).  Computed once
 * per weight matrix; its layout is internal to the library.
 *   w8a8_chunk_plan_size: the number of uint32 words of the plan (>= 1).
 *   Wq [N,K] int8, read;  plan [w8a8_chunk_plan_size(N, K)] uint32, written.
 */
W8A8_API long long w8a8_chunk_plan_size(int N, int K);
W8A8_API w8a8_status w8a8_chunk_plan(const int8_t *Wq, int N, int K, uint32_t *plan, void *stream);

/* ------------------------------------------------------------------------
 * GGUF weight-only layers (Sec. 3, "GGUF k-quants": the DiT serialized to
 * Q8_0, 8.5 bits per weight, and Q4_K, 4.5 bits, the paper's memory-Pareto
 * variant, which it ran with a Torch dequantization).
 * ---------------------------------------------------------------------- */

#define W8A8_GGUF_Q8_0 0
#define W8A8_GGUF_Q4_K 1

/*
 * Weight blocks in the public GGUF/ggml layouts, little-endian, each weight
 * row [K] a run of consecutive blocks (row stride = K/32*34 bytes for Q8_0,
 * K/256*144 for Q4_K):
 *   Q8_0: 32 weights in 34 bytes, fp16 d then 32 int8 q;  w = d * q.
 *   Q4_K: 256 weights in 144 bytes, fp16 d, fp16 dmin, 12 bytes of eight
 *     6-bit scales sc_j and mins m_j (j < 4: sc = s[j] & 63, m = s[j+4] & 63;
 *     j >= 4: sc = (s[j+4] & 15) | (s[j-4] >> 6) << 4,
 *             m  = (s[j+4] >> 4) | (s[j] >> 6) << 4),
 *     then 128 bytes of 4-bit quants: weights 64c..64c+31 are the low
 *     nibbles of quant bytes 32c..32c+31 (j = 2c), weights 64c+32..64c+63
 *     their high nibbles (j = 2c+1);  w = (d * sc_j) * q - dmin * m_j.
 * Decoding runs in fp32 (only the Q4_K subtraction rounds: the products of
 * these small integers and fp16 values are exact); the layer consumes the
 * decoded weights rounded to bf16 (nearest even).
 *
 * Weight-only linear:
 *     Y_mn = bf16_rne(fl32(sum_k X_mk * bf16(w_nk)) + bias_n)
 * with fp32 tensor-core accumulation, as w8a8_linear_bf16.
 *   X [M,K] bf16, Wraw [N rows of blocks], bias [N] fp32 or NULL, read.
 *   Y [M,N] bf16, written.  fmt W8A8_GGUF_Q8_0 or W8A8_GGUF_Q4_K, else
 *   W8A8_ERR_INVALID_ARG; N a multiple of 8 and K of 256, else
 *   W8A8_ERR_UNSUPPORTED_SHAPE.
 */
W8A8_API w8a8_status w8a8_linear_gguf(const uint16_t *X, const uint8_t *Wraw, int fmt,
                                      const float *bias, int M, int N, int K, uint16_t *Y,
                                      void *stream);

/* Test export: the decoded weights W [N,K] bf16, written. */
W8A8_API w8a8_status w8a8_debug_gguf_dequant(const uint8_t *Wraw, int fmt, int N, int K,
                                             uint16_t *W, void *stream);

/* ------------------------------------------------------------------------
 * a3 fused with its neighbours in the DiT block.
 * ---------------------------------------------------------------------- */

/* One branch of the dual-branch activation quantization. */
typedef struct {
    const uint16_t *X;     /* [M,K] bf16 */
    const float *smooth;   /* [K] fp32 (this branch's lambda) or NULL */
    int M;                 /* tokens of this branch, >= 0 */
    int8_t *Xq;            /* [M,K] int8, written */
    float *x_scale;        /* [M] fp32, written */
} w8a8_act_branch;

/*
 * a3 for both separate-weight branches (conditional br[0], unconditional
 * br[1]; each with its own smoothing vector) in one launch whose row space
 * covers both (two launches when K > 16384).  Results are bitwise identical
 * to two w8a8_quant_act calls.
 *   br  host pointer to an array of 2 w8a8_act_branch (read during the call).
 */
W8A8_API w8a8_status w8a8_quant_act_dual(const w8a8_act_branch *br, int K, void *stream);

/*
 * a3 of the FFN down-projection input GELU(H) in one pass over H, the
 * up-projection's bf16 output (the down-projections are the fragile layers
 * of Sec. 3, "Activation-fragility profiling and protection"; the paper does
 * not name the activation, the exact erf form is taken):
 *     g_mj = GELU(H_mj) = (H_mj / 2) * erfc(-H_mj / sqrt 2)
 *            evaluated in binary64 and rounded once to fp32,
 *     then w8a8_quant_act's arithmetic on g (no rounding of g to bf16).
 * g is exact as defined: H is bf16, so the pass reads g from a table that
 * holds it for each of the 65536 bf16 bit patterns.  The library builds the
 * table (256 KB of device memory, kept until the process exits) on each
 * device the first time a GELU pass runs there, synchronously and outside
 * the caller's stream: make that first call before capturing a stream into
 * a CUDA graph (later calls are capturable).
 *   H [M,K] bf16, read.   smooth [K] fp32 or NULL.
 *   Xq [M,K] int8, x_scale [M] fp32, written.
 */
W8A8_API w8a8_status w8a8_gelu_quant_act(const uint16_t *H, const float *smooth, int M, int K,
                                         int8_t *Xq, float *x_scale, void *stream);

/*
 * Test export of the GELU that w8a8_gelu_quant_act uses: G[i] = g(H[i]) in
 * fp32 for n values (n >= 0), read from the same table (built on first use
 * as above).  H [n] bf16, read; G [n] fp32, written.
 */
W8A8_API w8a8_status w8a8_debug_gelu(const uint16_t *H, int n, float *G, void *stream);

/* ------------------------------------------------------------------------
 * Around the W8A8 layer: the ablation's per-tensor activation scale, the
 * activation statistics of fragility profiling, and the protected (bf16)
 * layers with per-layer dispatch.
 * ---------------------------------------------------------------------- */

/*
 * Per-tensor INT8 activations: the naive arm of the activation-quant ablation
 * (Sec. 5, "What drives INT8 recovery"; the naive per-tensor INT8 that
 * SmoothQuant is contrasted with in Sec. 2).  Same arithmetic as
 * w8a8_quant_act with the maximum taken over the whole tensor:
 *     x'_mj = X_mj * (1/lambda_j);  a = max_mj |x'_mj|;
 *     x_scale_m = a / 127 for every m;  Xq_mj = clamp(rne(x'_mj * (127/a)), +-127);
 *     a == 0 gives scale 0 and codes 0.
 * Because every row carries the same scale, w8a8_linear consumes the result
 * unchanged.
 *   X [M,K] bf16, read.   smooth [K] fp32 or NULL (lambda = 1), read.
 *   Xq [M,K] int8, x_scale [M] fp32, written.   amax [1] fp32, written (a).
 * Two passes over X (the second usually from L2): 4MK bytes read, MK + 4M
 * written.
 */
W8A8_API w8a8_status w8a8_quant_act_per_tensor(const uint16_t *X, const float *smooth, int M,
                                               int K, int8_t *Xq, float *x_scale, float *amax,
                                               void *stream);

/*
 * Activation statistics for fragility profiling (Sec. 3, "Activation-fragility
 * profiling and protection": every linear's input is recorded over the
 * denoising trajectory as max-abs, standard deviation and kurtosis).
 * Accumulates, for each input channel j over the T tokens of X,
 *     sums[(p-1)*K + j] += sum_t (X_tj - c_j)^p     p = 1, 2, 3, 4  (fp64)
 *     absmax[j]          = max(absmax[j], max_t |X_tj|)
 * with c = shift (or 0 when shift is NULL).  Call it once per recorded batch
 * (any number of times, same shift); the caller zeroes sums [4K] and absmax
 * [K] before the first call and keeps the total token count.  A shift near
 * each channel's mean (for example from a first batch) keeps the power sums
 * well conditioned.  Each thread sums at most 64 of its rows in fp32, adds at
 * most 64 such group sums in fp32, a block adds its 8 warps' sums in fp32,
 * and only those block sums are added into fp64: every returned sum is within
 * (2 * 64 + 12) * 2^-24 of sum_t |X_tj - c_j|^p of its exact value.  T == 0
 * is a no-op.
 *   X [T,K] bf16, read.   shift [K] fp32 or NULL, read.
 *   sums [4,K] fp64, absmax [K] fp32: read and written (accumulators).
 */
W8A8_API w8a8_status w8a8_act_stats_update(const uint16_t *X, int T, int K, const float *shift,
                                           double *sums, float *absmax, void *stream);

/*
 * Statistics from the accumulators of w8a8_act_stats_update over `count`
 * tokens (count >= 1), in fp64, rounded to fp32 on output:
 *   chan [4,K]: plane 0 max-abs, 1 mean, 2 population standard deviation,
 *               3 Pearson kurtosis m4 / m2^2 (3 for a normal distribution),
 *               per input channel;
 *   tensor [4]: the same four over all count*K elements (channels pooled
 *               about the grand mean).
 * A variance within the accumulation error of zero (at most 1e-5 of the
 * second power sum about the shift) is reported as 0, with kurtosis 0.
 * chan must not overlap sums, absmax or shift (W8A8_ERR_INVALID_ARG): during
 * the call its first floats hold per-32-channel partial sums, overwritten with
 * their final values before the call completes (stream order).
 */
W8A8_API w8a8_status w8a8_act_stats_finalize(const double *sums, const float *absmax,
                                             const float *shift, long long count, int K,
                                             float *chan, float *tensor, void *stream);

/* Largest K of w8a8_act_stats_noalloc (its static scratch holds 36 bytes per
 * input channel: 1.125 MB). */
#define W8A8_NOALLOC_STATS_MAX_K 32768

/*
 * No counterpart in the paper: the statistics of ONE batch without caller
 * accumulators, for callers that want max-abs / mean / std / kurtosis of a
 * single activation tensor and no allocation.  Same arithmetic as
 * w8a8_act_stats_update then w8a8_act_stats_finalize with count = T; the
 * power sums and max-abs live in a file-scope static device scratch of the
 * library (36 bytes x W8A8_NOALLOC_STATS_MAX_K), which every call clears
 * (cudaMemsetAsync) before use.  The library allocates nothing.
 *   - K <= W8A8_NOALLOC_STATS_MAX_K, else W8A8_ERR_UNSUPPORTED_SHAPE; T >= 1,
 *     else W8A8_ERR_INVALID_ARG.
 *   - Calls that overlap in time (different streams, host threads or graphs
 *     in flight at once) share the scratch and race: order them.
 *   - The first call on a device looks the scratch address up
 *     (cudaGetSymbolAddress); make one call before capturing a stream into a
 *     CUDA graph, the later ones are capturable.
 *   X [T,K] bf16, shift [K] fp32 or NULL, read.  chan [4,K], tensor [4] fp32,
 *   written, as w8a8_act_stats_finalize.
 */
W8A8_API w8a8_status w8a8_act_stats_noalloc(const uint16_t *X, int T, int K, const float *shift,
                                            float *chan, float *tensor, void *stream);

/*
 * Protected layer (Sec. 3, "Activation-fragility profiling and protection":
 * the most fragile layers keep bf16 weights and no activation quantization):
 *     Y_mn = bf16_rne(fl32(sum_k X_mk W_nk) + bias_n)
 * with the products of bf16 values exact and the sum accumulated in fp32 by
 * the tensor cores (order unspecified), the bias added in fp32.
 *   X [M,K] bf16, W [N,K] bf16, bias [N] fp32 or NULL, read.  Y [M,N] bf16,
 *   written.  Same shape rules as w8a8_linear.
 */
W8A8_API w8a8_status w8a8_linear_bf16(const uint16_t *X, const uint16_t *W, const float *bias,
                                      int M, int N, int K, uint16_t *Y, void *stream);

/* One linear layer of the protected-INT8 recipe. */
typedef struct {
    int protect;               /* nonzero: protected layer (bf16 path) */
    int N, K;                  /* output and input channels */
    const float *smooth;       /* W8A8: lambda [K] fp32 or NULL */
    const int8_t *Wq;          /* W8A8: [N,K] int8 */
    const float *w_scale;      /* W8A8: [N] fp32 */
    const uint16_t *W_bf16;    /* protected: [N,K] bf16 */
    const float *bias;         /* [N] fp32 or NULL, both paths */
    const uint32_t *chunk_plan;  /* W8A8: w8a8_chunk_plan of Wq, or NULL */
} w8a8_layer;

/*
 * Per-layer dispatch: a protected layer runs w8a8_linear_bf16 on X; any other
 * layer quantizes X (a3) and runs the quantized linear (a4 + a5).
 *   layer  host pointer, read during the call only.
 *   X [M,K] bf16, read.   Y [M,N] bf16, written.
 *   x_scale_work [M] fp32: the token scales (W8A8 path; ignored, may be
 *   NULL, for a protected layer).
 *   workspace: NULL, or w8a8_linear_workspace_size(M, K) bytes as for
 *     w8a8_linear.  With one and K <= 16384, a3 writes the codes as fp16
 *     values with their token sums into it (w8a8_quant_act_f16codes) and the
 *     fp16-code GEMM runs on them; Xq_work is then unused and may be NULL.
 *     Otherwise w8a8_quant_act writes Xq_work [M,K] int8 and w8a8_linear runs
 *     with the workspace (or without one).  Same bits on every path.
 */
W8A8_API w8a8_status w8a8_layer_forward(const w8a8_layer *layer, const uint16_t *X, int M,
                                        int8_t *Xq_work, float *x_scale_work, uint16_t *Y,
                                        void *workspace, void *stream);

/*
 * Choice of the protected set (Sec. 3: the N most fragile of the model's
 * linears stay in bf16; the paper keeps 17 of 211): protect_flags[i] = 1 for
 * the n_protect layers with the largest fragility score, 0 for the others.
 * A NaN score ranks above every number; equal scores keep the lower index
 * first.  How the score is formed from the statistics is the caller's
 * choice.  Host arrays: score [L] read, protect_flags [L] written; no device
 * work.  0 <= n_protect <= L, else W8A8_ERR_INVALID_ARG.
 */
W8A8_API w8a8_status w8a8_select_protected(const float *score, int L, int n_protect,
                                           int *protect_flags);

/*
 * Test hook for failure detection (no counterpart in the paper): enqueues one
 * small kernel whose bounded barrier wait is never satisfied, through the
 * same wait routine the tcgen05 GEMMs use.  After limit_us microseconds
 * (1 .. 2000000, else W8A8_ERR_INVALID_ARG) the wait records code 128 in the
 * device error word and the kernel returns; the context stays usable and the
 * next w8a8_device_status reports W8A8_ERR_TIMEOUT.
 */
W8A8_API w8a8_status w8a8_debug_wait_timeout(uint32_t limit_us, void *stream);

/*
 * Waits for `stream`, then reads and clears the library's device-side error
 * word on the current device.  Kernels that wait on barriers give up after a
 * bounded number of polls, record a code there and return; this call then
 * reports W8A8_ERR_TIMEOUT.  *detail (optional) receives the raw word.
 */
W8A8_API w8a8_status w8a8_device_status(void *stream, uint32_t *detail);

#ifdef __cplusplus
}
#endif

#endif /* W8A8_H */
