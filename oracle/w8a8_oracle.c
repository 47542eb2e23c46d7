/*
 * w8a8_oracle.c -- plain, slow CPU oracle of the W8A8 quantized linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file: only the test-suite, the smoke check and the CPU-baseline leg
 * of the benchmark use it.  It shares no code, header, table or helper with the
 * CUDA library; the two meet only through the seeded input generators.
 *
 * What it computes follows the "INT8 W8A8" paragraph of the paper's Method
 * section (Sec. 3):
 *   - per-output-channel symmetric INT8 weights,
 *   - per-token dynamic symmetric INT8 activations,
 *   - SmoothQuant outlier migration with smoothing vector
 *         lambda_j = s_j^alpha / max_i |W_ij|^(1-alpha),
 *     activations divided by lambda and weights multiplied by it before
 *     quantization,
 * plus the exact INT32 product of the two INT8 operands and the dequantizing
 * epilogue (per-token scale x per-channel scale + bias, rounded to bf16) that
 * the paper names as the missing fused INT8 GEMM (Sec. 7, Limitations).
 *
 * Precision.  The quantization decisions are taken in IEEE binary32 with a
 * pinned operation order (every operation rounded to nearest-even, no fused
 * multiply-add: build with -ffp-contract=off), because INT8 codes and FP32
 * scales are required to be bit-exact between this oracle and the GPU path.
 * The integer product is accumulated in int64 and is exact.  The only step
 * with a transcendental (lambda for alpha not in {0, 1/2, 1}) is evaluated in
 * binary64 and rounded once; that single value is "parity unpinned" at the
 * last fp32 bit and is compared within 1 ulp.
 *
 * Readings where the paper is silent (each listed in the design notes):
 *   - rounding is round-half-to-even, clamp is symmetric [-127, 127];
 *   - max_i |W_ij| runs over output rows i for each input channel j;
 *   - the divide by lambda is a multiply by the correctly rounded reciprocal;
 *   - the per-token scale is taken after smoothing;
 *   - s_j == 0 or max_i|W_ij| == 0 gives lambda_j = 1; an all-zero row gives
 *     scale 0 and codes 0; a NaN product quantizes to 0;
 *   - the epilogue is t = float(acc); t *= sx_m; t *= sw_n; t += b_n;
 *     y = bf16_rne(t).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ */
/* scalar helpers                                                      */
/* ------------------------------------------------------------------ */

static float f32_from_bits(uint32_t u)
{
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

static uint32_t bits_from_f32(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return u;
}

/* bf16 -> fp32 is exact: the bf16 pattern is the top half of the fp32 one. */
float oracle_bf16_to_f32(uint16_t h)
{
    return f32_from_bits((uint32_t)h << 16);
}

/* fp32 -> bf16, round to nearest, ties to even (the IEEE default mode). */
uint16_t oracle_f32_to_bf16_rne(float t)
{
    uint32_t u = bits_from_f32(t);
    if ((u & 0x7fffffffu) > 0x7f800000u)      /* NaN: keep it a quiet NaN */
        return (uint16_t)((u >> 16) | 0x0040u);
    uint32_t keep_lsb = (u >> 16) & 1u;       /* tie goes to the even half */
    u += 0x7fffu + keep_lsb;
    return (uint16_t)(u >> 16);
}

/* the same rounding over an array */
void oracle_f32_to_bf16_rne_array(const float *x, int64_t n, uint16_t *out)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = oracle_f32_to_bf16_rne(x[i]);
}

/* q = clamp(round_half_even(v), -127, 127); a NaN product gives 0. */
static int8_t quantize_rne_clamp(float v)
{
    if (v != v)
        return 0;
    float r = rintf(v);        /* default rounding mode: nearest, ties even */
    if (r > 127.0f)
        r = 127.0f;
    if (r < -127.0f)
        r = -127.0f;
    return (int8_t)r;
}

int8_t oracle_quantize_value(float v) { return quantize_rne_clamp(v); }

/* ------------------------------------------------------------------ */
/* calibration statistic: s_j = max_t |X_tj| (the per-channel          */
/* activation scale that feeds lambda, Sec. 3 "INT8 W8A8")            */
/* ------------------------------------------------------------------ */

void oracle_channel_absmax(const uint16_t *X, int64_t M, int64_t K, float *s)
{
    for (int64_t j = 0; j < K; ++j) {
        float m = 0.0f;
        for (int64_t t = 0; t < M; ++t) {
            float a = fabsf(oracle_bf16_to_f32(X[t * K + j]));
            if (a > m)
                m = a;
        }
        s[j] = m;
    }
}

/* ------------------------------------------------------------------ */
/* a1: smoothing vector, lambda_j = s_j^alpha / max_i|W_ij|^(1-alpha)  */
/* ------------------------------------------------------------------ */

void oracle_smooth_scales(const float *s, const float *W, int64_t N, int64_t K,
                          float alpha, float *lambda)
{
    for (int64_t j = 0; j < K; ++j) {
        float m = 0.0f;                       /* column absmax over output rows */
        for (int64_t i = 0; i < N; ++i) {
            float a = fabsf(W[i * K + j]);
            if (a > m)
                m = a;
        }
        float sj = s[j];
        float l;
        if (sj == 0.0f || m == 0.0f)
            l = 1.0f;
        else if (alpha == 0.5f)
            l = sqrtf(sj) / sqrtf(m);         /* s^(1/2) / m^(1/2), each RN */
        else if (alpha == 1.0f)
            l = sj;                           /* s^1 / m^0 */
        else if (alpha == 0.0f)
            l = 1.0f / m;                     /* s^0 / m^1 */
        else
            l = (float)exp2((double)alpha * log2((double)sj) -
                            (1.0 - (double)alpha) * log2((double)m));
        lambda[j] = l;
    }
}

/* ------------------------------------------------------------------ */
/* a2: per-output-channel symmetric INT8 weights of W' = W diag(lambda) */
/* ------------------------------------------------------------------ */

void oracle_quantize_weights(const float *W, const float *lambda, int64_t N,
                             int64_t K, int8_t *Wq, float *w_scale)
{
    for (int64_t i = 0; i < N; ++i) {
        const float *row = W + i * K;
        float a = 0.0f;
        for (int64_t j = 0; j < K; ++j) {
            float w = lambda ? row[j] * lambda[j] : row[j];
            float aw = fabsf(w);
            if (aw > a)
                a = aw;
        }
        int8_t *q = Wq + i * K;
        if (a == 0.0f) {
            w_scale[i] = 0.0f;
            memset(q, 0, (size_t)K);
            continue;
        }
        w_scale[i] = a / 127.0f;
        float inv = 127.0f / a;
        for (int64_t j = 0; j < K; ++j) {
            float w = lambda ? row[j] * lambda[j] : row[j];
            q[j] = quantize_rne_clamp(w * inv);
        }
    }
}

/* ------------------------------------------------------------------ */
/* a3: per-token dynamic INT8 activations of X' = X diag(lambda)^-1     */
/* ------------------------------------------------------------------ */

void oracle_quant_act(const uint16_t *X, const float *lambda, int64_t M,
                      int64_t K, int8_t *Xq, float *x_scale, float *recip_tmp)
{
    /* r_j = 1 / lambda_j, rounded once; recip_tmp is caller storage of K floats */
    for (int64_t j = 0; j < K; ++j)
        recip_tmp[j] = lambda ? 1.0f / lambda[j] : 1.0f;

    for (int64_t t = 0; t < M; ++t) {
        const uint16_t *row = X + t * K;
        float a = 0.0f;
        for (int64_t j = 0; j < K; ++j) {
            float x = oracle_bf16_to_f32(row[j]) * recip_tmp[j];
            float ax = fabsf(x);
            if (ax > a)
                a = ax;
        }
        int8_t *q = Xq + t * K;
        if (a == 0.0f) {
            x_scale[t] = 0.0f;
            memset(q, 0, (size_t)K);
            continue;
        }
        x_scale[t] = a / 127.0f;
        float inv = 127.0f / a;
        for (int64_t j = 0; j < K; ++j) {
            float x = oracle_bf16_to_f32(row[j]) * recip_tmp[j];
            q[j] = quantize_rne_clamp(x * inv);
        }
    }
}

/* ------------------------------------------------------------------ */
/* a4: exact integer product acc = Xq Wq^T over rows [m0, m1)           */
/* ------------------------------------------------------------------ */

void oracle_gemm_i32(const int8_t *Xq, const int8_t *Wq, int64_t M, int64_t N,
                     int64_t K, int64_t m0, int64_t m1, int32_t *acc)
{
    (void)M;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t m = m0; m < m1; ++m) {
        const int8_t *x = Xq + m * K;
        for (int64_t n = 0; n < N; ++n) {
            const int8_t *w = Wq + n * K;
            int64_t sum = 0;
            for (int64_t k = 0; k < K; ++k)
                sum += (int64_t)x[k] * (int64_t)w[k];
            acc[(m - m0) * N + n] = (int32_t)sum;
        }
    }
}

/* ------------------------------------------------------------------ */
/* a5: dequantizing epilogue, y = bf16_rne(((float)acc * sx) * sw + b)  */
/* ------------------------------------------------------------------ */

uint16_t oracle_epilogue_value(int32_t acc, float sx, float sw, const float *b)
{
    float t = (float)acc;
    t = t * sx;
    t = t * sw;
    if (b)
        t = t + *b;
    return oracle_f32_to_bf16_rne(t);
}

void oracle_epilogue(const int32_t *acc, const float *x_scale,
                     const float *w_scale, const float *bias, int64_t rows,
                     int64_t N, uint16_t *Y)
{
    for (int64_t m = 0; m < rows; ++m)
        for (int64_t n = 0; n < N; ++n)
            Y[m * N + n] = oracle_epilogue_value(acc[m * N + n], x_scale[m],
                                                 w_scale[n],
                                                 bias ? bias + n : 0);
}

/* a4 + a5 for the rows [m0, m1); Y holds (m1 - m0) rows; acc_tmp is caller
 * storage of (m1 - m0) * N int32. */
void oracle_linear_rows(const int8_t *Xq, const float *x_scale,
                        const int8_t *Wq, const float *w_scale,
                        const float *bias, int64_t M, int64_t N, int64_t K,
                        int64_t m0, int64_t m1, int32_t *acc_tmp, uint16_t *Y)
{
    oracle_gemm_i32(Xq, Wq, M, N, K, m0, m1, acc_tmp);
    oracle_epilogue(acc_tmp, x_scale + m0, w_scale, bias, m1 - m0, N, Y);
}

/* ------------------------------------------------------------------ */
/* ablation arm: one activation scale for the whole tensor             */
/* (the "naive per-tensor INT8 activations" that SmoothQuant is        */
/* contrasted with, Sec. 2 "Weight-activation PTQ"; the naive W8A8     */
/* arm of the activation-quant ablation, Sec. 5 "What drives INT8      */
/* recovery").  Same steps as oracle_quant_act with the max taken      */
/* over every element of X diag(lambda)^-1 instead of one row; the     */
/* common scale is written to every row's x_scale so that the same     */
/* epilogue applies.                                                    */
/* ------------------------------------------------------------------ */

void oracle_quant_act_per_tensor(const uint16_t *X, const float *lambda,
                                 int64_t M, int64_t K, int8_t *Xq,
                                 float *x_scale, float *amax_out,
                                 float *recip_tmp)
{
    for (int64_t j = 0; j < K; ++j)
        recip_tmp[j] = lambda ? 1.0f / lambda[j] : 1.0f;

    float a = 0.0f;                           /* max over the whole tensor */
    for (int64_t t = 0; t < M; ++t)
        for (int64_t j = 0; j < K; ++j) {
            float ax = fabsf(oracle_bf16_to_f32(X[t * K + j]) * recip_tmp[j]);
            if (ax > a)
                a = ax;
        }
    *amax_out = a;
    float scale = (a == 0.0f) ? 0.0f : a / 127.0f;
    float inv = (a == 0.0f) ? 0.0f : 127.0f / a;
    for (int64_t t = 0; t < M; ++t) {
        x_scale[t] = scale;
        for (int64_t j = 0; j < K; ++j) {
            if (a == 0.0f) {
                Xq[t * K + j] = 0;
                continue;
            }
            float x = oracle_bf16_to_f32(X[t * K + j]) * recip_tmp[j];
            Xq[t * K + j] = quantize_rne_clamp(x * inv);
        }
    }
}

/* threads the row loop of oracle_gemm_i32 runs on (1 without OpenMP) */
int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
