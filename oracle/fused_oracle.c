/*
 * fused_oracle.c -- plain, slow CPU oracle of the activation quantization
 * fused with the FFN's GELU.
 *
 * TEST INFRASTRUCTURE ONLY, like w8a8_oracle.c: only the test-suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it; it shares no
 * code with the CUDA library.
 *
 * The FFN down-projections are the most fragile linears of the model
 * (Sec. 3, "Activation-fragility profiling and protection"); their input is
 * the activation of the up-projection's output.  The paper does not name the
 * activation function; the reading taken here is the exact (erf) GELU,
 *     GELU(h) = h * Phi(h) = (h / 2) * erfc(-h / sqrt(2)),
 * evaluated in binary64 and rounded once to binary32, and the fused pass
 * quantizes that fp32 value directly (no bf16 rounding in between):
 *     g_mj = fl32(GELU(H_mj));  x'_mj = g_mj * (1/lambda_j)   (fp32, RN)
 *     a_m = max_j |x'_mj|;  x_scale_m = a_m / 127;
 *     Xq_mj = clamp(rne(x'_mj * (127 / a_m)), +-127)
 * i.e. the per-token quantization of Sec. 3 ("INT8 W8A8") applied to GELU(H).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static float h_value(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

static int8_t rne_clamp(float v)
{
    if (v != v)
        return 0;
    float r = rintf(v);
    if (r > 127.0f)
        r = 127.0f;
    if (r < -127.0f)
        r = -127.0f;
    return (int8_t)r;
}

/* GELU(h) = (h/2) erfc(-h/sqrt(2)) in binary64, rounded once to binary32 */
float oracle_gelu_value(float h)
{
    double x = (double)h;
    return (float)(0.5 * x * erfc(-x / sqrt(2.0)));
}

/* pre (optional, [M,K]): the fp32 value x'_mj * (127 / a_m) that is rounded
 * to the code, for tests that need to know how close it was to a tie. */
void oracle_gelu_quant_act(const uint16_t *H, const float *lambda, int64_t M,
                           int64_t K, int8_t *Xq, float *x_scale,
                           float *recip_tmp, float *row_tmp, float *pre)
{
    for (int64_t j = 0; j < K; ++j)
        recip_tmp[j] = lambda ? 1.0f / lambda[j] : 1.0f;
    for (int64_t t = 0; t < M; ++t) {
        float a = 0.0f;
        for (int64_t j = 0; j < K; ++j) {
            float x = oracle_gelu_value(h_value(H[t * K + j])) * recip_tmp[j];
            row_tmp[j] = x;
            if (fabsf(x) > a)
                a = fabsf(x);
        }
        int8_t *q = Xq + t * K;
        if (a == 0.0f) {
            x_scale[t] = 0.0f;
            memset(q, 0, (size_t)K);
            if (pre)
                for (int64_t j = 0; j < K; ++j)
                    pre[t * K + j] = 0.0f;
            continue;
        }
        x_scale[t] = a / 127.0f;
        float inv = 127.0f / a;
        for (int64_t j = 0; j < K; ++j) {
            float v = row_tmp[j] * inv;
            q[j] = rne_clamp(v);
            if (pre)
                pre[t * K + j] = v;
        }
    }
}
