/*
 * protect_oracle.c -- plain, slow CPU oracle of the fragility-protection
 * pieces around the W8A8 layer.
 *
 * TEST INFRASTRUCTURE ONLY, like w8a8_oracle.c: only the test-suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it; it shares no
 * code with the CUDA library.
 *
 * Sec. 3, "Activation-fragility profiling and protection": every linear's
 * input activation is recorded over the denoising trajectory as max-abs,
 * standard deviation and kurtosis; the N most fragile layers keep bf16 weights
 * and skip activation quantization, the others run W8A8.  This file holds
 *
 *   oracle_act_stats            the statistics, from their definitions, in
 *                               binary64 (two passes: mean, then central
 *                               moments), per input channel and for the whole
 *                               tensor;
 *   oracle_shifted_power_sums   sum_t (x_tj - c_j)^p for p = 1..4 in binary64,
 *                               the accumulator form a streaming pass keeps;
 *   oracle_linear_bf16_rows     the protected (unquantized) layer: the exact
 *                               value sum_k x_mk w_nk + b_n of bf16 operands,
 *                               accumulated in binary64 (every product of two
 *                               bf16 values is exact in binary64).
 *
 * Readings where the paper is silent (each listed in the design notes):
 *   - the statistics run over all recorded tokens pooled (rows of X), per
 *     input channel j, and over every element for the layer-level value;
 *   - standard deviation is the population one (divide by the count);
 *   - kurtosis is Pearson's m4 / m2^2 (3 for a normal distribution), and 0
 *     when the variance is 0;
 *   - the protected layer's result is that exact value rounded once to bf16.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static double bf16_value(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* mean, population std and Pearson kurtosis of n values given by a strided
 * walk; out = {maxabs, mean, std, kurtosis} */
static void moments_of(const uint16_t *X, int64_t count, int64_t stride,
                       int64_t offset, double out[4])
{
    double maxabs = 0.0, sum = 0.0;
    for (int64_t i = 0; i < count; ++i) {
        double x = bf16_value(X[offset + i * stride]);
        if (fabs(x) > maxabs)
            maxabs = fabs(x);
        sum += x;
    }
    double mean = sum / (double)count;
    double m2 = 0.0, m4 = 0.0;
    for (int64_t i = 0; i < count; ++i) {
        double d = bf16_value(X[offset + i * stride]) - mean;
        m2 += d * d;
        m4 += d * d * d * d;
    }
    m2 /= (double)count;
    m4 /= (double)count;
    out[0] = maxabs;
    out[1] = mean;
    out[2] = sqrt(m2);
    out[3] = (m2 > 0.0) ? m4 / (m2 * m2) : 0.0;
}

/* chan: 4 planes of K = maxabs, mean, std, kurtosis per input channel;
 * tensor: the same four over all T*K elements.  T >= 1. */
void oracle_act_stats(const uint16_t *X, int64_t T, int64_t K, double *chan,
                      double *tensor)
{
    for (int64_t j = 0; j < K; ++j) {
        double o[4];
        moments_of(X, T, K, j, o);
        for (int p = 0; p < 4; ++p)
            chan[p * K + j] = o[p];
    }
    moments_of(X, T * K, 1, 0, tensor);
}

/* S: 4 planes of K, S[(p-1)*K + j] = sum_t (x_tj - c_j)^p, c = shift or 0;
 * also A: 4 planes of K with sum_t |x_tj - c_j|^p (the size of each sum's
 * terms, for rounding-error bounds). */
void oracle_shifted_power_sums(const uint16_t *X, int64_t T, int64_t K,
                               const float *shift, double *S, double *A)
{
    for (int64_t j = 0; j < K; ++j) {
        double c = shift ? (double)shift[j] : 0.0;
        double s[4] = {0, 0, 0, 0}, a[4] = {0, 0, 0, 0};
        for (int64_t t = 0; t < T; ++t) {
            double d = bf16_value(X[t * K + j]) - c;
            double pw = 1.0;
            for (int p = 0; p < 4; ++p) {
                pw *= d;
                s[p] += pw;
                a[p] += fabs(pw);
            }
        }
        for (int p = 0; p < 4; ++p) {
            S[p * K + j] = s[p];
            if (A)
                A[p * K + j] = a[p];
        }
    }
}

/* rows [m0, m1) of y = X W^T + b with X [M, K] and W [N, K] bf16, b [N] fp32
 * or NULL: Y[(m - m0) * N + n] = sum_k x_mk w_nk + b_n in binary64, and
 * Yabs (or NULL) = sum_k |x_mk w_nk| + |b_n| (the size of the terms). */
void oracle_linear_bf16_rows(const uint16_t *X, const uint16_t *W,
                             const float *bias, int64_t M, int64_t N,
                             int64_t K, int64_t m0, int64_t m1, double *Y,
                             double *Yabs)
{
    (void)M;
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t m = m0; m < m1; ++m) {
        for (int64_t n = 0; n < N; ++n) {
            double y = 0.0, ya = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double p = bf16_value(X[m * K + k]) * bf16_value(W[n * K + k]);
                y += p;
                ya += fabs(p);
            }
            if (bias) {
                y += (double)bias[n];
                ya += fabs((double)bias[n]);
            }
            Y[(m - m0) * N + n] = y;
            if (Yabs)
                Yabs[(m - m0) * N + n] = ya;
        }
    }
}
