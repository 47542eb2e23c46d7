/*
 * gguf_oracle.c -- plain, slow CPU oracle of the GGUF weight-only formats
 * the paper serializes its DiT to (Sec. 3, "GGUF k-quants": Q8_0 at 8.5 bits
 * per weight, round to nearest; Q4_K at 4.5 bits per weight), decoded for a
 * linear layer with bf16 activations.
 *
 * TEST INFRASTRUCTURE ONLY, like w8a8_oracle.c: only the test-suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it; it shares no
 * code with the CUDA library.
 *
 * Block layouts (the public GGUF/ggml formats; little-endian):
 *   Q8_0, 32 weights in 34 bytes: fp16 d, then 32 int8 q;  w_i = d * q_i.
 *   Q4_K, 256 weights in 144 bytes: fp16 d, fp16 dmin, 12 bytes holding eight
 *     6-bit scales sc_j and eight 6-bit mins m_j, then 128 bytes of 4-bit
 *     quants.  For j < 4: sc_j = s[j] & 63, m_j = s[j+4] & 63; for j >= 4:
 *     sc_j = (s[j+4] & 15) | ((s[j-4] >> 6) << 4),
 *     m_j  = (s[j+4] >> 4) | ((s[j] >> 6) << 4).
 *     Weights 64c .. 64c+31 are the low nibbles of quant bytes 32c .. 32c+31
 *     (sub-block j = 2c), weights 64c+32 .. 64c+63 their high nibbles
 *     (j = 2c+1); w = (d * sc_j) * q - dmin * m_j.
 * A row of a weight matrix [N, K] is K/32 (Q8_0) or K/256 (Q4_K) consecutive
 * blocks.
 *
 * Readings (the paper is silent): the decode runs in binary32 as written
 * above (every product of these small integers and an fp16 value is exact, so
 * only the final subtraction of Q4_K rounds), and the layer consumes the
 * decoded weight rounded to bf16 (round to nearest even), its compute dtype.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* IEEE binary16 -> binary32, exact (normal, subnormal, zero, inf, NaN) */
float oracle_f16_to_f32(uint16_t h)
{
    uint32_t sign = (uint32_t)(h >> 15) << 31;
    int exp = (h >> 10) & 31;
    uint32_t man = h & 1023;
    float f;
    if (exp == 31) {
        uint32_t u = sign | 0x7f800000u | (man << 13);
        memcpy(&f, &u, sizeof f);
        return f;
    }
    if (exp == 0) {                 /* zero or subnormal: man * 2^-24 */
        f = (float)man * 5.9604644775390625e-08f;
        return sign ? -f : f;
    }
    uint32_t u = sign | ((uint32_t)(exp - 15 + 127) << 23) | (man << 13);
    memcpy(&f, &u, sizeof f);
    return f;
}

static uint16_t rd16(const uint8_t *p) { return (uint16_t)(p[0] | (p[1] << 8)); }

/* raw: N rows of K/32 blocks; out [N, K] fp32 */
void oracle_dequant_q8_0(const uint8_t *raw, int64_t N, int64_t K, float *out)
{
    const int64_t nb = K / 32;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t b = 0; b < nb; ++b) {
            const uint8_t *blk = raw + (n * nb + b) * 34;
            float d = oracle_f16_to_f32(rd16(blk));
            for (int i = 0; i < 32; ++i)
                out[n * K + b * 32 + i] = d * (float)(int8_t)blk[2 + i];
        }
}

static void q4k_scale_min(const uint8_t *s, int j, int *sc, int *m)
{
    if (j < 4) {
        *sc = s[j] & 63;
        *m = s[j + 4] & 63;
    } else {
        *sc = (s[j + 4] & 15) | ((s[j - 4] >> 6) << 4);
        *m = (s[j + 4] >> 4) | ((s[j] >> 6) << 4);
    }
}

/* raw: N rows of K/256 blocks; out [N, K] fp32 */
void oracle_dequant_q4_k(const uint8_t *raw, int64_t N, int64_t K, float *out)
{
    const int64_t nb = K / 256;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t b = 0; b < nb; ++b) {
            const uint8_t *blk = raw + (n * nb + b) * 144;
            float d = oracle_f16_to_f32(rd16(blk));
            float dmin = oracle_f16_to_f32(rd16(blk + 2));
            const uint8_t *sc = blk + 4;
            const uint8_t *qs = blk + 16;
            float *o = out + n * K + b * 256;
            for (int c = 0; c < 4; ++c) {
                int s0, m0, s1, m1;
                q4k_scale_min(sc, 2 * c, &s0, &m0);
                q4k_scale_min(sc, 2 * c + 1, &s1, &m1);
                float d0 = d * (float)s0, mm0 = dmin * (float)m0;
                float d1 = d * (float)s1, mm1 = dmin * (float)m1;
                for (int l = 0; l < 32; ++l) {
                    o[64 * c + l] = d0 * (float)(qs[32 * c + l] & 15) - mm0;
                    o[64 * c + 32 + l] = d1 * (float)(qs[32 * c + l] >> 4) - mm1;
                }
            }
        }
}
