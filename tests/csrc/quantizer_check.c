/*
 * CPU check of the kernels' quantizer formulas (test code, not part of the
 * library), restated in C and compared with the oracle's code functions:
 *
 *  1. Activation codes on the Markstein path with the top clip taken on the
 *     input (tiled, one-pass and epilogue kernels):
 *         x = min_keep_nan(a, s); q0 = RN(x * r); q = fma(fma(-q0, s, x), r, q0);
 *         u = cvt_rni_u32(RN(q * L))     (saturating; NaN -> 0)
 *  2. The gather kernel's calibrated variant of the same:
 *         u = low byte of RN(max(RN(q * L), 0) + 1.5 * 2^23)
 *  3. Weight codes of the pack kernel: the estimate y = RN(w * RN(RN(1/s) * 2^(n-1)))
 *     used while that product is finite and y lies more than 8 ulps of 128 from a
 *     half-integer, the IEEE rule otherwise; integer clip after a saturating
 *     conversion (NaN -> 0).
 *
 * Inputs: every fp16 pattern (NaNs as the quiet NaNs the GPU's fp16 -> fp32
 * conversion gives) against activation scales across [2^-60, 2^60] for every
 * width 1..8; weights on a grid of multiples of the scale, plus seeded random
 * fp32 values, for scales from the smallest fp32 subnormal to FLT_MAX.
 * Prints the mismatch counts of the three formulas and the number of cases.
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math quantizer_check.c <oracle>.c -lm
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

int32_t orc_act_code(float a, float s, int32_t n);
int32_t orc_weight_code(float w, float s, int32_t n);

static float bits_f(uint32_t b) {
    float f;
    memcpy(&f, &b, 4);
    return f;
}

static float half_to_float(uint16_t h) {
    uint32_t sign = (uint32_t)(h >> 15) << 31, e = (h >> 10) & 31u, m = h & 1023u;
    if (e == 0) {
        float v = ldexpf((float)m, -24);
        return sign ? -v : v;
    }
    if (e == 31) return bits_f(sign | 0x7F800000u | (m << 13) | (m ? 0x400000u : 0u));
    return bits_f(sign | ((e + 112u) << 23) | (m << 13));
}

static float min_keep_nan(float x, float s) { return isnan(x) ? x : (x < s ? x : s); }

static uint32_t cvt_rni_u32(float t) {
    if (isnan(t)) return 0u;
    const float r = rintf(t);
    if (r <= 0.0f) return 0u;
    if (r >= 4294967295.0f) return 4294967295u;
    return (uint32_t)r;
}

static int32_t cvt_rni_s32(float t) {
    if (isnan(t)) return 0;
    const float r = rintf(t);
    if (r <= -2147483648.0f) return INT32_MIN;
    if (r >= 2147483647.0f) return INT32_MAX;
    return (int32_t)r;
}

static int32_t cvt_rzi_s32(float t) {
    if (isnan(t)) return 0;
    if (t <= -2147483648.0f) return INT32_MIN;
    if (t >= 2147483647.0f) return INT32_MAX;
    return (int32_t)t;
}

static float markstein(float x, float s, float r) {
    const float q0 = x * r;
    return fmaf(fmaf(-q0, s, x), r, q0);
}

static uint32_t act_clip_input(float a, float s, float r, float levels) {
    return cvt_rni_u32(markstein(min_keep_nan(a, s), s, r) * levels);
}

static uint32_t act_gather_calibrated(float a, float s, float r, float levels) {
    const float u = fmaxf(markstein(min_keep_nan(a, s), s, r) * levels, 0.0f);
    const float b = u + 12582912.0f;
    uint32_t bits;
    memcpy(&bits, &b, 4);
    return bits & 0xFFu;
}

static int32_t clip_i(int32_t v, int32_t lo, int32_t hi) { return v < lo ? lo : (v > hi ? hi : v); }

static int32_t weight_ieee(float w, float s, float half) {
    const int32_t h = (int32_t)half;
    return clip_i(cvt_rni_s32((w / s) * half), -h, h - 1);
}

static int32_t weight_pack(float w, float s, int n) {
    if (!(s > 0.0f)) return 0;
    const float half = (float)(1 << (n - 1));
    const float rh = (1.0f / s) * half;
    const int est = rh <= FLT_MAX;
    const float y = w * rh, k = rintf(y);
    const int32_t h = 1 << (n - 1);
    if (!est || fabsf(fabsf(y - k) - 0.5f) <= 8.0f * 0x1p-16f) return weight_ieee(w, s, half);
    return clip_i(cvt_rzi_s32(k), -h, h - 1);
}

static uint64_t state = 0x2545F4914F6CDD1Dull;
static uint64_t next_u64(void) { /* splitmix64 */
    uint64_t z = (state += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

int main(void) {
    const float act_scales[] = {0x1p-60f, 1e-7f, 6.1e-5f, 0.37f, 0.9f, 1.0f, 1.7f, 2.5f, 3.14159f,
                                255.0f, 65504.0f, 7e4f, 1e9f, 0x1p60f};
    const float w_scales[] = {1.4e-45f, 1e-42f, 1e-40f, 2.9e-39f, 3e-39f, 1e-38f, 1.2e-38f, 1e-37f, 3.7e-37f,
                              3.9e-37f, 1e-36f, 1e-30f, 1e-3f, 1.0f, 0.02f, 1e30f, 8.6e37f, 3e38f, FLT_MAX};
    long bad_act = 0, bad_gather = 0, bad_w = 0, cases = 0;
    for (unsigned i = 0; i < sizeof act_scales / sizeof act_scales[0]; ++i) {
        const float s = act_scales[i], r = 1.0f / s;
        for (int n = 1; n <= 8; ++n) {
            const float levels = (float)((1 << n) - 1);
            for (uint32_t h = 0; h < 65536; ++h) {
                const float a = half_to_float((uint16_t)h);
                const int32_t ref = orc_act_code(a, s, n);
                bad_act += (int32_t)act_clip_input(a, s, r, levels) != ref;
                bad_gather += (int32_t)act_gather_calibrated(a, s, r, levels) != ref;
                ++cases;
            }
        }
    }
    for (unsigned i = 0; i < sizeof w_scales / sizeof w_scales[0]; ++i) {
        const float s = w_scales[i];
        for (int n = 1; n <= 8; ++n) {
            for (int k = -2048; k <= 2048; ++k) {   /* multiples of s / 2048: every half-level tie */
                const float w = s * ((float)k / 2048.0f);
                bad_w += weight_pack(w, s, n) != orc_weight_code(w, s, n);
                ++cases;
            }
            for (int k = 0; k < 4096; ++k) {        /* random values in [-s, s] */
                const float u = (float)((double)(next_u64() >> 11) * 0x1p-53) * 2.0f - 1.0f;
                const float w = s * u;
                bad_w += weight_pack(w, s, n) != orc_weight_code(w, s, n);
                ++cases;
            }
            const float specials[] = {NAN, INFINITY, -INFINITY, s, -s, 0.0f, -0.0f};
            for (unsigned j = 0; j < sizeof specials / sizeof specials[0]; ++j) {
                bad_w += weight_pack(specials[j], s, n) != orc_weight_code(specials[j], s, n);
                ++cases;
            }
        }
    }
    printf("%ld %ld %ld %ld\n", bad_act, bad_gather, bad_w, cases);
    return 0;
}
