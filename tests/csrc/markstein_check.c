/*
 * Exhaustive check of the activation quantizer's quotient (test code, not
 * part of the library).  The kernels form q = a / s for every fp16 input a
 * with one correction step of Markstein's method on r = RN(1 / s):
 *     q0 = RN(a * r),  q = RN(fma(RN(fma(-q0, s, a)), r, q0))
 * and claim it equals the correctly rounded IEEE quotient RN(a / s) whenever
 * s lies in [2^-60, 2^60] (outside that range the kernels divide).  This
 * program compares the two for every finite fp16 value a (both signs) against
 * every positive finite fp16 scale and a set of seeded random fp32 scales
 * spread over [2^-60, 2^60], and prints the number of mismatches (values
 * compared with ==, so the sign of a zero quotient is not counted: both zeros
 * quantize to code 0).  Under a calibrated scale the kernels clip an input
 * above s to s before the quotient, so for every scale it also checks that
 * the corrected quotient of s itself is exactly 1.
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math markstein_check.c -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

static float half_to_float(uint16_t h) {
    uint32_t sign = (uint32_t)(h >> 15) << 31, e = (h >> 10) & 31u, m = h & 1023u, bits;
    if (e == 0) {
        float v = ldexpf((float)m, -24);
        return sign ? -v : v;
    }
    bits = sign | ((e + 112u) << 23) | (m << 13);
    float f;
    memcpy(&f, &bits, 4);
    return f;
}

static uint64_t state = 0x9E3779B97F4A7C15ull;
static uint64_t next_u64(void) { /* splitmix64 */
    uint64_t z = (state += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static long check_scale(float s, const float *a, int na) {
    long bad = 0;
    const float r = 1.0f / s;
    for (int i = 0; i < na; ++i) {
        const float q0 = a[i] * r;
        const float q = fmaf(fmaf(-q0, s, a[i]), r, q0);
        const float ref = a[i] / s;
        /* equal values (a zero quotient may differ in sign only: -0 / s is -0,
           the corrected quotient +0; both give code 0) */
        if (!(q == ref)) ++bad;
    }
    {   /* the clipped input a = s */
        const float q0 = s * r;
        if (!(fmaf(fmaf(-q0, s, s), r, q0) == 1.0f)) ++bad;
    }
    return bad;
}

int main(int argc, char **argv) {
    int n_random = argc > 1 ? atoi(argv[1]) : 20000;
    static float a[65536];
    int na = 0;
    for (uint32_t h = 0; h < 65536; ++h)
        if (((h >> 10) & 31u) != 31u) a[na++] = half_to_float((uint16_t)h);
    long bad = 0, scales = 0;
    for (uint32_t h = 1; h < 0x7C00u; ++h) {   /* every positive finite fp16 scale */
        bad += check_scale(half_to_float((uint16_t)h), a, na);
        ++scales;
    }
    for (int k = 0; k < n_random; ++k) {        /* random fp32 scales in [2^-60, 2^60] */
        const uint64_t u = next_u64();
        const int e = (int)(u % 121) - 60;
        const uint32_t mant = (uint32_t)(u >> 32) & 0x7FFFFFu;
        uint32_t bits = ((uint32_t)(e + 127) << 23) | mant;
        float s;
        memcpy(&s, &bits, 4);
        if (s < 0x1p-60f || s > 0x1p60f) continue;
        bad += check_scale(s, a, na);
        ++scales;
    }
    printf("%ld %ld %d\n", bad, scales, na);
    return 0;
}
