/*
 * soniq_oracle.c -- plain, slow CPU oracle for SONIQ's inference hot path
 * (arXiv 2311.14114): per-channel two-level mixed-precision quantization of
 * activations and weights, channel permutation and padding, exact integer
 * dot products per precision group, and the scale epilogue.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load this file.  It shares no code, header,
 * table or helper with the CUDA library; neither includes the other.
 *
 * Precision: a quantized code is an integer decided by floating point, so it
 * is decided here in fp32 with the operation order of the paper's formulas
 * (divide by the scale, then multiply by the level count), IEEE round to
 * nearest even, no contraction (build with -ffp-contract=off).  Integer dot
 * products are exact int64.  The epilogue is fp64.
 *
 * Conventions (one precision group per contiguous run of packed channels):
 *   K            logical channels (conv: input channels C)
 *   count[g]     channels in group g; group 0 holds the low precision
 *   perm[j]      original channel stored at packed position j; positions
 *                [0,count[0]) form group 0 and [count[0],K) group 1
 *   PA_g         activation codes per row and group  = roundup(count[g], pad)
 *   PW_g(taps)   weight codes per row and group      = roundup(taps*PA_g, 128)
 *                (weight K order inside a group: tap-major, then channel)
 *
 * Packed block layout (the library's storage format for codes, chosen so a
 * SIMD-in-register expansion restores natural code order; the paper leaves
 * the bit layout open and only asks for contiguous, padded, uniform-precision
 * blocks, Fig. 2 and Sec. 4.1 "Channel re-ordering and padding"):
 *   32 consecutive codes of one group form a block of n 32-bit little-endian
 *   words (4n bytes).  The n bits of a code are cut into slices of width 4,
 *   2, 1 (in that order, least-significant bits first; n = 8 is one slice of
 *   width 8).  A slice of width w takes w words; code i (t = i/4, b = i%4)
 *   sits in slice word t/(8/w) at bit 8*b + w*(t%(8/w)).
 *
 * Parity pins for every function live in tests/test_oracle_*.py.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_GROUPS 2

static int64_t roundup64(int64_t x, int64_t u) { return (x + u - 1) / u * u; }

/* ------------------------------------------------------------------------- */
/* Layout sizes                                                              */
/* ------------------------------------------------------------------------- */

int64_t orc_act_group_codes(int32_t count, int32_t pad_unit) {
    return roundup64(count, pad_unit);
}

int64_t orc_weight_group_codes(int32_t count, int32_t pad_unit, int32_t taps) {
    return roundup64((int64_t)taps * roundup64(count, pad_unit), 128);
}

/* Bytes of one packed row: activation rows (is_weight = 0, taps ignored) or
 * weight rows (is_weight = 1). */
int64_t orc_row_bytes(const int32_t count[2], const int32_t bits[2], int32_t pad_unit,
                      int32_t taps, int32_t is_weight) {
    int64_t bytes = 0;
    for (int g = 0; g < ORC_GROUPS; ++g) {
        int64_t codes = is_weight ? orc_weight_group_codes(count[g], pad_unit, taps)
                                  : orc_act_group_codes(count[g], pad_unit);
        bytes += codes / 32 * 4 * bits[g];
    }
    return bytes;
}

/* ------------------------------------------------------------------------- */
/* a1  Group-wise scale selection, Sec. 3 "Enabling Low-Cost Fixed-Point     */
/*     Operations", step 1: s_g = max over the group of |x|.                 */
/* ------------------------------------------------------------------------- */

/* Activations A[M][K] (fp16 values held in fp32).  per_row = 0: one scale per
 * (tensor, group) -> s[2]; per_row = 1: one scale per (row, group) -> s[M][2]. */
void orc_act_scales(const float *A, int64_t M, int32_t K, const int32_t *perm,
                    const int32_t count[2], int32_t per_row, float *s) {
    int32_t base[2] = {0, count[0]};
    if (!per_row) { s[0] = 0.0f; s[1] = 0.0f; }
    for (int64_t m = 0; m < M; ++m) {
        for (int g = 0; g < ORC_GROUPS; ++g) {
            float mx = per_row ? 0.0f : s[g];
            for (int32_t j = 0; j < count[g]; ++j) {
                float v = fabsf(A[m * K + perm[base[g] + j]]);
                if (v > mx) mx = v;
            }
            if (per_row) s[m * 2 + g] = mx; else s[g] = mx;
        }
    }
}

/* Weights W[N][taps][K].  per_row = 1: one scale per (output row n, group),
 * taken over all taps of the group's channels; per_row = 0: one scale per
 * group over the whole tensor.  Output s[N][2] (per-tensor values repeated). */
void orc_weight_scales(const float *W, int32_t N, int32_t taps, int32_t K,
                       const int32_t *perm, const int32_t count[2], int32_t per_row,
                       float *s) {
    int32_t base[2] = {0, count[0]};
    float tensor_max[2] = {0.0f, 0.0f};
    for (int32_t n = 0; n < N; ++n) {
        for (int g = 0; g < ORC_GROUPS; ++g) {
            float mx = 0.0f;
            for (int32_t t = 0; t < taps; ++t)
                for (int32_t j = 0; j < count[g]; ++j) {
                    float v = fabsf(W[((int64_t)n * taps + t) * K + perm[base[g] + j]]);
                    if (v > mx) mx = v;
                }
            s[n * 2 + g] = mx;
            if (mx > tensor_max[g]) tensor_max[g] = mx;
        }
    }
    if (!per_row)
        for (int32_t n = 0; n < N; ++n) { s[n * 2 + 0] = tensor_max[0]; s[n * 2 + 1] = tensor_max[1]; }
}

/* ------------------------------------------------------------------------- */
/* a3a Unsigned activation code, Sec. 3 step 2:                              */
/*     b = clip(round(a / s_g * (2^n - 1)), 0, 2^n - 1)                      */
/* A zero scale (all-zero group) gives code 0.  Non-finite inputs: the clip  */
/* takes +inf to 2^n - 1 and -inf to 0; a NaN quotient (a NaN input, or      */
/* inf / inf) lies on neither side of the clip and is read as code 0.        */
/* ------------------------------------------------------------------------- */
int32_t orc_act_code(float a, float s, int32_t n) {
    if (!(s > 0.0f)) return 0;
    float levels = (float)((1 << n) - 1);
    float q = a / s;           /* fp32, IEEE division */
    float t = q * levels;      /* fp32 multiply, no fused op */
    float r = rintf(t);        /* round half to even */
    if (isnan(r)) return 0;
    if (r < 0.0f) r = 0.0f;
    if (r > levels) r = levels;
    return (int32_t)r;
}

/* ------------------------------------------------------------------------- */
/* a3b Signed weight code, Sec. 3 step 3 and Eq. (1): the nearest n-bit      */
/*     two's-complement fraction q = j / 2^(n-1), j in [-2^(n-1), 2^(n-1)-1], */
/*     to w' = w / s_g (ties to even j).  Multiplying w' by 2^(n-1) is exact.*/
/*     Non-finite inputs as for activations: +-inf clip to the end levels, a  */
/*     NaN quotient is read as code 0.                                        */
/* ------------------------------------------------------------------------- */
int32_t orc_weight_code(float w, float s, int32_t n) {
    if (!(s > 0.0f)) return 0;
    float half_range = (float)(1 << (n - 1));
    float wp = w / s;
    float t = wp * half_range;
    float r = rintf(t);
    if (isnan(r)) return 0;
    if (r < -half_range) r = -half_range;
    if (r > half_range - 1.0f) r = half_range - 1.0f;
    return (int32_t)r;
}

/* Activation codes for rows A[M][K]; U[M][K] in packed channel order. */
void orc_act_codes(const float *A, int64_t M, int32_t K, const int32_t *perm,
                   const int32_t count[2], const int32_t bits[2], const float *s,
                   int32_t per_row, uint8_t *U) {
    int32_t base[2] = {0, count[0]};
    for (int64_t m = 0; m < M; ++m)
        for (int g = 0; g < ORC_GROUPS; ++g) {
            float sg = per_row ? s[m * 2 + g] : s[g];
            for (int32_t j = 0; j < count[g]; ++j) {
                int32_t p = base[g] + j;
                U[m * K + p] = (uint8_t)orc_act_code(A[m * K + perm[p]], sg, bits[g]);
            }
        }
}

/* Weight codes for W[N][taps][K] with scales s[N][2]; J[N][taps][K] in packed
 * channel order. */
void orc_weight_codes(const float *W, int32_t N, int32_t taps, int32_t K,
                      const int32_t *perm, const int32_t count[2], const int32_t bits[2],
                      const float *s, int8_t *J) {
    int32_t base[2] = {0, count[0]};
    for (int32_t n = 0; n < N; ++n)
        for (int32_t t = 0; t < taps; ++t)
            for (int g = 0; g < ORC_GROUPS; ++g)
                for (int32_t j = 0; j < count[g]; ++j) {
                    int32_t p = base[g] + j;
                    int64_t row = ((int64_t)n * taps + t) * K;
                    J[row + p] = (int8_t)orc_weight_code(W[row + perm[p]], s[n * 2 + g], bits[g]);
                }
}

/* ------------------------------------------------------------------------- */
/* a2  Packing of n-bit code patterns into blocks of 32 (layout above).      */
/* ------------------------------------------------------------------------- */

/* Slice widths and bit offsets of an n-bit code; returns the slice count. */
static int code_slices(int32_t n, int32_t width[3], int32_t offset[3]) {
    int k = 0, off = 0;
    if (n == 8) { width[0] = 8; offset[0] = 0; return 1; }
    if (n & 4) { width[k] = 4; offset[k] = off; off += 4; ++k; }
    if (n & 2) { width[k] = 2; offset[k] = off; off += 2; ++k; }
    if (n & 1) { width[k] = 1; offset[k] = off; off += 1; ++k; }
    return k;
}

/* codes[32] are n-bit patterns (0 <= code < 2^n); words[n] receive the block. */
void orc_pack_block(const uint32_t *codes, int32_t n, uint32_t *words) {
    int32_t width[3], offset[3];
    int ns = code_slices(n, width, offset);
    memset(words, 0, sizeof(uint32_t) * (size_t)n);
    int word0 = 0;
    for (int k = 0; k < ns; ++k) {
        int32_t w = width[k], per_byte = 8 / w;
        for (int i = 0; i < 32; ++i) {
            int32_t t = i / 4, b = i % 4;
            uint32_t v = (codes[i] >> offset[k]) & ((1u << w) - 1u);
            int32_t q = t / per_byte;
            int32_t bit = 8 * b + w * (t % per_byte);
            words[word0 + q] |= v << bit;
        }
        word0 += w;
    }
}

void orc_unpack_block(const uint32_t *words, int32_t n, uint32_t *codes) {
    int32_t width[3], offset[3];
    int ns = code_slices(n, width, offset);
    for (int i = 0; i < 32; ++i) codes[i] = 0;
    int word0 = 0;
    for (int k = 0; k < ns; ++k) {
        int32_t w = width[k], per_byte = 8 / w;
        for (int i = 0; i < 32; ++i) {
            int32_t t = i / 4, b = i % 4;
            int32_t q = t / per_byte;
            int32_t bit = 8 * b + w * (t % per_byte);
            uint32_t v = (words[word0 + q] >> bit) & ((1u << w) - 1u);
            codes[i] |= v << offset[k];
        }
        word0 += w;
    }
}

static void put_words(uint8_t *dst, const uint32_t *words, int32_t n) {
    for (int32_t q = 0; q < n; ++q)
        for (int byte = 0; byte < 4; ++byte)
            dst[4 * q + byte] = (uint8_t)((words[q] >> (8 * byte)) & 0xFFu);
}

/* Packed activation rows: out[M][row_bytes].  Group g's segment holds PA_g
 * codes: U[m][base_g + c] for c < count[g], then zero padding. */
void orc_pack_act_rows(const uint8_t *U, int64_t M, int32_t K, const int32_t count[2],
                       const int32_t bits[2], int32_t pad_unit, uint8_t *out) {
    int64_t row_bytes = orc_row_bytes(count, bits, pad_unit, 1, 0);
    int32_t base[2] = {0, count[0]};
    for (int64_t m = 0; m < M; ++m) {
        uint8_t *dst = out + m * row_bytes;
        for (int g = 0; g < ORC_GROUPS; ++g) {
            int64_t codes_g = orc_act_group_codes(count[g], pad_unit);
            for (int64_t blk = 0; blk < codes_g / 32; ++blk) {
                uint32_t codes[32], words[8];
                for (int i = 0; i < 32; ++i) {
                    int64_t c = blk * 32 + i;
                    codes[i] = c < count[g] ? U[m * K + base[g] + c] : 0u;
                }
                orc_pack_block(codes, bits[g], words);
                put_words(dst, words, bits[g]);
                dst += 4 * bits[g];
            }
        }
    }
}

/* Packed weight rows: out[N][row_bytes].  Group g's segment holds PW_g codes
 * in tap-major order: position p -> tap p / PA_g, channel p % PA_g; codes are
 * stored as n-bit two's complement; padding is code 0. */
void orc_pack_weight_rows(const int8_t *J, int32_t N, int32_t taps, int32_t K,
                          const int32_t count[2], const int32_t bits[2], int32_t pad_unit,
                          uint8_t *out) {
    int64_t row_bytes = orc_row_bytes(count, bits, pad_unit, taps, 1);
    int32_t base[2] = {0, count[0]};
    for (int32_t n = 0; n < N; ++n) {
        uint8_t *dst = out + (int64_t)n * row_bytes;
        for (int g = 0; g < ORC_GROUPS; ++g) {
            int64_t pa = orc_act_group_codes(count[g], pad_unit);
            int64_t codes_g = orc_weight_group_codes(count[g], pad_unit, taps);
            uint32_t mask = (1u << bits[g]) - 1u;
            for (int64_t blk = 0; blk < codes_g / 32; ++blk) {
                uint32_t codes[32], words[8];
                for (int i = 0; i < 32; ++i) {
                    int64_t p = blk * 32 + i;
                    int64_t t = p / pa, c = p % pa;
                    int32_t j = 0;
                    if (t < taps && c < count[g])
                        j = J[((int64_t)n * taps + t) * K + base[g] + c];
                    codes[i] = (uint32_t)j & mask;
                }
                orc_pack_block(codes, bits[g], words);
                put_words(dst, words, bits[g]);
                dst += 4 * bits[g];
            }
        }
    }
}

/* ------------------------------------------------------------------------- */
/* a4  Integer dot products per precision group (Sec. 3, "a pure fixed-point */
/*     MAC" per fused dot product; Sec. 4.2 unsigned x signed -> int32).     */
/*     acc[g][i][n] = sum over c in group g of U[row_i][c] * J[n][c].        */
/* ------------------------------------------------------------------------- */
void orc_gemm_acc(const uint8_t *U, int32_t K, const int8_t *J, int32_t N,
                  const int32_t count[2], const int64_t *rows, int64_t n_rows,
                  int64_t *acc) {
    int32_t base[2] = {0, count[0]};
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t m = rows[i];
        for (int g = 0; g < ORC_GROUPS; ++g)
            for (int32_t n = 0; n < N; ++n) {
                int64_t sum = 0;
                for (int32_t c = 0; c < count[g]; ++c)
                    sum += (int64_t)U[m * K + base[g] + c] * (int64_t)J[(int64_t)n * K + base[g] + c];
                acc[((int64_t)g * n_rows + i) * N + n] = sum;
            }
    }
}

/* a7  Convolution as the same dot products over the receptive field.
 * U[(img*H + h)*Wd + w][K] are the activation codes of the input pixels
 * (NHWC), J[Cout][R*S][K] the weight codes.  Output pixel index
 * o = (img*P + p)*Q + q with P = (H + 2ph - R)/sh + 1, Q = (Wd + 2pw - S)/sw + 1.
 * Input positions outside the image contribute nothing (zero padding). */
void orc_conv_acc(const uint8_t *U, int32_t Nimg, int32_t H, int32_t Wd, int32_t K,
                  const int8_t *J, int32_t Cout, int32_t R, int32_t S, int32_t sh,
                  int32_t sw, int32_t ph, int32_t pw, const int32_t count[2],
                  const int64_t *pix, int64_t n_pix, int64_t *acc) {
    int32_t base[2] = {0, count[0]};
    int32_t P = (H + 2 * ph - R) / sh + 1, Q = (Wd + 2 * pw - S) / sw + 1;
    (void)Nimg;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n_pix; ++i) {
        int64_t o = pix[i];
        int64_t img = o / ((int64_t)P * Q);
        int32_t p = (int32_t)((o / Q) % P), q = (int32_t)(o % Q);
        for (int g = 0; g < ORC_GROUPS; ++g)
            for (int32_t n = 0; n < Cout; ++n) {
                int64_t sum = 0;
                for (int32_t r = 0; r < R; ++r)
                    for (int32_t s = 0; s < S; ++s) {
                        int32_t h = p * sh - ph + r, w = q * sw - pw + s;
                        if (h < 0 || h >= H || w < 0 || w >= Wd) continue;
                        const uint8_t *u = U + ((img * H + h) * Wd + w) * K + base[g];
                        const int8_t *j = J + ((int64_t)n * R * S + r * S + s) * K + base[g];
                        for (int32_t c = 0; c < count[g]; ++c)
                            sum += (int64_t)u[c] * (int64_t)j[c];
                    }
                acc[((int64_t)g * n_pix + i) * Cout + n] = sum;
            }
    }
}

/* ------------------------------------------------------------------------- */
/* a5  Epilogue: decode a = s_a * u / (2^na - 1) (Sec. 3 step 2) and          */
/*     w = s_w * j / 2^(nw-1) (Eq. (1) rescaled, step 3), so each group adds */
/*     s_a * s_w * Acc_g / ((2^na - 1) * 2^(nw-1)).  fp64.                    */
/*     s_a: [2] (per tensor) or [M][2] indexed by rows[i] (per row).          */
/* ------------------------------------------------------------------------- */
void orc_epilogue(const int64_t *acc, const int64_t *rows, int64_t n_rows, int32_t N,
                  const float *s_a, int32_t s_a_per_row, const float *s_w,
                  const int32_t bits_a[2], const int32_t bits_w[2], double *Y) {
    for (int64_t i = 0; i < n_rows; ++i)
        for (int32_t n = 0; n < N; ++n) {
            double y = 0.0;
            for (int g = 0; g < ORC_GROUPS; ++g) {
                double sa = s_a_per_row ? (double)s_a[rows[i] * 2 + g] : (double)s_a[g];
                double sw = (double)s_w[(int64_t)n * 2 + g];
                double la = (double)((1 << bits_a[g]) - 1);
                double lw = (double)(1 << (bits_w[g] - 1));
                y += sa * sw * (double)acc[((int64_t)g * n_rows + i) * N + n] / (la * lw);
            }
            Y[i * N + n] = y;
        }
}

/* ------------------------------------------------------------------------- */
/* f3  Variants the paper describes beside the default path (linear layers,  */
/*     codes in packed channel order, int32).                                */
/*  kind[g] 0: unsigned activation code, Sec. 3 step 2 (the default);         */
/*          1: signed activation code, Eq. (1) applied to the activation     */
/*             (u in [-2^(n-1), 2^(n-1)-1], decoded as s u / 2^(n-1)), the   */
/*             transformer-layer reading of Sec. 3;                           */
/*          2: one-bit +-1 code on both sides (Sec. 4.2: XNOR and POPCOUNT   */
/*             for one-bit channels): +1 for x >= 0, else -1, decoded as     */
/*             s * code; over m channels the dot product of two such rows is */
/*             m - 2 popcount(bits XOR bits).                                 */
/*  sub_k > 0: scale sub-groups along K (the fine scale groups, "GroupSize",  */
/*     of the evaluation setup): a group's packed positions are cut into runs */
/*     of sub_k, each with its own max-abs scale and exact accumulator; the  */
/*     epilogue sums the runs.  sub_k = 0: one run per group (the default).  */
/*  Scale arrays are [rows or 1][2][nb], nb = the larger group's run count.  */
/* ------------------------------------------------------------------------- */
int32_t orc_pm1_code(float x) { return x >= 0.0f ? 1 : -1; }

static int32_t run_of(int32_t j, int32_t sub_k) { return sub_k > 0 ? j / sub_k : 0; }

/* Max |x| over each run's real channels (per row, or over all rows). */
void orc_sub_scales(const float *X, int64_t M, int32_t K, const int32_t *perm, const int32_t count[2],
                    int32_t sub_k, int32_t nb, int32_t per_row, float *s) {
    int32_t base[2] = {0, count[0]};
    int64_t n_out = per_row ? M : 1;
    for (int64_t i = 0; i < n_out * 2 * nb; ++i) s[i] = 0.0f;
    for (int64_t m = 0; m < M; ++m)
        for (int g = 0; g < ORC_GROUPS; ++g)
            for (int32_t j = 0; j < count[g]; ++j) {
                float v = fabsf(X[m * K + perm[base[g] + j]]);
                float *t = &s[((per_row ? m : 0) * 2 + g) * nb + run_of(j, sub_k)];
                if (v > *t) *t = v;
            }
}

/* Codes C[M][K] of rows X[M][K] with scales s (layout above). */
void orc_codes_variant(const float *X, int64_t M, int32_t K, const int32_t *perm, const int32_t count[2],
                       const int32_t bits[2], const int32_t kind[2], int32_t sub_k, int32_t nb, const float *s,
                       int32_t per_row, int32_t *C) {
    int32_t base[2] = {0, count[0]};
    for (int64_t m = 0; m < M; ++m)
        for (int g = 0; g < ORC_GROUPS; ++g)
            for (int32_t j = 0; j < count[g]; ++j) {
                int32_t p = base[g] + j;
                float x = X[m * K + perm[p]];
                float sg = s[((per_row ? m : 0) * 2 + g) * nb + run_of(j, sub_k)];
                int32_t c;
                if (kind[g] == 2)
                    c = orc_pm1_code(x);
                else if (kind[g] == 1)
                    c = orc_weight_code(x, sg, bits[g]);   /* Eq. (1), the same rule as for weights */
                else
                    c = orc_act_code(x, sg, bits[g]);
                C[m * K + p] = c;
            }
}

/* acc[2][nb][n_rows][N]: exact sums of U * J over each run of each group. */
void orc_gemm_acc_runs(const int32_t *U, int32_t K, const int32_t *J, int32_t N, const int32_t count[2],
                       int32_t sub_k, int32_t nb, const int64_t *rows, int64_t n_rows, int64_t *acc) {
    int32_t base[2] = {0, count[0]};
    for (int64_t i = 0; i < 2 * nb * n_rows * N; ++i) acc[i] = 0;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n_rows; ++i) {
        int64_t m = rows[i];
        for (int g = 0; g < ORC_GROUPS; ++g)
            for (int32_t n = 0; n < N; ++n)
                for (int32_t j = 0; j < count[g]; ++j) {
                    int32_t b = run_of(j, sub_k);
                    acc[(((int64_t)g * nb + b) * n_rows + i) * N + n] +=
                        (int64_t)U[m * K + base[g] + j] * (int64_t)J[(int64_t)n * K + base[g] + j];
                }
    }
}

/* Y = sum_g sum_b s_a[g][b] s_w[n][g][b] acc[g][b] / (La_g Lw_g), fp64, with
 * La = 2^na - 1 (kind 0), 2^(na-1) (kind 1), 1 (kind 2) and Lw = 2^(nw-1),
 * or 1 for kind 2. */
void orc_epilogue_runs(const int64_t *acc, const int64_t *rows, int64_t n_rows, int32_t N, int32_t nb,
                       const float *s_a, int32_t s_a_per_row, const float *s_w, const int32_t bits_a[2],
                       const int32_t bits_w[2], const int32_t kind[2], double *Y) {
    for (int64_t i = 0; i < n_rows; ++i)
        for (int32_t n = 0; n < N; ++n) {
            double y = 0.0;
            for (int g = 0; g < ORC_GROUPS; ++g) {
                double la = kind[g] == 2 ? 1.0 : (kind[g] == 1 ? (double)(1 << (bits_a[g] - 1))
                                                               : (double)((1 << bits_a[g]) - 1));
                double lw = kind[g] == 2 ? 1.0 : (double)(1 << (bits_w[g] - 1));
                for (int32_t b = 0; b < nb; ++b) {
                    double sa = (double)s_a[((s_a_per_row ? rows[i] : 0) * 2 + g) * nb + b];
                    double sw = (double)s_w[((int64_t)n * 2 + g) * nb + b];
                    y += sa * sw * (double)acc[(((int64_t)g * nb + b) * n_rows + i) * N + n] / (la * lw);
                }
            }
            Y[i * N + n] = y;
        }
}
