/*
 * soniq.h -- C ABI of the GB300 (sm_103a) SONIQ inference library.
 *
 * SONIQ (arXiv 2311.14114) quantizes every input channel of a layer to one of
 * two precisions.  Inference needs (Sec. 3 "Enabling Low-Cost Fixed-Point
 * Operations", Sec. 4.1 "Channel re-ordering and padding"):
 *   - a channel permutation that makes each precision group contiguous along
 *     the reduction axis K (Sec. 3 "Dynamic channel re-ordering"),
 *   - one max-abs scale per group (step 1),
 *   - unsigned activation codes (step 2) and two's-complement-fraction weight
 *     codes, Eq. (1) (step 3),
 *   - integer dot products inside each group, combined by the group scales.
 *
 * Conventions for every call:
 *   * Device pointers are CUDA global-memory addresses owned by the caller;
 *     the library never allocates, frees or retains them.  Calls that need
 *     working memory take it from the caller as a `scratch` pointer and its
 *     size in bytes; a *_scratch_bytes() query (host only) says how much.
 *   * Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  Argument errors are detected on the host before any
 *     CUDA call and returned synchronously.  Launch failures return
 *     SONIQ_ERR_CUDA.  Kernels never trap: a bounded device-side wait that
 *     runs out records an error word, read back by soniq_sync_status().
 *   * No C++ exception crosses this interface.
 *   * Packed rows, codes and accumulators follow the layout described at
 *     soniq_layout below; packed bytes and int32 accumulators are bit-exact
 *     functions of the inputs.
 */
#ifndef SONIQ_H_
#define SONIQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SONIQ_ABI_VERSION 3

/* Exported symbols (the library is built with hidden default visibility). */
#if defined(__GNUC__)
#define SONIQ_API __attribute__((visibility("default")))
#else
#define SONIQ_API
#endif

typedef enum soniq_status {
    SONIQ_OK = 0,
    SONIQ_ERR_INVALID_ARG = 1,  /* null pointer, negative size, inconsistent layout */
    SONIQ_ERR_UNSUPPORTED = 2,  /* well-formed but outside the kernels' limits */
    SONIQ_ERR_ALIGNMENT = 3,    /* a pointer is not aligned as the call requires */
    SONIQ_ERR_CUDA = 4,         /* a CUDA runtime call or kernel launch failed */
    SONIQ_ERR_TIMEOUT = 5       /* a kernel's bounded wait ran out (see soniq_sync_status) */
} soniq_status;

/* A cudaStream_t, passed opaquely so this header needs no CUDA headers. */
typedef void *soniq_stream_t;

/*
 * Per-layer precision layout (Sec. 3 "Dynamic channel re-ordering"; Fig. 2;
 * Sec. 4.1).  Group 0 is the low precision, group 1 the high one.
 *
 *   K          logical input channels (for a convolution: C_in).
 *   n_groups   1 or 2; with 1, count[1] must be 0.
 *   count[g]   channels in group g, count[0] + count[1] == K.
 *   bits_w[g]  weight bits of group g, 1..8 (Eq. (1), n).
 *   bits_a[g]  activation bits of group g, 1..8 (Sec. 3 step 2, n).
 *   perm       DEVICE pointer, K int32: perm[j] is the original channel stored
 *              at packed position j.  Positions [0,count[0]) form group 0,
 *              [count[0],K) group 1.  Must be a permutation of 0..K-1
 *              (soniq_validate_layout checks a host copy).
 *   pad_unit   32 or 128: each group of a packed activation row holds
 *              PA_g = roundup(count[g], pad_unit) codes; pad codes are 0.
 *
 * Packed rows.  An activation row is [group 0: PA_0 codes][group 1: PA_1
 * codes].  A weight row for `taps` filter taps is [group 0: PW_0][group 1:
 * PW_1] with PW_g = roundup(taps * PA_g, 128), in tap-major order (position p
 * holds tap p / PA_g, channel p % PA_g of the group; positions beyond
 * taps * PA_g are 0).  Codes are stored in blocks of 32: a block of n-bit
 * codes is n little-endian 32-bit words; the code bits are cut into slices of
 * width 4, 2, 1 (low bits first; n = 8 is one 8-bit slice); a w-bit slice
 * takes w words and code i (t = i/4, b = i%4) sits in slice word t/(8/w) at
 * bit 8*b + w*(t % (8/w)).  Activation codes are unsigned, weight codes n-bit
 * two's complement.  Row strides are soniq_packed_row_bytes().
 *
 * Variants (all zero by default; linear layers only: taps = 1, pad_unit 128,
 * per-row weight scales, the staged tensor-core path of soniq_mp_gemm):
 *   act_kind[g]  SONIQ_ACT_UNSIGNED (Sec. 3 step 2), SONIQ_ACT_SIGNED (Eq. (1)
 *              applied to the activation: codes in [-2^(n-1), 2^(n-1) - 1],
 *              stored as n-bit two's complement, decoded as s u / 2^(n-1)),
 *              or SONIQ_ACT_PM1 (one-bit groups, Sec. 4.2 XNOR / POPCOUNT:
 *              both operands take code +1 for x >= 0 and -1 otherwise, stored
 *              as the bit (code + 1) / 2 and decoded as s * code; needs
 *              bits_w[g] = bits_a[g] = 1).
 *   sub_k      0, or a multiple of 128: scale runs along K.  Group g's packed
 *              positions are cut into runs of sub_k codes, each with its own
 *              max-abs scale (activations per tensor or per row, weights per
 *              row) and its own exact accumulator; the epilogue sums the runs.
 *              Scale arrays then hold nb entries per (row, group):
 *              [rows][2][nb], nb = soniq_scale_runs(layout).  Groups with
 *              fp16 operands (codes above 4 bits) need sub_k <= 2^24 /
 *              ((2^na - 1) 2^(nw - 1)) (512 for 8-bit groups).
 */
typedef struct soniq_layout {
    int32_t K;
    int32_t n_groups;
    int32_t count[2];
    int32_t bits_w[2];
    int32_t bits_a[2];
    const int32_t *perm;
    int32_t pad_unit;
    int32_t act_kind[2];
    int32_t sub_k;
} soniq_layout;

enum { SONIQ_ACT_UNSIGNED = 0, SONIQ_ACT_SIGNED = 1, SONIQ_ACT_PM1 = 2 };

/* Scale granularity (Sec. 3 step 1: one max-abs scale per group; C2: one
 * scale per fused dot product).  Scale arrays are fp32 with 2 entries per
 * scale (group 0, group 1). */
enum {
    SONIQ_SCALE_PER_TENSOR = 0,  /* one scale per (tensor, group): [2] ([N][2] replicated for weights) */
    SONIQ_SCALE_PER_ROW = 1,     /* one scale per (row, group): [rows][2] */
    SONIQ_SCALE_CALIBRATED = 2   /* activations only: caller supplies s_a[2]; inputs beyond it clip */
};

enum { SONIQ_OUT_F16 = 0, SONIQ_OUT_BF16 = 1 };

enum {
    SONIQ_FLAG_FORCE_GEMV = 1u,          /* soniq_mp_gemm: use the CUDA-core GEMV for any M <= 16 */
    SONIQ_FLAG_FORCE_MMA = 2u,           /* soniq_mp_gemm: use a tensor-core kernel for any M */
    SONIQ_FLAG_FORCE_FUSED = 4u,         /* tensor-core work takes the fused kernel even when
                                            scratch for the staged path is given */
    SONIQ_FLAG_FORCE_STAGED = 8u,        /* tensor-core work takes the staged path whenever the
                                            scratch suffices, however small the problem (without
                                            it the staged path is used from about 2^30
                                            multiply-adds) */
    SONIQ_FLAG_FORCE_SKINNY = 16u,       /* tensor-core work takes the skinny swap-AB kernel
                                            (M <= 32, taps = 1, groups padded to 128 codes) */
    SONIQ_FLAG_TEST_DROP_ARRIVE = 0x100u /* test hook: the tensor-core kernels' operand producer
                                            skips its first arrival (fused) or its first K-stage
                                            (staged, skinny), so the consumer's bounded wait runs
                                            out and the call reports SONIQ_ERR_TIMEOUT */
};

/* Kernels behind soniq_mp_gemm (see soniq_mp_gemm_path). */
enum {
    SONIQ_PATH_GEMV = 0,           /* CUDA-core GEMV streaming the packed weights (small M) */
    SONIQ_PATH_TENSOR = 1,         /* tcgen05 kernel expanding packed tiles on chip (no scratch) */
    SONIQ_PATH_TENSOR_STAGED = 2,  /* codes expanded once into scratch, then a tcgen05 GEMM */
    SONIQ_PATH_TENSOR_SKINNY = 3   /* swap-AB tcgen05 kernel for few rows: packed weight rows
                                      are the MMA's M = 128 side, converted on chip */
};
/* Without flags, soniq_mp_gemm runs the GEMV for M <= SONIQ_GEMV_MAX_M and the
 * skinny tensor-core kernel for M <= SONIQ_SKINNY_MAX_M. */
#define SONIQ_GEMV_MAX_M 12
#define SONIQ_SKINNY_MAX_M 32

/* Convolution geometry.  Input NHWC [batch][H][W][C_in], output NHWC
 * [batch][P][Q][C_out], P = (H + 2*pad_h - R)/stride_h + 1, Q likewise. */
typedef struct soniq_conv_desc {
    int32_t batch, H, W;
    int32_t C_out;
    int32_t R, S;
    int32_t stride_h, stride_w;
    int32_t pad_h, pad_w;
} soniq_conv_desc;

/*
 * Quantize-in-epilogue: the next layer's activation quantization fused into
 * this layer's GEMM / convolution epilogue (Sec. 4.1: the CPU back-end fuses
 * Conv2D + BatchNorm + Quantize so the next layer receives its codes
 * directly).  The next layer's codes are those soniq_quantize_act computes
 * with SONIQ_SCALE_CALIBRATED on the fp16 outputs of this call: every output
 * y is rounded to fp16 first, then u = clip(round_half_even(fp32(y16 / s) *
 * (2^n - 1)), 0, 2^n - 1) with the next layer's scale s and bits n.
 *
 * Convention: this call's output column j is packed position j of the next
 * layer's activation rows, so N must equal PA_0' + PA_1' of its layout (the
 * padded row length) and the caller arranges this layer's weight rows once,
 * offline, in that order: the rows of the next layer's group-0 channels in
 * its permutation order, zero rows up to PA_0', then its group-1 channels and
 * zero rows up to PA_1'.  The next layer's permutation is thereby folded into
 * this layer's output order and needs no gather at run time.  Codes at pad
 * positions are 0.
 */
typedef struct soniq_next_layer {
    const soniq_layout *layout;  /* the next layer's layout; layout->perm is not read */
    const float *s_a;            /* device fp32 [2]: its calibrated activation scales */
    uint8_t *Ap;                 /* device out [M][soniq_packed_row_bytes(layout, 0, 1)], 4-byte aligned */
} soniq_next_layer;

/* ---- sizes and checks (host only, no CUDA calls) ------------------------ */

SONIQ_API int32_t soniq_abi_version(void);
SONIQ_API const char *soniq_status_string(soniq_status status);

/* Codes per row of group `group`: activation rows (is_weight = 0) or weight
 * rows with `taps` taps (is_weight = 1).  -1 on a bad argument. */
SONIQ_API int64_t soniq_group_codes(const soniq_layout *layout, int32_t group, int32_t is_weight,
                          int32_t taps);

/* Bytes per packed row (a multiple of 4; of 16 for weight rows).  -1 on a bad
 * argument. */
SONIQ_API int64_t soniq_packed_row_bytes(const soniq_layout *layout, int32_t is_weight, int32_t taps);

/* Scale runs per (row, group) in scale arrays: ceil(max PA_g / sub_k) with
 * scale runs (layout->sub_k > 0), else 1.  -1 on a bad layout. */
SONIQ_API int32_t soniq_scale_runs(const soniq_layout *layout);

/* Checks the layout fields; if perm_host is non-NULL also checks that it is a
 * permutation of 0..K-1.  Does not read layout->perm. */
SONIQ_API soniq_status soniq_validate_layout(const soniq_layout *layout, const int32_t *perm_host);

/* Kernels this library has launched since load (all threads, all devices). */
SONIQ_API int64_t soniq_launch_count(void);

/* ---- the hot path ------------------------------------------------------- */

/*
 * Weight quantize-and-pack (offline, once per layer).  Sec. 3 steps 1 and 3,
 * Eq. (1): per scale group s = max|w|, w' = w / s (fp32, IEEE), code
 * j = clamp(round_half_even(w' * 2^(n-1)), -2^(n-1), 2^(n-1) - 1), the nearest
 * level of Eq. (1); s = 0 gives j = 0.  Non-finite weights: the max-abs scale
 * skips NaN and keeps infinities (a group holding one gets s = inf, and every
 * code of it is 0); a NaN w' (a NaN weight, or inf / inf) gives j = 0.
 *
 *   W          device fp32 [N][taps][K] (taps = 1: a linear layer [N][K];
 *              a convolution OHWI [C_out][R*S][C_in]), 4-byte aligned.
 *   N          output rows (>= 0; 0 is a no-op).
 *   taps       filter taps R*S, 1 to 4096.
 *   scale_mode SONIQ_SCALE_PER_ROW (one scale per (n, group) over all taps)
 *              or SONIQ_SCALE_PER_TENSOR (one per group; written to every row).
 *   Wp         device out [N][soniq_packed_row_bytes(layout, 1, taps)], 16-byte aligned.
 *   s_w        device out fp32 [N][2] ([N][2][nb] with scale runs).
 * Layout variants (act_kind, sub_k): SONIQ_ACT_PM1 groups take code +1 / -1;
 * scales are per row and per run; SONIQ_SCALE_PER_TENSOR is unsupported.
 */
SONIQ_API soniq_status soniq_pack_weights(const soniq_layout *layout, const float *W, int32_t N,
                                int32_t taps, int32_t scale_mode, uint8_t *Wp, float *s_w,
                                soniq_stream_t stream);

/*
 * Activation quantize-and-pack (per inference call).  Sec. 3 steps 1 and 2:
 * s = max|a| per scale group, code u = clip(round_half_even(fp32(a / s) *
 * (2^n - 1)), 0, 2^n - 1); s = 0 gives u = 0.  Channels are gathered through
 * layout->perm and each group is zero-padded to PA_g codes.  Non-finite
 * inputs: under a finite scale +inf clips to 2^n - 1 and -inf to 0; a NaN
 * quotient (a NaN input, or inf / inf) gives u = 0; max-abs scales skip NaN
 * and keep infinities.
 *
 *   A          device fp16 [M][K] (IEEE binary16 bits), 2-byte aligned; K <= 32768.
 *   M          rows (tokens, or pixels of an NHWC image); 0 is a no-op.
 *   scale_mode SONIQ_SCALE_PER_TENSOR: s_a is an output [2];
 *              SONIQ_SCALE_PER_ROW:    s_a is an output [M][2];
 *              SONIQ_SCALE_CALIBRATED: s_a is an input [2].
 *              With scale runs each entry is nb entries ([2][nb], [M][2][nb]).
 *              Signed (SONIQ_ACT_SIGNED) groups take the Eq. (1) code, +-1
 *              groups the sign; the variants need no scratch.
 *   s_a        device fp32, see scale_mode.
 *   Ap         device out [M][soniq_packed_row_bytes(layout, 0, 1)], 4-byte aligned.
 *   scratch, scratch_bytes
 *              optional caller-owned device memory, 16-byte aligned.  With
 *              SONIQ_SCALE_PER_TENSOR and scratch_bytes >=
 *              soniq_quantize_act_scratch_bytes(), inputs whose rows fit on
 *              chip (about M * K <= 15 * 2^20) are quantized in one pass over
 *              A by a cooperative kernel whose grid barrier and per-CTA maxima
 *              live in the scratch; otherwise (or with scratch = NULL) the
 *              scale is found by a separate max-abs pass first.  Other modes
 *              ignore the scratch.
 *              Contract: the scratch must be zero-filled before its first use
 *              (cudaMemsetAsync once after allocating it); every completed
 *              call leaves it zero-filled again.  After soniq_sync_status
 *              reports SONIQ_ERR_TIMEOUT, zero it again before reuse.  Calls
 *              that may overlap on the GPU (different streams) must use
 *              different scratch buffers.
 */
SONIQ_API soniq_status soniq_quantize_act(const soniq_layout *layout, const void *A, int64_t M,
                                int32_t scale_mode, float *s_a, uint8_t *Ap, void *scratch,
                                size_t scratch_bytes, soniq_stream_t stream);

/* Scratch bytes that soniq_quantize_act can use for these arguments (0 when
 * the call needs none).  Host only; -1 on a bad argument. */
SONIQ_API int64_t soniq_quantize_act_scratch_bytes(const soniq_layout *layout, int64_t M,
                                                   int32_t scale_mode);

/*
 * Per-tensor activation quantize-and-pack that allocates nothing and takes no
 * scratch argument.  The paper has no counterpart; this is an engineering
 * variant of soniq_quantize_act (SONIQ_SCALE_PER_TENSOR, one pass) for
 * callers that cannot call cudaMalloc or hand the library device memory of
 * their own: for instance a host that only gives the library the tensors of
 * the layer (an inference runtime whose allocator is not reachable from the
 * code that calls this library, or a real-time loop in which allocating, and
 * the device synchronization that cudaMalloc/cudaFree may cause, is not
 * allowed).
 *
 * It computes exactly what soniq_quantize_act computes in per-tensor mode
 * (same s_a and packed bytes).  Its working memory is a file-scope static
 * device array of the library (8 KB on every device that loads the library,
 * held until the process exits): a grid barrier (arrival count, generation)
 * and the per-CTA maxima of at most 1024 CTAs.
 *   Set-up: the first call on each device, with that device current, looks up
 *   the array's device address (cudaGetSymbolAddress) and sets the kernel's
 *   shared-memory attributes; make that first call before any stream capture.
 *   Limits: one CTA of 1024 threads per SM, each holding its M / (number of
 *   SMs) rows in at most 200 KB of shared memory (2 * K bytes per row plus the
 *   permutation): M * K up to about 15 * 2^20 on a 152-SM GB300.  Larger
 *   inputs return SONIQ_ERR_UNSUPPORTED before anything is launched; there is
 *   no two-pass fallback.
 *   Sharing: every call uses the same array.  The barrier count must start at
 *   zero: it is zero when the library loads and every completed call leaves it
 *   at zero; the per-CTA maxima are written before they are read.  Two calls
 *   that overlap on the GPU (different streams) race on the array and give
 *   wrong results; serialize them.
 *   Timeouts: a barrier wait that runs out (2 s) makes soniq_sync_status
 *   return SONIQ_ERR_TIMEOUT; that call then waits for the whole device and
 *   resets the barrier, so the next call starts clean.
 * Arguments as for soniq_quantize_act; s_a is an output [2].
 */
SONIQ_API soniq_status soniq_quantize_act_oneshot(const soniq_layout *layout, const void *A, int64_t M,
                                        float *s_a, uint8_t *Ap, soniq_stream_t stream);

/*
 * Mixed-precision quantized GEMM Y = A W^T.  Sec. 3 (integer MAC per fused
 * dot product, decode rules of steps 2-3) and Sec. 4.2 (unsigned x signed
 * integer dot products):
 *   Acc_g[m][n] = sum over k in group g of u[m][k] * j[n][k]   (exact int32)
 *   Y[m][n]     = sum_g s_a(m,g) * s_w[n][g] / ((2^na_g - 1) * 2^(nw_g - 1)) * Acc_g[m][n]
 * computed in fp32 and rounded to nearest fp16 (or bf16).  M <= SONIQ_GEMV_MAX_M
 * runs a bandwidth-bound CUDA-core GEMV, M <= SONIQ_SKINNY_MAX_M the skinny
 * swap-AB tensor-core kernel, larger M the tcgen05 GEMM (flags can force a
 * kernel; the GEMV takes M <= 16, the skinny kernel M <= 32);
 * soniq_mp_gemm_path tells which.
 *
 *   Ap, s_a    from soniq_quantize_act with the same layout (pad_unit 32 or 128);
 *              s_a [2] (PER_TENSOR / CALIBRATED) or [M][2] (PER_ROW).
 *   Wp, s_w    from soniq_pack_weights with the same layout and taps = 1.
 *   Y          device out [M][N], fp16 or bf16 per out_dtype, 16-byte aligned.
 *   acc_dbg    NULL, or device out int32 [2][M][N]: the exact Acc_g.
 *   next       NULL, or the next layer whose codes the epilogue also writes
 *              (soniq_next_layer above; out_dtype must be SONIQ_OUT_F16, Y may
 *              then be NULL).  Needs the staged path: scratch of at least
 *              soniq_mp_gemm_scratch_bytes(..., flags | SONIQ_FLAG_FORCE_STAGED),
 *              else SONIQ_ERR_UNSUPPORTED.
 *   Limits (SONIQ_ERR_UNSUPPORTED otherwise): K <= 65536, M < 2^31.  The tensor-core
 *   kernel accumulates integer codes in fp32, exact while every partial sum
 *   stays within 2^24; a group whose worst-case sum over its K range could
 *   exceed that is accumulated in bounded segments that are drained to int32,
 *   and at most one of the two groups may need segments.
 */
SONIQ_API soniq_status soniq_mp_gemm(const soniq_layout *layout, const uint8_t *Ap, const float *s_a,
                           int32_t scale_mode, int64_t M, const uint8_t *Wp, const float *s_w,
                           int32_t N, void *Y, int32_t out_dtype, int32_t *acc_dbg,
                           uint32_t flags, void *scratch, size_t scratch_bytes,
                           const soniq_next_layer *next, soniq_stream_t stream);

/* Scratch of soniq_mp_gemm and soniq_mp_conv2d.  With scratch (256-byte
 * aligned) of at least the *_scratch_bytes() size, the tensor-core work takes
 * the staged path: every packed code is expanded once into tensor-pipe
 * operands in the scratch (E4M3 bytes for groups of <= 4-bit codes, fp16 for
 * wider ones; a convolution's activations as implicit-GEMM rows), and a
 * persistent tcgen05 GEMM reads them.  Without it (scratch = NULL or too
 * small) the fused kernel expands packed tiles on chip.  Both give the same
 * bits.  The scratch needs no initialization; calls that may overlap on the
 * GPU must use different scratch buffers. */

/* The kernel soniq_mp_gemm runs for these arguments (SONIQ_PATH_*), or -1
 * if it would return an error.  Host only (reads the device's SM count). */
SONIQ_API int32_t soniq_mp_gemm_path(const soniq_layout *layout, int64_t M, int32_t N, uint32_t flags,
                                     size_t scratch_bytes);

/* Scratch bytes soniq_mp_gemm can use for these arguments (0: none).  Host
 * only; -1 on a bad argument. */
SONIQ_API int64_t soniq_mp_gemm_scratch_bytes(const soniq_layout *layout, int64_t M, int32_t N,
                                              uint32_t flags);

/*
 * Mixed-precision quantized convolution as implicit GEMM (Sec. 4.1: the CPU
 * and GPU back-ends run convolutions on the re-ordered, padded channel
 * blocks; Sec. 6 evaluates conv layers).  K = R*S*C_in in the weight order
 * (group, tap, channel); input positions outside the image contribute 0.
 *
 *   cd         geometry; P, Q > 0 and R * S <= 4096 (SONIQ_ERR_INVALID_ARG otherwise);
 *              batch * P * Q < 2^31 (SONIQ_ERR_UNSUPPORTED otherwise).
 *   Xp, s_a    soniq_quantize_act of the NHWC input viewed as [batch*H*W][C_in],
 *              with a per-tensor or calibrated scale (a per-pixel scale would
 *              break the shared scale of one dot product, C2).
 *   Wp, s_w    soniq_pack_weights of OHWI weights with taps = R*S.
 *   Y          device out NHWC [batch][P][Q][C_out], 16-byte aligned.
 *   acc_dbg    NULL or device out int32 [2][batch*P*Q][C_out].
 *   next       NULL, or the next layer whose codes the epilogue also writes,
 *              as for soniq_mp_gemm (C_out = PA_0' + PA_1').
 */
SONIQ_API soniq_status soniq_mp_conv2d(const soniq_layout *layout, const soniq_conv_desc *cd,
                             const uint8_t *Xp, const float *s_a, int32_t scale_mode,
                             const uint8_t *Wp, const float *s_w, void *Y, int32_t out_dtype,
                             int32_t *acc_dbg, uint32_t flags, void *scratch, size_t scratch_bytes,
                             const soniq_next_layer *next, soniq_stream_t stream);

/* Scratch bytes soniq_mp_conv2d can use for these arguments (0: none).  Host
 * only; -1 on a bad argument. */
SONIQ_API int64_t soniq_mp_conv2d_scratch_bytes(const soniq_layout *layout, const soniq_conv_desc *cd,
                                                uint32_t flags);

/* Waits for `stream`, then returns SONIQ_ERR_TIMEOUT if any kernel of this
 * library on the current device recorded a timed-out wait since the last
 * call (and clears that record), SONIQ_ERR_CUDA on a CUDA error, else
 * SONIQ_OK.  When the timed-out wait was the grid barrier of
 * soniq_quantize_act_oneshot, it also waits for the whole device and then
 * resets that barrier. */
SONIQ_API soniq_status soniq_sync_status(soniq_stream_t stream);

/* Test hook, not for production use.  When armed (armed != 0), the next
 * launch of the one-pass per-tensor quantize kernel, from soniq_quantize_act
 * or soniq_quantize_act_oneshot, has its first CTA skip its grid-barrier
 * arrival: the other CTAs' bounded waits run out after 2 s, the outputs are
 * not written, and soniq_sync_status reports SONIQ_ERR_TIMEOUT.  The hook
 * disarms itself at that launch.  No fault, trap or hang is involved. */
SONIQ_API void soniq_test_drop_barrier_arrival(int32_t armed);

#ifdef __cplusplus
}
#endif

#endif /* SONIQ_H_ */
