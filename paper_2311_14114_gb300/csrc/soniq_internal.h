// Internal declarations shared by the SONIQ CUDA translation units.
// Host code (validation, dispatch) and kernels see the same geometry structs.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "soniq.h"

namespace soniq {

// One precision group as the kernels see it (Sec. 3 "Dynamic channel
// re-ordering": each group is a contiguous run of packed channels).
struct GroupGeom {
    int32_t count;      // logical channels
    int32_t bits_a;     // activation bits
    int32_t bits_w;     // weight bits
    int32_t pa;         // activation codes per row (per pixel for conv): roundup(count, pad)
    int32_t pw;         // weight codes per row: roundup(taps * pa, 128)
    int32_t a_off;      // byte offset of the group in a packed activation row
    int32_t w_off;      // byte offset of the group in a packed weight row
    int32_t perm_base;  // first packed position of the group
};

struct LayoutGeom {
    int32_t K;
    int32_t taps;
    int32_t a_row_bytes;
    int32_t w_row_bytes;
    GroupGeom g[2];
    // layout variants: SONIQ_ACT_* per group, scale runs along K (0: none),
    // scale entries per (row, group), and whether any variant is on
    int32_t act_kind[2];
    int32_t sub_k;
    int32_t nb;
    int32_t variant;
};

// Fills `geo` from a layout; returns SONIQ_OK or the validation error.
soniq_status make_geom(const soniq_layout* L, int32_t taps, LayoutGeom* geo);

// Device address of the library's error word on the current device (0 on failure).
unsigned* device_error_word();
// Bits of the device error word, by the kind of wait that ran out.
constexpr unsigned kErrWait = 1u;             // a bounded mbarrier wait (tensor-core kernel, GEMV)
constexpr unsigned kErrQuantBarrier = 2u;     // grid barrier of the one-pass quantize, caller scratch
constexpr unsigned kErrOneshotBarrier = 4u;   // grid barrier of soniq_quantize_act_oneshot
// Caller scratch of the one-pass per-tensor quantize: the barrier words in the
// first 256 bytes, then the per-CTA maxima [kMaxGridPartials][2].
constexpr int kMaxGridPartials = 1024;
constexpr int64_t kQuantScratchBytes = 256 + 8 * kMaxGridPartials;
// Per-tensor inputs up to this size are read by the absmax pass with an L2
// evict-last policy, so that the quantize pass reads them from L2 (the L2
// holds about 126 MB).
constexpr int64_t kKeepInL2Bytes = 80ll << 20;
// True once for the launch that the test hook soniq_test_drop_barrier_arrival armed.
bool take_drop_arrival();
void note_launch(int n = 1);
int num_sms();
// Asks for the largest shared-memory carve-out for `func` (once per device):
// every kernel of the library then runs in one L1 / shared-memory split, so
// consecutive calls do not make the SMs reconfigure between kernels.
cudaError_t prefer_max_shared(const void* func);

// Launches `kernel` with programmatic stream serialization: it may start (and
// run up to its pdl_wait) while the previous kernel in the stream finishes.
template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// ---- launchers (return the CUDA error of the launch) ----------------------

// keep_l2: read with an L2 evict-last policy for a quantize pass that follows
// with demote set (launch_quantize_gather).
cudaError_t launch_act_absmax(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A,
                              int64_t M, float* s_out, bool keep_l2, cudaStream_t st);
// One-pass per-tensor quantize (cooperative launch); its grid barrier (two
// words, zero between launches) and per-CTA maxima [max_ctas][2] are `bar` and
// `part`; a barrier wait that runs out ORs `err_bit` into the error word.
// cudaErrorNotSupported when the rows do not fit on chip.
cudaError_t launch_quantize_fused(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                  float* s_a, uint8_t* Ap, cudaStream_t st, unsigned* bar, float* part,
                                  int max_ctas, unsigned err_bit);
// Tiled quantize-and-pack (per-tensor scale given in s_a, calibrated, or per
// row); with tensor_in_cta a single CTA holds every row and computes the
// per-tensor scale itself (cudaErrorNotSupported if M is too large).
cudaError_t launch_quantize_rows(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                 int32_t scale_mode, bool tensor_in_cta, float* s_a, uint8_t* Ap, cudaStream_t st);
// Tiled quantize with bulk-staged rows and permutation gathers (rows of
// 16-byte multiples, 16-byte aligned); scale_mode PER_ROW finds the scales,
// the other modes read s_a[2].  demote: the rows were read by
// launch_act_absmax with keep_l2, and their L2 priority is reset here.
// Returns cudaErrorNotSupported when the layout does not fit it
// (quantize_gather_supported false).
bool quantize_gather_supported(const LayoutGeom& geo, int32_t scale_mode, const void* A);
cudaError_t launch_quantize_gather(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                   int32_t scale_mode, bool demote, float* s_a, uint8_t* Ap, cudaStream_t st);
cudaError_t launch_weight_absmax(const LayoutGeom& geo, const int32_t* perm, const float* W,
                                 int32_t N, float* s_out, cudaStream_t st);
cudaError_t launch_pack_weights(const LayoutGeom& geo, const int32_t* perm, const float* W,
                                int32_t N, int32_t per_row, uint8_t* Wp, float* s_w,
                                cudaStream_t st);

// Layout variants (variant.cu): scales per (row or tensor, group, run), then
// codes and packing; weights always per row.
cudaError_t launch_variant_quantize_act(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                        int32_t scale_mode, float* s_a, uint8_t* Ap, cudaStream_t st);
cudaError_t launch_variant_pack_weights(const LayoutGeom& geo, const int32_t* perm, const float* W, int32_t N,
                                        float* s_w, uint8_t* Wp, cudaStream_t st);

struct GemvArgs {
    const uint8_t* Ap;
    const uint8_t* Wp;
    const float* s_a;
    const float* s_w;
    void* Y;
    int32_t* acc_dbg;
    int32_t M;
    int32_t N;
    int32_t s_a_per_row;
    int32_t out_bf16;
};
// Returns cudaErrorNotSupported if the shape does not fit the GEMV kernel.
cudaError_t launch_gemv(const LayoutGeom& geo, const GemvArgs& a, cudaStream_t st);
bool gemv_supported(const LayoutGeom& geo, int64_t M, int64_t N);

struct MmaArgs {
    const uint8_t* Ap;
    const uint8_t* Wp;
    const float* s_a;
    const float* s_w;
    void* Y;
    int32_t* acc_dbg;
    int64_t M;        // output rows (conv: batch * P * Q)
    int32_t N;        // output columns (conv: C_out)
    int32_t s_a_per_row;
    int32_t out_bf16;
    uint32_t flags;
    // convolution geometry; conv = 0 for a plain GEMM
    int32_t conv;
    int32_t H, W, P, Q, R, S, sh, sw, ph, pw;
    // quantize-in-epilogue (staged path only): the next layer's geometry, scales and codes
    const LayoutGeom* next;
    const float* next_s_a;
    uint8_t* next_Ap;
};
// Host-side planning of the tensor-core kernel (exactness segments etc.).
soniq_status mma_check(const LayoutGeom& geo);
cudaError_t launch_mma(const LayoutGeom& geo, const MmaArgs& a, cudaStream_t st);

// ---- the skinny swap-AB tensor-core path (skinny_gemm.cu) ------------------
// M <= 32 activation rows against packed weight rows converted on chip.
bool skinny_supported(const LayoutGeom& geo, int64_t M, int64_t N);
cudaError_t launch_skinny(const LayoutGeom& geo, const MmaArgs& a, cudaStream_t st);

// ---- the staged tensor-core path (staged_gemm.cu) ---------------------------
// Packed codes are expanded once into tensor-pipe operands in caller scratch
// (E4M3 bytes for groups with <= 4-bit codes on both sides, fp16 otherwise),
// then a persistent tcgen05 GEMM runs over them.
struct StagedGroup {
    int32_t kind;          // 0: E4M3, 1: fp16, 2: E2M1 (kind::mxf4)
    int32_t stages;        // K-stages of the ring (128 bytes of K each)
    int32_t x0;            // byte offset of the group in an expanded row
    int32_t seg_stages;    // K-stages per exact fp32 segment
    int32_t n_seg;         // segments (> 1: drained to int32)
    int32_t center;        // fp16 activations are stored as u - center
};
struct StagedPlan {
    StagedGroup g[2];
    int64_t eb;            // bytes of an expanded row (both groups)
    int32_t seg_group;     // the group that needs segments, or -1
    int32_t f4;            // some group runs on E2M1 operands (240-column tiles)
};
// False when the layout cannot take the staged path (two segmented groups).
// With allow_f4, groups of <= 2-bit unsigned activations and <= 2-bit weights
// run on E2M1 operands (their expanded rows are never longer than E4M3 ones,
// so scratch sized without allow_f4 serves both).
bool staged_plan(const LayoutGeom& geo, StagedPlan* sp, bool allow_f4 = false);
// Scratch bytes of the staged path for rows_a activation rows (conv: output
// pixels) and N weight rows; 0 if the layout cannot take it.
int64_t staged_scratch_bytes(const LayoutGeom& geo, int64_t rows_a, int64_t N);
// Expansion kernels and the GEMM on `st`; cudaErrorNotSupported if the
// scratch is too small.
cudaError_t launch_staged(const LayoutGeom& geo, const MmaArgs& a, void* scratch, size_t scratch_bytes,
                          cudaStream_t st);

}  // namespace soniq
