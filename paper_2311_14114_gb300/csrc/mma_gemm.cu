// Mixed-precision GEMM / implicit-GEMM convolution on the sm_103a tensor
// cores (tcgen05 + TMEM + TMA).
//
// What it computes (Sec. 3 "Enabling Low-Cost Fixed-Point Operations";
// Sec. 4.2): for each precision group g, the exact integer dot products
//   Acc_g[m][n] = sum over k in group g of u[m][k] * j[n][k]
// and Y = sum_g s_a * s_w * Acc_g / ((2^na - 1) * 2^(nw - 1)) in fp32.
//
// sm_103a has no integer tcgen05 MMA, so the integer codes ride the floating
// point tensor pipes encoded exactly:
//   * groups with <= 4-bit codes on both sides use kind::f8f6f4 with E4M3
//     operands.  An unsigned code c < 16 stored in a byte as-is is the E4M3
//     value c * 2^-9 (subnormals continue linearly into the first normal
//     binade), so activations need no conversion at all; weights are made
//     unsigned by flipping the sign bit (j + 2^(n-1)) and the epilogue
//     subtracts 2^(n-1) * R_g[m] with R_g the activation row sums;
//   * wider groups use kind::f16 with fp16 operands (exact for |x| <= 2048).
// Products accumulate in fp32 TMEM.  A partial sum is an exact integer while
// its magnitude stays <= 2^24; the host splits a group's K range into
// segments short enough for the worst case, and the epilogue warps drain each
// finished segment into an int32 sum kept in TMEM.
//
// CTA = 128x128 output tile, 14 warps:
//   warp 0      TMA producer: packed weight tiles -> shared memory ring
//   warp 1      MMA issuer (one thread) + TMEM owner
//   warps 2-5   expand the 128 activation rows of each K-stage (a conv gathers
//               its im2col rows here; pixels outside the image are code 0)
//   warps 6-9   expand the 128 weight rows from the TMA ring
//   warps 10-13 segment drains and the epilogue (tcgen05.ld -> fp32 -> fp16)
// A K-stage is 128 bytes of operand per row (128 E4M3 codes or 64 fp16
// codes) in the 128-byte-swizzled K-major layout the MMA descriptors read.
//
// Every wait is bounded; a wait that runs out records an error bit in the
// device error word, raises a CTA-wide abort flag and the CTA winds down
// (in-flight MMAs and TMA copies are waited for, TMEM is freed).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstring>

#include "soniq_device.cuh"
#include "soniq_internal.h"

namespace soniq {
namespace mma {

constexpr int BM = 128;
constexpr int BN = 128;
constexpr int OP_STAGES = 4;
constexpr int W_STAGES = 3;
constexpr int ROW_BYTES = 128;                       // operand bytes per row per K-stage
constexpr int OP_A_BYTES = BM * ROW_BYTES;           // 16 KB
constexpr int OP_B_BYTES = BN * ROW_BYTES;           // 16 KB
constexpr int OP_STAGE_BYTES = OP_A_BYTES + OP_B_BYTES;
constexpr int W_STAGE_BYTES = BN * 128;              // BN rows x (16 * n <= 128) packed bytes
constexpr int NUM_WARPS = 14;
constexpr int NUM_THREADS = NUM_WARPS * 32;
constexpr int WARP_TMA = 0, WARP_MMA = 1, WARP_EXPA = 2, WARP_EXPW = 6, WARP_EPI = 10;

constexpr int SMEM_OP = 0;
constexpr int SMEM_W = SMEM_OP + OP_STAGES * OP_STAGE_BYTES;
constexpr int SMEM_BAR = SMEM_W + W_STAGES * W_STAGE_BYTES;
// barriers: w_full[3] w_empty[3] op_full[4] op_empty[4] seg_full[2] slot_free[2]
//           acc_full rowsum_ready teardown
constexpr int BAR_W_FULL = 0, BAR_W_EMPTY = 3, BAR_OP_FULL = 6, BAR_OP_EMPTY = 10,
              BAR_SEG_FULL = 14, BAR_SLOT_FREE = 16, BAR_ACC_FULL = 18, BAR_ROWSUM = 19,
              BAR_TEARDOWN = 20, NUM_BARS = 21;
constexpr int SMEM_MISC = SMEM_BAR + NUM_BARS * 8;   // tmem base, abort flag
constexpr int SMEM_ROWSUM = (SMEM_MISC + 16 + 15) & ~15;   // int32 [2][128]
constexpr int SMEM_SW = SMEM_ROWSUM + 2 * BM * 4;          // fp32 [2][128]
constexpr int SMEM_TOTAL = SMEM_SW + 2 * BN * 4;
constexpr int SMEM_ALLOC = SMEM_TOTAL + 1024;              // slack for 1024-byte alignment

struct Group {
    int32_t bits_a, bits_w;
    int32_t kind;          // 0: E4M3 codes (offset-binary weights), 1: fp16 codes
    int32_t pa;            // activation codes per tap
    int32_t pw;            // weight codes per row
    int32_t a_off, w_off;
    int32_t n_stages;      // K-stages
    int32_t seg_stages;    // K-stages per exact accumulation segment
    int32_t n_seg;
    int32_t w_offset;      // 2^(nw-1) for kind 0, else 0
    int32_t chunk_base;    // index of the group's first 128-code weight chunk
    float acc_scale;       // 2^18 for kind 0 (E4M3 codes carry 2^-9 each), 1 for kind 1
    float inv_levels;      // 1 / ((2^na - 1) * 2^(nw-1))
};

struct Params {
    CUtensorMap tmw[2];    // packed weights, one box width per group
    const uint8_t* Ap;
    const uint8_t* Wp;
    const float* s_a;
    const float* s_w;
    void* Y;
    int32_t* acc_dbg;
    unsigned* err;
    int64_t M;
    int32_t N;
    int32_t a_row_bytes;
    int32_t conv;
    int32_t H, W, P, Q, R, S, sh, sw, ph, pw;
    int32_t s_a_per_row;
    int32_t out_bf16;
    uint32_t flags;
    int32_t seg_group;     // group accumulated in drained segments, or -1
    int32_t tmem_cols;     // 256 or 512
    int32_t acc_col[2];    // TMEM column of each group's accumulator (non-segmented)
    int32_t total_stages;
    int32_t total_chunks;
    long long timeout_ns;
    Group g[2];
};

// ---- small PTX wrappers ------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ long long globaltimer() {
    long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(bar),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: gives up when the CTA is aborting or after timeout_ns; on a
// timeout it records the error and raises the abort flag.
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             const Params& p) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = globaltimer();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer() - t0 > p.timeout_ns) {
            *abort_flag = 1;
            atomicOr(p.err, 1u);
            return false;
        }
    }
}

__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// 128-byte-swizzle K-major shared-memory matrix descriptor: 8-row x 128-byte
// atoms stacked along M/N every 1024 bytes.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;              // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;    // stride byte offset: next 8-row atom
    d |= (uint64_t)1 << 46;              // descriptor version
    d |= (uint64_t)2 << 61;              // SWIZZLE_128B
    return d;
}

// Instruction descriptor: fp32 accumulator, A/B format 0 (E4M3 for
// kind::f8f6f4, F16 for kind::f16), both K-major, N = BN, M = BM.
constexpr uint32_t IDESC = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ void mma_f8(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(IDESC), "r"(acc));
}

__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(IDESC), "r"(acc));
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

#define SONIQ_R32(r)                                                                                   \
    "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),   \
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),      \
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),    \
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),    \
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
#define SONIQ_W32(r)                                                                                   \
    "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), \
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), \
        "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), \
        "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])

// 32 consecutive TMEM columns of this thread's lane.  The load and its wait
// sit in one asm statement: the destination registers are undefined until
// tcgen05.wait::ld, so no instruction may read them in between.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : SONIQ_R32(r)
        : "r"(taddr)
        : "memory");
}

// Likewise the store keeps reading its source registers until tcgen05.wait::st.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n\t"
        "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
        SONIQ_W32(r)
        : "memory");
}

// Swizzled byte offset of 16-byte chunk `chunk` of operand row `row`.
__device__ __forceinline__ uint32_t sw128_off(uint32_t row, uint32_t chunk) {
    return row * 128u + ((chunk ^ (row & 7u)) << 4);
}

// ---- stage bookkeeping -------------------------------------------------------

struct StageInfo {
    int g;        // group
    int ls;       // stage index inside the group
    int kind;
    int kb0;      // first 32-code block of the stage inside the group's weight K range
    int nblk;     // blocks per stage: 4 (E4M3) or 2 (fp16)
};

__device__ __forceinline__ StageInfo stage_info(const Params& p, int s) {
    StageInfo si;
    si.g = s < p.g[0].n_stages ? 0 : 1;
    si.ls = si.g ? s - p.g[0].n_stages : s;
    si.kind = p.g[si.g].kind;
    si.nblk = si.kind == 0 ? 4 : 2;
    si.kb0 = si.ls * si.nblk;
    return si;
}

// ---- activation-side loads (GEMM rows or im2col gather) -----------------------

// Loads the packed activation words of one K-stage for output row `m` into
// `buf` (block i at buf[i * n]); blocks outside the data are zero.
__device__ __forceinline__ void load_act_stage(const Params& p, const StageInfo& si, int64_t m,
                                               int img, int pp, int qq, uint32_t* buf) {
    const Group& G = p.g[si.g];
    const int n = G.bits_a;
    const int cpt = G.pa >> 5;           // blocks per tap
    const int taps = p.conv ? p.R * p.S : 1;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (i >= si.nblk) break;
        const int kb = si.kb0 + i;
        const uint32_t* src = nullptr;
        if (m < p.M && cpt > 0) {
            const int tap = kb / cpt;
            const int cb = kb - tap * cpt;
            if (tap < taps) {
                if (!p.conv) {
                    src = reinterpret_cast<const uint32_t*>(p.Ap + m * p.a_row_bytes + G.a_off + cb * 4 * n);
                } else {
                    const int r = tap / p.S, s = tap - (tap / p.S) * p.S;
                    const int h = pp * p.sh - p.ph + r, w = qq * p.sw - p.pw + s;
                    if (h >= 0 && h < p.H && w >= 0 && w < p.W)
                        src = reinterpret_cast<const uint32_t*>(
                            p.Ap + (((int64_t)img * p.H + h) * p.W + w) * p.a_row_bytes + G.a_off + cb * 4 * n);
                }
            }
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (q >= n) break;
            buf[i * 8 + q] = src ? __ldg(src + q) : 0u;
        }
    }
}

// ---- expansion into the swizzled operand tile --------------------------------

// Activation row: unsigned codes.  E4M3: the byte is the code (value c*2^-9);
// fp16: 1024 + c - 1024.
__device__ __forceinline__ uint32_t expand_act_stage(const StageInfo& si, int n, const uint32_t* buf,
                                                     uint8_t* tile, int row) {
    uint32_t rsum = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (i >= si.nblk) break;
        uint32_t o[8];
        block_to_bytes_n(n, buf + i * 8, o);
        if (si.kind == 0) {
#pragma unroll
            for (int t = 0; t < 8; ++t) rsum = __dp4a(o[t], 0x01010101u, rsum);
            *reinterpret_cast<uint4*>(tile + sw128_off(row, 2 * i)) = make_uint4(o[0], o[1], o[2], o[3]);
            *reinterpret_cast<uint4*>(tile + sw128_off(row, 2 * i + 1)) = make_uint4(o[4], o[5], o[6], o[7]);
        } else {
            const __half2 bias = __half2half2(__ushort_as_half((unsigned short)0x6400u));
            uint32_t h[16];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                uint32_t lo, hi;
                bytes_to_magic_half2(o[t], lo, hi);
                h[2 * t] = half2_sub(lo, bias);
                h[2 * t + 1] = half2_sub(hi, bias);
            }
#pragma unroll
            for (int c = 0; c < 4; ++c)
                *reinterpret_cast<uint4*>(tile + sw128_off(row, 4 * i + c)) =
                    make_uint4(h[4 * c], h[4 * c + 1], h[4 * c + 2], h[4 * c + 3]);
        }
    }
    return rsum;
}

// Weight row: n-bit two's complement -> offset binary (sign-bit flip).
// E4M3: the offset-binary byte is the code; fp16: 1024 + (j + 2^(n-1)) - (1024 + 2^(n-1)) = j.
__device__ __forceinline__ void expand_w_stage(const StageInfo& si, int n, const uint32_t* buf,
                                               uint8_t* tile, int row) {
    const uint32_t flip = sign_flip_mask(n);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (i >= si.nblk) break;
        uint32_t o[8];
        block_to_bytes_n(n, buf + i * 8, o);
#pragma unroll
        for (int t = 0; t < 8; ++t) o[t] ^= flip;
        if (si.kind == 0) {
            *reinterpret_cast<uint4*>(tile + sw128_off(row, 2 * i)) = make_uint4(o[0], o[1], o[2], o[3]);
            *reinterpret_cast<uint4*>(tile + sw128_off(row, 2 * i + 1)) = make_uint4(o[4], o[5], o[6], o[7]);
        } else {
            const __half2 bias = __half2half2(__ushort_as_half((unsigned short)(0x6400u + (1u << (n - 1)))));
            uint32_t h[16];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                uint32_t lo, hi;
                bytes_to_magic_half2(o[t], lo, hi);
                h[2 * t] = half2_sub(lo, bias);
                h[2 * t + 1] = half2_sub(hi, bias);
            }
#pragma unroll
            for (int c = 0; c < 4; ++c)
                *reinterpret_cast<uint4*>(tile + sw128_off(row, 4 * i + c)) =
                    make_uint4(h[4 * c], h[4 * c + 1], h[4 * c + 2], h[4 * c + 3]);
        }
    }
}

// ---- the kernel ----------------------------------------------------------------

__global__ void __launch_bounds__(NUM_THREADS, 1) mp_mma_kernel(const __grid_constant__ Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t m0 = (int64_t)blockIdx.y * BM;
    const int n0 = blockIdx.x * BN;

    uint32_t bar0 = smem_u32(smem + SMEM_BAR);
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + SMEM_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + SMEM_MISC + 4);
    int32_t* rowsum_s = reinterpret_cast<int32_t*>(smem + SMEM_ROWSUM);
    float* sw_s = reinterpret_cast<float*>(smem + SMEM_SW);

    if (threadIdx.x == 0) {
        for (int i = 0; i < W_STAGES; ++i) {
            mbar_init(bar(BAR_W_FULL + i), 1);
            mbar_init(bar(BAR_W_EMPTY + i), 4);
        }
        for (int i = 0; i < OP_STAGES; ++i) {
            mbar_init(bar(BAR_OP_FULL + i), 8);
            mbar_init(bar(BAR_OP_EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(BAR_SEG_FULL + i), 1);
            mbar_init(bar(BAR_SLOT_FREE + i), 4);
        }
        mbar_init(bar(BAR_ACC_FULL), 1);
        mbar_init(bar(BAR_ROWSUM), 4);
        mbar_init(bar(BAR_TEARDOWN), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == WARP_MMA) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(p.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (warp >= WARP_EPI) {
        // scale of each output column and group, with the level counts folded in
        const int c = threadIdx.x - WARP_EPI * 32;
        const int n = n0 + c;
#pragma unroll
        for (int g = 0; g < 2; ++g)
            sw_s[g * BN + c] = n < p.N ? __ldg(p.s_w + (int64_t)n * 2 + g) * p.g[g].inv_levels : 0.0f;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == WARP_TMA) {
        // ------------------------------------------------------------------ TMA
        if (lane == 0) {
            int issued = 0;
            for (int ci = 0; ci < p.total_chunks; ++ci) {
                const int slot = ci % W_STAGES;
                if (!wait_bounded(bar(BAR_W_EMPTY + slot), ((ci / W_STAGES) & 1) ^ 1, abort_flag, p)) break;
                const int g = ci < p.g[1].chunk_base ? 0 : 1;
                const Group& G = p.g[g];
                const int c = ci - G.chunk_base;
                const uint32_t bytes = (uint32_t)BN * 16u * (uint32_t)G.bits_w;
                mbar_arrive_expect_tx(bar(BAR_W_FULL + slot), bytes);
                tma_load_2d(smem_u32(smem + SMEM_W + slot * W_STAGE_BYTES), &p.tmw[g],
                            G.w_off + c * 16 * G.bits_w, n0, bar(BAR_W_FULL + slot));
                ++issued;
            }
            // copies still in flight must land before the CTA's memory is released
            for (int ci = issued - W_STAGES < 0 ? 0 : issued - W_STAGES; ci < issued; ++ci) {
                volatile int no_abort = 0;
                wait_bounded(bar(BAR_W_FULL + ci % W_STAGES), (ci / W_STAGES) & 1, &no_abort, p);
            }
        }
    } else if (warp == WARP_MMA) {
        // ------------------------------------------------------------------ MMA
        if (lane == 0) {
            bool ok = true;
            for (int s = 0; s < p.total_stages && ok; ++s) {
                const StageInfo si = stage_info(p, s);
                const Group& G = p.g[si.g];
                const int slot = s % OP_STAGES;
                uint32_t col;
                bool first;
                bool seg_end = false;
                int seg = 0;
                if (si.g == p.seg_group) {
                    seg = si.ls / G.seg_stages;
                    const int in_seg = si.ls - seg * G.seg_stages;
                    first = in_seg == 0;
                    seg_end = in_seg == G.seg_stages - 1 || si.ls == G.n_stages - 1;
                    col = (uint32_t)(BN + (seg & 1) * BN);
                    if (first && seg >= 2) {
                        if (!wait_bounded(bar(BAR_SLOT_FREE + (seg & 1)), ((seg >> 1) - 1) & 1, abort_flag, p)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                    }
                } else {
                    first = si.ls == 0;
                    col = (uint32_t)p.acc_col[si.g];
                }
                if (!wait_bounded(bar(BAR_OP_FULL + slot), (s / OP_STAGES) & 1, abort_flag, p)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a_addr = smem_u32(smem + SMEM_OP + slot * OP_STAGE_BYTES);
                const uint32_t b_addr = a_addr + OP_A_BYTES;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const uint64_t ad = sw128_desc(a_addr + 32 * k), bd = sw128_desc(b_addr + 32 * k);
                    const uint32_t acc = (first && k == 0) ? 0u : 1u;
                    if (si.kind == 0) mma_f8(tmem_base + col, ad, bd, acc);
                    else mma_f16(tmem_base + col, ad, bd, acc);
                }
                mma_commit(bar(BAR_OP_EMPTY + slot));
                if (seg_end) mma_commit(bar(BAR_SEG_FULL + (seg & 1)));
            }
            if (ok) mma_commit(bar(BAR_ACC_FULL));
            // all issued MMAs complete before TMEM and shared memory are released
            mma_commit(bar(BAR_TEARDOWN));
            volatile int no_abort = 0;
            wait_bounded(bar(BAR_TEARDOWN), 0, &no_abort, p);
        }
    } else if (warp < WARP_EPI) {
        // ------------------------------------------------------------ expanders
        const bool is_a = warp < WARP_EXPW;
        const int row = threadIdx.x - (is_a ? WARP_EXPA : WARP_EXPW) * 32;
        if (is_a) {
            const int64_t m = m0 + row;
            int img = 0, pp = 0, qq = 0;
            if (p.conv && m < p.M) {
                const int64_t pq = (int64_t)p.P * p.Q;
                img = (int)(m / pq);
                const int rem = (int)(m - (int64_t)img * pq);
                pp = rem / p.Q;
                qq = rem - pp * p.Q;
            }
            uint32_t cur[32], nxt[32];
            if (p.total_stages > 0) load_act_stage(p, stage_info(p, 0), m, img, pp, qq, cur);
            uint32_t rsum = 0;
            for (int s = 0; s < p.total_stages; ++s) {
                const StageInfo si = stage_info(p, s);
                if (s + 1 < p.total_stages) load_act_stage(p, stage_info(p, s + 1), m, img, pp, qq, nxt);
                const int slot = s % OP_STAGES;
                if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_OP_EMPTY + slot), ((s / OP_STAGES) & 1) ^ 1,
                                                            abort_flag, p)))
                    break;
                rsum += expand_act_stage(si, p.g[si.g].bits_a, cur, smem + SMEM_OP + slot * OP_STAGE_BYTES, row);
                if (si.ls == p.g[si.g].n_stages - 1) {
                    rowsum_s[si.g * BM + row] = (int32_t)rsum;
                    rsum = 0;
                }
                fence_proxy_async();
                __syncwarp();
                const bool drop = (p.flags & SONIQ_FLAG_TEST_DROP_ARRIVE) && s == 0 && warp == WARP_EXPA;
                if (lane == 0 && !drop) mbar_arrive(bar(BAR_OP_FULL + slot));
#pragma unroll
                for (int i = 0; i < 32; ++i) cur[i] = nxt[i];
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(BAR_ROWSUM));
        } else {
            int ci = 0;
            for (int s = 0; s < p.total_stages; ++s) {
                const StageInfo si = stage_info(p, s);
                const Group& G = p.g[si.g];
                const int n = G.bits_w;
                const int half = si.kind == 0 ? 0 : (si.ls & 1);
                const int wslot = ci % W_STAGES;
                if (half == 0 &&
                    !__all_sync(0xffffffffu, wait_bounded(bar(BAR_W_FULL + wslot), (ci / W_STAGES) & 1, abort_flag, p)))
                    break;
                // this stage's blocks of the packed row: 128 codes (E4M3) or one half of them (fp16)
                uint32_t buf[32];
                const uint32_t* src = reinterpret_cast<const uint32_t*>(
                    smem + SMEM_W + wslot * W_STAGE_BYTES + row * 16 * n + half * 8 * n);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    if (i >= si.nblk) break;
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        if (q >= n) break;
                        buf[i * 8 + q] = src[i * n + q];
                    }
                }
                const int slot = s % OP_STAGES;
                if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_OP_EMPTY + slot), ((s / OP_STAGES) & 1) ^ 1,
                                                            abort_flag, p)))
                    break;
                expand_w_stage(si, n, buf, smem + SMEM_OP + slot * OP_STAGE_BYTES + OP_A_BYTES, row);
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(BAR_OP_FULL + slot));
                // The packed slot goes back to the TMA producer only after its words have
                // been consumed by the expansion above: releasing it right after the
                // shared-memory loads let the next TMA copy land before those loads had
                // read the slot (an intermittent wrong 32-row block of weights).
                if (si.kind == 0 || half == 1) {
                    if (lane == 0) mbar_arrive(bar(BAR_W_EMPTY + wslot));
                    ++ci;
                }
            }
        }
    } else {
        // ---------------------------------------------------- drains + epilogue
        const int quad = warp & 3;                 // TMEM lanes 32*quad .. +31
        const int row = quad * 32 + lane;
        const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16);
        bool ok = true;
        const int gs = p.seg_group;
        if (gs >= 0) {
            const uint32_t sum_col = 3 * BN;
            for (int i = 0; i < p.g[gs].n_seg && ok; ++i) {
                if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_SEG_FULL + (i & 1)), (i >> 1) & 1, abort_flag, p))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t ring_col = BN + (i & 1) * BN;
#pragma unroll 1
                for (int cc = 0; cc < BN / 32; ++cc) {
                    uint32_t v[32], s[32];
                    tmem_ld32(lane_base + ring_col + cc * 32, v);
                    if (i > 0) tmem_ld32(lane_base + sum_col + cc * 32, s);
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int32_t x = __float2int_rn(__uint_as_float(v[j]) * p.g[gs].acc_scale);
                        s[j] = (uint32_t)((i > 0 ? (int32_t)s[j] : 0) + x);
                    }
                    tmem_st32(lane_base + sum_col + cc * 32, s);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(BAR_SLOT_FREE + (i & 1)));
            }
        }
        // warp-uniform outcomes: the TMEM loads below are .sync.aligned
        if (ok) ok = __all_sync(0xffffffffu, wait_bounded(bar(BAR_ACC_FULL), 0, abort_flag, p));
        if (ok) ok = __all_sync(0xffffffffu, wait_bounded(bar(BAR_ROWSUM), 0, abort_flag, p));
        if (ok) {
            tc_fence_after();
            const int64_t m = m0 + row;
            float sa[2];
#pragma unroll
            for (int g = 0; g < 2; ++g)
                sa[g] = m < p.M ? (p.s_a_per_row ? __ldg(p.s_a + m * 2 + g) : __ldg(p.s_a + g)) : 0.0f;
            int32_t corr[2];
#pragma unroll
            for (int g = 0; g < 2; ++g) corr[g] = p.g[g].w_offset * rowsum_s[g * BM + row];
#pragma unroll 1
            for (int cc = 0; cc < BN / 32; ++cc) {
                int32_t acc[2][32];
#pragma unroll
                for (int g = 0; g < 2; ++g) {
                    uint32_t v[32];
                    if (p.g[g].n_stages == 0) {
#pragma unroll
                        for (int j = 0; j < 32; ++j) acc[g][j] = 0;
                        continue;
                    }
                    if (g == gs) {
                        tmem_ld32(lane_base + 3 * BN + cc * 32, v);
#pragma unroll
                        for (int j = 0; j < 32; ++j) acc[g][j] = (int32_t)v[j] - corr[g];
                    } else {
                        tmem_ld32(lane_base + p.acc_col[g] + cc * 32, v);
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            acc[g][j] = __float2int_rn(__uint_as_float(v[j]) * p.g[g].acc_scale) - corr[g];
                    }
                }
                const int nb = n0 + cc * 32;
                if (m < p.M) {
                    if (p.acc_dbg != nullptr) {
#pragma unroll
                        for (int g = 0; g < 2; ++g) {
                            int32_t* dst = p.acc_dbg + ((int64_t)g * p.M + m) * p.N;
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (nb + j < p.N) dst[nb + j] = acc[g][j];
                        }
                    }
                    float y[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int c = cc * 32 + j;
                        y[j] = fmaf(sa[1] * sw_s[BN + c], (float)acc[1][j], sa[0] * sw_s[c] * (float)acc[0][j]);
                    }
                    if (p.out_bf16) {
                        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.Y) + m * p.N;
                        if (nb + 32 <= p.N && (p.N & 7) == 0) {
#pragma unroll
                            for (int v8 = 0; v8 < 4; ++v8) {
                                uint32_t w[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    __nv_bfloat162 h = __floats2bfloat162_rn(y[v8 * 8 + 2 * e], y[v8 * 8 + 2 * e + 1]);
                                    w[e] = *reinterpret_cast<uint32_t*>(&h);
                                }
                                *reinterpret_cast<uint4*>(dst + nb + v8 * 8) = make_uint4(w[0], w[1], w[2], w[3]);
                            }
                        } else {
                            for (int j = 0; j < 32; ++j)
                                if (nb + j < p.N) dst[nb + j] = __float2bfloat16_rn(y[j]);
                        }
                    } else {
                        __half* dst = reinterpret_cast<__half*>(p.Y) + m * p.N;
                        if (nb + 32 <= p.N && (p.N & 7) == 0) {
#pragma unroll
                            for (int v8 = 0; v8 < 4; ++v8) {
                                uint32_t w[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    __half2 h = __floats2half2_rn(y[v8 * 8 + 2 * e], y[v8 * 8 + 2 * e + 1]);
                                    w[e] = *reinterpret_cast<uint32_t*>(&h);
                                }
                                *reinterpret_cast<uint4*>(dst + nb + v8 * 8) = make_uint4(w[0], w[1], w[2], w[3]);
                            }
                        } else {
                            for (int j = 0; j < 32; ++j)
                                if (nb + j < p.N) dst[nb + j] = __float2half_rn(y[j]);
                        }
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == WARP_MMA) {
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(p.tmem_cols)
                     : "memory");
    }
}

// ---- host side -----------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

// Per-group planning: operand kind, K-stages and exact accumulation segments.
bool plan_group(const GroupGeom& G, Group& out) {
    out.bits_a = G.bits_a;
    out.bits_w = G.bits_w;
    out.pa = G.pa;
    out.pw = G.pw;
    out.a_off = G.a_off;
    out.w_off = G.w_off;
    out.kind = (G.bits_a <= 4 && G.bits_w <= 4) ? 0 : 1;
    const int codes_per_stage = out.kind == 0 ? 128 : 64;
    out.n_stages = G.pw / codes_per_stage;
    // worst-case |product|: offset-binary weights for E4M3, signed for fp16
    const int64_t la = (1 << G.bits_a) - 1;
    const int64_t maxprod = out.kind == 0 ? la * ((1 << G.bits_w) - 1) : la * (1 << (G.bits_w - 1));
    const int64_t seg_codes = maxprod > 0 ? (int64_t(1) << 24) / maxprod : (int64_t(1) << 24);
    int64_t seg_stages = seg_codes / codes_per_stage;
    if (seg_stages < 1) return false;
    if (seg_stages > out.n_stages) seg_stages = out.n_stages > 0 ? out.n_stages : 1;
    out.seg_stages = (int32_t)seg_stages;
    out.n_seg = out.n_stages > 0 ? (int32_t)((out.n_stages + seg_stages - 1) / seg_stages) : 0;
    out.w_offset = out.kind == 0 ? (1 << (G.bits_w - 1)) : 0;
    out.acc_scale = out.kind == 0 ? 262144.0f : 1.0f;   // 2^18
    out.inv_levels = (float)(1.0 / ((double)la * (double)(1 << (G.bits_w - 1))));
    return true;
}

}  // namespace mma

soniq_status mma_check(const LayoutGeom& geo) {
    mma::Group g0, g1;
    if (!mma::plan_group(geo.g[0], g0) || !mma::plan_group(geo.g[1], g1)) return SONIQ_ERR_UNSUPPORTED;
    if (g0.n_seg > 1 && g1.n_seg > 1) return SONIQ_ERR_UNSUPPORTED;
    return SONIQ_OK;
}

cudaError_t launch_mma(const LayoutGeom& geo, const MmaArgs& a, cudaStream_t st) {
    using namespace mma;
    Params p;
    memset(&p, 0, sizeof(p));
    if (!plan_group(geo.g[0], p.g[0]) || !plan_group(geo.g[1], p.g[1])) return cudaErrorNotSupported;
    p.Ap = a.Ap;
    p.Wp = a.Wp;
    p.s_a = a.s_a;
    p.s_w = a.s_w;
    p.Y = a.Y;
    p.acc_dbg = a.acc_dbg;
    p.err = device_error_word();
    if (p.err == nullptr) return cudaErrorUnknown;
    p.M = a.M;
    p.N = a.N;
    p.a_row_bytes = geo.a_row_bytes;
    p.conv = a.conv;
    p.H = a.H; p.W = a.W; p.P = a.P; p.Q = a.Q; p.R = a.R; p.S = a.S;
    p.sh = a.sh; p.sw = a.sw; p.ph = a.ph; p.pw = a.pw;
    p.s_a_per_row = a.s_a_per_row;
    p.out_bf16 = a.out_bf16;
    p.flags = a.flags;
    p.timeout_ns = 2000000000LL;
    p.seg_group = p.g[0].n_seg > 1 ? 0 : (p.g[1].n_seg > 1 ? 1 : -1);
    if (p.seg_group < 0) {
        p.tmem_cols = 256;
        p.acc_col[0] = 0;
        p.acc_col[1] = BN;
    } else {
        p.tmem_cols = 512;
        p.acc_col[p.seg_group ^ 1] = 0;
        p.acc_col[p.seg_group] = 3 * BN;   // the drained int32 sum
    }
    p.total_stages = p.g[0].n_stages + p.g[1].n_stages;
    p.g[0].chunk_base = 0;
    p.g[1].chunk_base = geo.g[0].pw / 128;
    p.total_chunks = geo.g[0].pw / 128 + geo.g[1].pw / 128;

    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return cudaErrorNotSupported;
    for (int g = 0; g < 2; ++g) {
        const int box_x = 16 * (geo.g[g].pw > 0 ? geo.g[g].bits_w : 1);
        cuuint64_t dims[2] = {(cuuint64_t)geo.w_row_bytes, (cuuint64_t)a.N};
        cuuint64_t strides[1] = {(cuuint64_t)geo.w_row_bytes};
        cuuint32_t box[2] = {(cuuint32_t)box_x, (cuuint32_t)BN};
        cuuint32_t estr[2] = {1, 1};
        CUresult r = enc(&p.tmw[g], CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(a.Wp), dims, strides, box,
                         estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    static bool attr_done[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(mp_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_ALLOC);
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    dim3 grid((unsigned)((a.N + BN - 1) / BN), (unsigned)((a.M + BM - 1) / BM));
    mp_mma_kernel<<<grid, NUM_THREADS, SMEM_ALLOC, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

}  // namespace soniq
