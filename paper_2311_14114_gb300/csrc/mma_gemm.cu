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
//   * wider groups use kind::f16 with fp16 operands (exact for |x| <= 2048);
//     activations are centred (u - 2^(n-1)), which halves the worst-case
//     product, and the epilogue adds back 2^(n-1) * C_g[n] with C_g the
//     weight column sums.
// Products accumulate in fp32 TMEM.  A partial sum is an exact integer while
// its magnitude stays <= 2^24; the host splits a group's K range into
// segments short enough for the worst case, and the epilogue warps drain each
// finished segment into an int32 sum kept in TMEM.
//
// Data movement.  K is walked in chunks of 128 codes.  Each chunk's packed
// activation rows (128 x 16*na bytes) and packed weight rows (128 x 16*nw
// bytes) land in one slot of a byte ring in shared memory whose slots are
// sized per precision group, so low-bit chunks keep many copies in flight.
// Weights always arrive by TMA; activations by TMA when the rows allow it
// (GEMM with 128-code padding), otherwise the producer warp gathers them with
// cp.async (implicit-GEMM conv: one pixel row per output row and tap, zero
// fill outside the image).  Packed tiles with 2-, 4- or 8-bit codes use the
// TMA 32/64/128-byte swizzle so the converters read them without bank
// conflicts.
//
// CTA = 128x128 output tile, 17 warps:
//   warp 0      MMA issuer (one thread) + TMEM owner
//   warps 1-4   producers: ring space and TMA copies (warp 1, lane 0); in
//               gather mode every producer thread also copies one activation
//               row of each chunk with cp.async
//   warps 5-8   convert the 128 activation rows of each K-stage
//   warps 9-12  convert the 128 weight rows
//   warps 13-16 segment drains and the epilogue (tcgen05.ld -> fp32 -> fp16)
// A K-stage is 128 bytes of MMA operand per row (128 E4M3 codes or 64 fp16
// codes) in the 128-byte-swizzled K-major layout the MMA descriptors read;
// an E4M3 chunk is one stage, an fp16 chunk two.
//
// Converters run one specialised loop per precision group (bit width and
// operand kind fixed at compile time), so the inner loop has no dispatch.
//
// Every wait is bounded; a wait that runs out records an error bit in the
// device error word, raises a CTA-wide abort flag and the CTA winds down
// (in-flight MMAs and copies are waited for, TMEM is freed).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstring>

#include "soniq_device.cuh"
#include "soniq_internal.h"

namespace soniq {
namespace mma {

constexpr int BM = 128;
constexpr int BN = 128;
constexpr int OP_STAGES = 3;
constexpr int ROW_BYTES = 128;                       // operand bytes per row per K-stage
constexpr int OP_A_BYTES = BM * ROW_BYTES;           // 16 KB
constexpr int OP_B_BYTES = BN * ROW_BYTES;           // 16 KB
constexpr int OP_STAGE_BYTES = OP_A_BYTES + OP_B_BYTES;
constexpr int PK_BYTES = 96 * 1024;                  // packed chunk ring
constexpr int PK_SLOTS = 16;                         // chunks in flight at most
constexpr int A_TMEM_COL = 256;                      // activation stages in TMEM (32 columns each)
constexpr int NUM_WARPS = 17;
constexpr int NUM_THREADS = NUM_WARPS * 32;
constexpr int WARP_MMA = 0, WARP_PROD = 1, WARP_CVA = 5, WARP_CVW = 9, WARP_EPI = 13;
constexpr int NUM_PROD_THREADS = 128;

constexpr int SMEM_OP = 0;
constexpr int SMEM_PK = SMEM_OP + OP_STAGES * OP_STAGE_BYTES;
constexpr int SMEM_BAR = SMEM_PK + PK_BYTES;
constexpr int BAR_PK_FULL = 0, BAR_PK_EMPTY = 16, BAR_OP_FULL = 32, BAR_OP_EMPTY = 35,
              BAR_SEG_FULL = 38, BAR_SLOT_FREE = 40, BAR_ACC_FULL = 42, BAR_ROWSUM = 43,
              BAR_TEARDOWN = 44, BAR_HALO = 45, NUM_BARS = 46;
constexpr int SMEM_MISC = SMEM_BAR + NUM_BARS * 8;         // tmem base, abort flag, a zero word
constexpr int SMEM_ROWSUM = (SMEM_MISC + 16 + 15) & ~15;   // int32 [2][128]
constexpr int SMEM_SW = SMEM_ROWSUM + 2 * BM * 4;          // fp32 [2][128]
constexpr int SMEM_CS = SMEM_SW + 2 * BN * 4;              // int32 [2][128] weight column sums
constexpr int SMEM_TOTAL = SMEM_CS + 2 * BN * 4;
constexpr int SMEM_ALLOC = SMEM_TOTAL + 1024;              // slack for 1024-byte alignment

struct Group {
    int32_t bits_a, bits_w;
    int32_t kind;          // 0: E4M3 codes (offset-binary weights), 1: fp16 codes
    int32_t pa;            // activation codes per tap
    int32_t pw;            // weight codes per row
    int32_t a_off, w_off;  // byte offsets of the group in packed rows
    int32_t n_stages;      // K-stages
    int32_t seg_stages;    // K-stages per exact accumulation segment
    int32_t n_seg;
    int32_t w_offset;      // kind 0: weights carry +2^(nw-1) (offset binary), else 0
    int32_t a_offset;      // kind 1: activations carry -2^(na-1) (centred), else 0
    int32_t chunk_base;    // index of the group's first 128-code chunk
    int32_t a_bytes;       // packed activation bytes of one chunk (128 rows)
    int32_t w_bytes;       // packed weight bytes of one chunk (128 rows)
    int32_t copy_bytes;    // cp.async width of the activation gather (4, 8 or 16)
    float acc_scale;       // 2^18 for kind 0 (E4M3 codes carry 2^-9 each), 1 for kind 1
    float inv_levels;      // 1 / ((2^na - 1) * 2^(nw-1))
};

struct Params {
    CUtensorMap tmw[2];    // packed weights, one box width per group
    CUtensorMap tma[2];    // packed activations (used when a_tma)
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
    int32_t a_tma;         // 1: activation chunks by TMA, 0: cp.async gather
    int32_t a_halo;        // conv: 1 = each CTA loads its input rows once (the halo) and the
                           // activation converters read every tap from it; 0 = per-chunk gather
    int32_t halo_stride;   // bytes per halo pixel in shared memory (an odd multiple of 16)
    int32_t halo_copy;     // cp.async width of the halo load (4, 8 or 16)
    int32_t ring_cap;      // bytes of the packed ring; the halo follows it
    int32_t H, W, P, Q, R, S, sh, sw, ph, pw;
    int32_t s_a_per_row;
    int32_t out_bf16;
    uint32_t flags;
    int32_t seg_group;     // group accumulated in drained segments, or -1
    int32_t tmem_cols;     // 256 or 512
    int32_t a_in_tmem;     // 1: activation stages live in TMEM columns A_TMEM_COL.. (no segments)
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

// The CTA-wide abort flag lives in shared memory; it is read and written
// with explicit shared-space volatile accesses.
__device__ __forceinline__ int abort_raised(uint32_t flag) {
    int v;
    asm volatile("ld.volatile.shared.u32 %0, [%1];" : "=r"(v) : "r"(flag) : "memory");
    return v;
}

__device__ __forceinline__ void raise_abort(uint32_t flag) {
    asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(flag), "r"(1) : "memory");
}

// Bounded wait: polls the barrier tightly and only every 64 polls looks at the
// abort flag and the clock, so a completed phase is seen within one poll.
// Gives up when the CTA is aborting or after timeout_ns; on a timeout it
// records the error and raises the abort flag.
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, uint32_t abort_flag,
                                             const Params& p) {
    if (mbar_try_wait(bar, parity)) return true;
    long long t0 = 0;
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 63u) == 0u) {
            if (abort_raised(abort_flag)) return false;
            const long long t = globaltimer();
            if (t0 == 0) {
                t0 = t;
            } else if (t - t0 > p.timeout_ns) {
                raise_abort(abort_flag);
                atomicOr(p.err, 1u);
                return false;
            }
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

// A operand from TMEM (columns of this stage), B from shared memory.
__device__ __forceinline__ void mma_f8_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(IDESC), "r"(acc));
}

__device__ __forceinline__ void mma_f16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(IDESC), "r"(acc));
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


#define SONIQ_R16(r)                                                                                   \
    "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),   \
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
#define SONIQ_W16(r)                                                                                   \
    "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), \
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])

// 16 consecutive TMEM columns of this thread's lane (load + wait in one statement).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : SONIQ_R16(r)
        : "r"(taddr)
        : "memory");
}

// Two 16-column loads (one per accumulator) and one wait, in one statement so
// that no register is read before the wait.
__device__ __forceinline__ void tmem_ld16x2(uint32_t ta, uint32_t tb, uint32_t (&a)[16], uint32_t (&b)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%32];\n\t"
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%33];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : SONIQ_R16(a), SONIQ_R16(b)
        : "r"(ta), "r"(tb)
        : "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n\t"
        "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
        SONIQ_W16(r)
        : "memory");
}


// cp.async copies of 4, 8 or 16 bytes; src_bytes = 0 zero-fills the destination.
__device__ __forceinline__ void cp_async(uint32_t dst, const void* src, int bytes, uint32_t src_bytes) {
    if (bytes == 16)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
    else if (bytes == 8)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}

// Arrives on `bar` once all of this thread's earlier cp.async copies have landed.
__device__ __forceinline__ void cp_async_arrive(uint32_t bar) {
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

// XOR applied to the 16-byte chunk index of a packed row of n-bit codes
// (16*n bytes per 128 codes): the TMA 32/64/128-byte swizzle for n = 2/4/8,
// none otherwise.  Address bits [4, 4+k) are XORed with bits [7, 7+k).
__device__ __forceinline__ uint32_t pk_xor(int n, uint32_t row) {
    return (n == 2 || n == 4 || n == 8) ? ((row * (uint32_t)n) >> 3) & (uint32_t)(n - 1) : 0u;
}

// Byte offset of 16-byte chunk `chunk` of operand row `row` in the MMA tile
// (128-byte swizzle: 8-row x 128-byte atoms).
__device__ __forceinline__ uint32_t sw128_off(uint32_t row, uint32_t chunk) {
    return row * 128u + ((chunk ^ (row & 7u)) << 4);
}

// ---- chunk bookkeeping ---------------------------------------------------------

// Chunk sizes of the packed ring, held in registers (hot loops never index the
// parameter block with a runtime value).
struct RingGeo {
    int n0;              // chunks of group 0
    int total;           // chunks of both groups
    uint32_t sz0, sz1;   // slot bytes of a chunk of group 0 / group 1
    uint32_t cap;        // ring bytes
};

__device__ __forceinline__ RingGeo ring_geo(const Params& p) {
    RingGeo r;
    r.n0 = p.g[1].chunk_base;
    r.total = p.total_chunks;
    r.sz0 = (uint32_t)(p.g[0].a_bytes + p.g[0].w_bytes);
    r.sz1 = (uint32_t)(p.g[1].a_bytes + p.g[1].w_bytes);
    r.cap = (uint32_t)p.ring_cap;
    return r;
}

__device__ __forceinline__ uint32_t chunk_size(const RingGeo& r, int ci) { return ci < r.n0 ? r.sz0 : r.sz1; }

// Ring offset of chunk ci+1 from that of chunk ci: slots follow each other and
// wrap to 0 when the next one would not fit.
__device__ __forceinline__ uint32_t ring_next(const RingGeo& r, int ci, uint32_t off) {
    uint32_t nxt = off + chunk_size(r, ci);
    if (ci + 1 < r.total && nxt + chunk_size(r, ci + 1) > r.cap) nxt = 0;
    return nxt;
}

// ---- conversion of packed codes into the MMA operand tile ---------------------

// This row's packed words of one chunk (n 16-byte pieces, swizzled).
template <int N>
__device__ __forceinline__ void read_chunk(uint32_t row_base, uint32_t xr, uint32_t* w) {
#pragma unroll
    for (int j = 0; j < N; ++j) {
        const uint4 v = lds128(row_base + ((j ^ xr) << 4));
        w[4 * j] = v.x;
        w[4 * j + 1] = v.y;
        w[4 * j + 2] = v.z;
        w[4 * j + 3] = v.w;
    }
}

// E4M3 stage: 4 blocks of 32 codes -> 128 bytes.  Activations: the byte is the
// code; weights: sign bit flipped (offset binary).  Returns the code sum.
// Conversions write one stage row (128 bytes) as 32 words `out`, natural K
// order: 16-byte piece c of the row is out[4c .. 4c+3].
template <int N, bool A_SIDE>
__device__ __forceinline__ uint32_t cvt_e4m3(const uint32_t* w, uint32_t* out) {
    uint32_t rsum = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        uint32_t* o = out + 8 * i;
        block_to_bytes<N>(w + i * N, o);
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            if constexpr (A_SIDE) rsum = __dp4a(o[t], 0x01010101u, rsum);
            else o[t] ^= 0x01010101u << (N - 1);
        }
    }
    return rsum;
}

// fp16 stage: blocks 2h, 2h+1 of the chunk -> 64 fp16 values (128 bytes).
// Activations: 1024 + u - 1024; weights: 1024 + (j + 2^(n-1)) - (1024 + 2^(n-1)).
// Both sides subtract 1024 + 2^(n-1): activations become u - 2^(n-1) (centred),
// weights j.  Weights also return the sum of their offset-binary codes.
template <int N, bool A_SIDE>
__device__ __forceinline__ uint32_t cvt_f16(const uint32_t* w, int half, uint32_t* out) {
    const __half2 bias = __half2half2(__ushort_as_half((unsigned short)(0x6400u + (1u << (N - 1)))));
    uint32_t csum = 0;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        uint32_t o[8];
        block_to_bytes<N>(w + (2 * half + i) * N, o);
        uint32_t* h = out + 16 * i;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            uint32_t lo, hi;
            const uint32_t x = A_SIDE ? o[t] : (o[t] ^ (0x01010101u << (N - 1)));
            if constexpr (!A_SIDE) csum = __dp4a(x, 0x01010101u, csum);
            bytes_to_magic_half2(x, lo, hi);
            h[2 * t] = half2_sub(lo, bias);
            h[2 * t + 1] = half2_sub(hi, bias);
        }
    }
    return csum;
}

// A stage row into the 128-byte-swizzled shared-memory operand tile.
__device__ __forceinline__ void store_stage_smem(const uint32_t* out, uint32_t tile, uint32_t row) {
#pragma unroll
    for (int c = 0; c < 8; ++c) sts128(tile + sw128_off(row, c), out[4 * c], out[4 * c + 1], out[4 * c + 2], out[4 * c + 3]);
}

// A stage row into TMEM: this thread's lane, 32 consecutive columns; two
// stores, then one wait for both.
__device__ __forceinline__ void store_stage_tmem(const uint32_t* out, uint32_t taddr) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(out[0]), "r"(out[1]), "r"(out[2]), "r"(out[3]), "r"(out[4]), "r"(out[5]), "r"(out[6]), "r"(out[7]),
        "r"(out[8]), "r"(out[9]), "r"(out[10]), "r"(out[11]), "r"(out[12]), "r"(out[13]), "r"(out[14]), "r"(out[15])
        : "memory");
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n\t"
        "tcgen05.wait::st.sync.aligned;" ::"r"(taddr + 16),
        "r"(out[16]), "r"(out[17]), "r"(out[18]), "r"(out[19]), "r"(out[20]), "r"(out[21]), "r"(out[22]), "r"(out[23]),
        "r"(out[24]), "r"(out[25]), "r"(out[26]), "r"(out[27]), "r"(out[28]), "r"(out[29]), "r"(out[30]), "r"(out[31])
        : "memory");
}

// ---- the input halo of an implicit-GEMM tile -----------------------------------

// The output pixels m0 .. m0 + BM - 1 read input rows from the first one's
// first tap row to the last one's last tap row: one contiguous range of
// pixels [first, end) of the NHWC input (whole rows, images in between).
__device__ __forceinline__ int64_t halo_first(const Params& p, int64_t m0) {
    const int64_t pq = (int64_t)p.P * p.Q;
    const int64_t img = m0 / pq;
    const int pp = (int)((m0 - img * pq) / p.Q);
    int h = pp * p.sh - p.ph;
    if (h < 0) h = 0;
    return (img * p.H + h) * p.W;
}

__device__ __forceinline__ int64_t halo_end(const Params& p, int64_t m0) {
    const int64_t pq = (int64_t)p.P * p.Q;
    const int64_t m_last = (m0 + BM < p.M ? m0 + BM : p.M) - 1;
    const int64_t img = m_last / pq;
    const int pp = (int)((m_last - img * pq) / p.Q);
    int h = pp * p.sh - p.ph + p.R - 1;
    if (h > p.H - 1) h = p.H - 1;
    return (img * p.H + h) * p.W + p.W;
}

// Where an activation converter thread reads its row's codes in the halo.
// For tap (r, s) the input pixel is pix0 + r * W + s (halo-local index);
// bit r of mr / bit s of ms says whether that row / column is in the image.
struct HaloRow {
    uint32_t base;         // shared address of the halo plus the group's byte offset
    int32_t pix0;          // halo-local index of tap (0, 0) (may be negative)
    uint32_t mr, ms;       // in-image masks over filter rows / columns (0 for rows >= M)
    int tap, cb, r, s;     // position of the next block in its group
    uint32_t addr;         // shared address of the current tap's pixel (valid when in)
    bool in;               // the current tap reads real codes
};

__device__ __forceinline__ void halo_tap(const Params& p, HaloRow& hr, int taps) {
    hr.in = hr.tap < taps && ((hr.mr >> hr.r) & 1u) && ((hr.ms >> hr.s) & 1u);
    hr.addr = hr.base + (uint32_t)(hr.pix0 + hr.r * p.W + hr.s) * (uint32_t)p.halo_stride;
}

// This row's 4 blocks of the next chunk (n words each, block i at w[n*i]),
// read from the halo; taps outside the image read code 0.  The tap
// bookkeeping for the four blocks runs first, then all loads issue back to
// back (a tap outside the image loads from the halo base and is zeroed).
template <int N>
__device__ __forceinline__ void read_halo(const Params& p, const Group& G, HaloRow& hr, uint32_t* w) {
    const int taps = p.R * p.S;
    const int cpt = G.pa >> 5;
    const bool vec = N % 4 == 0 && ((hr.base + (uint32_t)G.a_off) & 15u) == 0;
    uint32_t addr[4];
    bool in[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        in[i] = hr.in;
        addr[i] = hr.in ? hr.addr + (uint32_t)G.a_off + (uint32_t)(hr.cb * 4 * N) : hr.base;
        if (++hr.cb == cpt) {
            hr.cb = 0;
            ++hr.tap;
            if (++hr.s == p.S) {
                hr.s = 0;
                ++hr.r;
            }
            halo_tap(p, hr, taps);
        }
    }
    if (vec) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < (N & ~3); j += 4) {
                const uint4 v = lds128(addr[i] + 4 * j);
                w[N * i + j] = in[i] ? v.x : 0u;
                w[N * i + j + 1] = in[i] ? v.y : 0u;
                w[N * i + j + 2] = in[i] ? v.z : 0u;
                w[N * i + j + 3] = in[i] ? v.w : 0u;
            }
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < N; ++j) {
                const uint32_t v = lds32(addr[i] + 4 * j);
                w[N * i + j] = in[i] ? v : 0u;
            }
    }
}

struct CvtCtx {
    RingGeo ring;
    bool drop_first;      // test hook: skip the first operand arrival of this warp
    uint32_t smem;        // shared-memory address of the aligned base
    uint32_t a_tmem;      // TMEM address (lane of this thread's row) of the activation stages, or 0
    uint32_t pk_base;
    uint32_t bar0;
    uint32_t abort_flag;
    int warp, lane;
    uint32_t row;
    int ci;               // next chunk
    int s;                // next operand stage
    uint32_t off;         // ring offset of chunk ci
    bool halo;            // activation side: read taps from the halo
    HaloRow hr;
};

// Converts all chunks of group g for this row: per chunk, waits for its packed
// slot, reads this row's words once, fills 1 (E4M3) or 2 (fp16) operand
// stages, and hands the slot back only after its words are consumed.
template <int N, int KIND, bool A_SIDE>
__device__ __forceinline__ bool convert_group(const Params& p, CvtCtx& cx, int g, int32_t* rowsum_s,
                                              int32_t* colsum_s) {
    const Group& G = p.g[g];
    const int nchunks = G.pw / 128;
    const uint32_t xr = pk_xor(N, cx.row);
    const uint32_t row_off = (A_SIDE ? 0u : (uint32_t)G.a_bytes) + cx.row * 16u * (uint32_t)N;
    if (A_SIDE && cx.halo) {
        cx.hr.tap = cx.hr.cb = cx.hr.r = cx.hr.s = 0;
        halo_tap(p, cx.hr, p.R * p.S);
    }
    uint32_t rsum = 0;
    for (int c = 0; c < nchunks; ++c) {
        const int ci = cx.ci;
        // the halo side reads no ring data: it only hands the slot back
        if (!(A_SIDE && cx.halo) &&
            !__all_sync(0xffffffffu, wait_bounded(cx.bar0 + 8u * (BAR_PK_FULL + ci % PK_SLOTS),
                                                    (ci / PK_SLOTS) & 1, cx.abort_flag, p)))
            return false;
        uint32_t w[4 * N];
        if (A_SIDE && cx.halo) read_halo<N>(p, G, cx.hr, w);
        else read_chunk<N>(cx.pk_base + cx.off + row_off, xr, w);
#pragma unroll
        for (int h = 0; h < (KIND == 0 ? 1 : 2); ++h) {
            const int s = cx.s;
            const int slot = s % OP_STAGES;
            if (!__all_sync(0xffffffffu, wait_bounded(cx.bar0 + 8u * (BAR_OP_EMPTY + slot),
                                                        ((s / OP_STAGES) & 1) ^ 1, cx.abort_flag, p)))
                return false;
            uint32_t out[32];
            if constexpr (KIND == 0) rsum += cvt_e4m3<N, A_SIDE>(w, out);
            else rsum += cvt_f16<N, A_SIDE>(w, h, out);
            if (A_SIDE && cx.a_tmem) {
                // after the MMA that read this stage, before the MMA that will
                tc_fence_after();
                store_stage_tmem(out, cx.a_tmem + (uint32_t)(slot * 32));
                tc_fence_before();
            } else {
                store_stage_smem(out, cx.smem + SMEM_OP + slot * OP_STAGE_BYTES + (A_SIDE ? 0 : OP_A_BYTES), cx.row);
                fence_proxy_async();
            }
            __syncwarp();
            const bool drop = cx.drop_first && s == 0;
            if (cx.lane == 0 && !drop) mbar_arrive(cx.bar0 + 8u * (BAR_OP_FULL + slot));
            cx.s = s + 1;
        }
        if (cx.lane == 0) mbar_arrive(cx.bar0 + 8u * (BAR_PK_EMPTY + ci % PK_SLOTS));
        cx.off = ring_next(cx.ring, ci, cx.off);
        cx.ci = ci + 1;
    }
    if constexpr (A_SIDE) {
        if constexpr (KIND == 0) rowsum_s[g * BM + cx.row] = (int32_t)rsum;   // sum of activation codes
    } else {
        // sum of the weight codes j over the group's K range (offset binary removed)
        if constexpr (KIND == 1) colsum_s[g * BN + cx.row] = (int32_t)rsum - (1 << (N - 1)) * G.pw;
    }
    return true;
}

template <bool A_SIDE>
__device__ __forceinline__ bool convert_group_n(const Params& p, CvtCtx& cx, int g, int32_t* rowsum_s,
                                                int32_t* colsum_s) {
    const Group& G = p.g[g];
    const int n = A_SIDE ? G.bits_a : G.bits_w;
    if (G.kind == 0) {
        switch (n) {
            case 1: return convert_group<1, 0, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
            case 2: return convert_group<2, 0, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
            case 3: return convert_group<3, 0, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
            default: return convert_group<4, 0, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        }
    }
    switch (n) {
        case 1: return convert_group<1, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        case 2: return convert_group<2, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        case 3: return convert_group<3, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        case 4: return convert_group<4, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        case 5: return convert_group<5, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        case 6: return convert_group<6, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        case 7: return convert_group<7, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
        default: return convert_group<8, 1, A_SIDE>(p, cx, g, rowsum_s, colsum_s);
    }
}

// ---- activation gather (implicit GEMM / unaligned rows) -----------------------

// Producer thread t copies block slot i = t & 3 of every chunk for the four
// rows (t >> 2) + 32 k, k = 0..3.  The four threads of a row copy its four
// blocks, which lie side by side in global memory when they share a tap, so a
// warp's copy instruction touches 8 rows instead of 32.  Block kb of a group's
// weight K range holds tap kb / cpt and channel block kb % cpt; slot i of
// chunk c is block 4c + i, so tap, channel block and the tap's filter offsets
// advance by counting.
struct Gather {
    int64_t base[4];   // GEMM: row m; conv: img * H
    int pp[4], qq[4];  // conv: output pixel
    uint32_t valid;    // bit k: row k is < M
    int tap, cb, r, s; // position of this thread's block slot in the next chunk
};

struct GatherGroup {
    int n;       // activation bits
    int cpt;     // 32-code blocks per tap
    int bw;      // cp.async width
    int a_off;   // byte offset of the group in a packed activation row
};

__device__ __forceinline__ void gather_start_group(Gather& gt, int slot_i, int cpt, int S) {
    gt.tap = slot_i / cpt;
    gt.cb = slot_i - gt.tap * cpt;
    gt.r = gt.tap / S;
    gt.s = gt.tap - gt.r * S;
}

__device__ __forceinline__ void gather_advance(Gather& gt, int cpt, int S) {
    gt.cb += 4;
    while (gt.cb >= cpt) {
        gt.cb -= cpt;
        ++gt.tap;
        if (++gt.s == S) {
            gt.s = 0;
            ++gt.r;
        }
    }
}

__device__ __forceinline__ void gather_chunk(const Params& p, const GatherGroup& gg, const Gather& gt, uint32_t t,
                                             uint32_t slot) {
    const int n = gg.n;
    const int bw = gg.bw;
    const int blk = 4 * n;
    const int taps = p.conv ? p.R * p.S : 1;
    const int i = (int)(t & 3u);
    const bool in_k = gt.tap < taps;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t row = (t >> 2) + 32u * (uint32_t)k;
        const uint8_t* src = p.Ap;   // any valid address when zero-filling
        uint32_t nbytes = 0;
        if (((gt.valid >> k) & 1u) && in_k) {
            if (!p.conv) {
                src = p.Ap + gt.base[k] * p.a_row_bytes + gg.a_off + gt.cb * blk;
                nbytes = (uint32_t)bw;
            } else {
                const int h = gt.pp[k] * p.sh - p.ph + gt.r, w = gt.qq[k] * p.sw - p.pw + gt.s;
                if (h >= 0 && h < p.H && w >= 0 && w < p.W) {
                    src = p.Ap + ((gt.base[k] + h) * p.W + w) * p.a_row_bytes + gg.a_off + gt.cb * blk;
                    nbytes = (uint32_t)bw;
                }
            }
        }
        const uint32_t xr = pk_xor(n, row);
        const uint32_t dst_row = slot + row * 16u * (uint32_t)n;
#pragma unroll 1
        for (int b = 0; b < blk; b += bw) {
            const int byte = i * blk + b;
            const uint32_t dst = dst_row + ((((uint32_t)byte >> 4) ^ xr) << 4) + (uint32_t)(byte & 15);
            cp_async(dst, nbytes ? (const void*)(src + b) : (const void*)p.Ap, bw, nbytes);
        }
    }
}

// MMA issue for one group whose activation stages are in TMEM: per stage,
// wait for the operands, 4 MMAs over the stage's 128 bytes of K, and a commit
// that frees the stage when they complete.
template <bool F8>
__device__ __forceinline__ bool mma_group_ta(const Params& p, uint32_t bar0, uint32_t abort_flag, uint32_t op_base,
                                             uint32_t tmem_base, uint32_t d, int nst, int& slot, uint32_t& phase) {
#pragma unroll 1
    for (int ls = 0; ls < nst; ++ls) {
        if (!wait_bounded(bar0 + 8u * (uint32_t)(BAR_OP_FULL + slot), phase, abort_flag, p)) return false;
        tc_fence_after();
        const uint32_t b = op_base + (uint32_t)(slot * OP_STAGE_BYTES + OP_A_BYTES);
        const uint32_t a = tmem_base + (uint32_t)(A_TMEM_COL + slot * 32);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint64_t bd = sw128_desc(b + 32 * k);
            const uint32_t acc = (ls == 0 && k == 0) ? 0u : 1u;
            if constexpr (F8) mma_f8_ta(d, a + 8 * k, bd, acc);
            else mma_f16_ta(d, a + 8 * k, bd, acc);
        }
        mma_commit(bar0 + 8u * (uint32_t)(BAR_OP_EMPTY + slot));
        if (++slot == OP_STAGES) {
            slot = 0;
            phase ^= 1u;
        }
    }
    return true;
}

// ---- the kernel ----------------------------------------------------------------

__global__ void __launch_bounds__(NUM_THREADS, 1) mp_mma_kernel(const __grid_constant__ Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t m0 = (int64_t)blockIdx.y * BM;
    const int n0 = blockIdx.x * BN;

    const uint32_t bar0 = smem_u32(smem + SMEM_BAR);
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + SMEM_MISC);
    const uint32_t abort_flag = smem_u32(smem + SMEM_MISC + 4);
    const uint32_t no_abort = smem_u32(smem + SMEM_MISC + 8);   // stays 0: waits that must run to completion
    int32_t* rowsum_s = reinterpret_cast<int32_t*>(smem + SMEM_ROWSUM);
    float* sw_s = reinterpret_cast<float*>(smem + SMEM_SW);
    int32_t* colsum_s = reinterpret_cast<int32_t*>(smem + SMEM_CS);
    const uint32_t pk_base = smem_u32(smem + SMEM_PK);

    if (threadIdx.x == 0) {
        for (int i = 0; i < PK_SLOTS; ++i) {
            // the TMA arrival, plus one cp.async arrival per producer thread when gathering
            mbar_init(bar(BAR_PK_FULL + i), (p.a_tma || p.a_halo) ? 1 : 1 + NUM_PROD_THREADS);
            mbar_init(bar(BAR_PK_EMPTY + i), 8);
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
        mbar_init(bar(BAR_ROWSUM), 8);
        mbar_init(bar(BAR_TEARDOWN), 1);
        mbar_init(bar(BAR_HALO), NUM_PROD_THREADS);   // one cp.async arrival per producer thread
        asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(abort_flag), "r"(0) : "memory");
        asm volatile("st.volatile.shared.u32 [%0], %1;" ::"r"(no_abort), "r"(0) : "memory");
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

    if (warp >= WARP_PROD && warp < WARP_CVA) {
        // ------------------------------------------------------------ producers
        const uint32_t prow = threadIdx.x - WARP_PROD * 32;     // producer thread index (see Gather)
        const bool lead = prow == 0;                           // issues the TMA copies
        if (p.a_halo) {
            // the tile's input rows, once: pixel first + i of the range goes to halo row i
            const int64_t first = halo_first(p, m0);
            const int64_t cnt = halo_end(p, m0) - first;
            const int cw = p.halo_copy;
            const int per_px = p.a_row_bytes / cw;
            const uint32_t hbase = pk_base + (uint32_t)p.ring_cap;
            const int total = cnt > 0 ? (int)cnt * per_px : 0;
            for (int i = (int)prow; i < total; i += NUM_PROD_THREADS) {
                const int px = i / per_px;
                const int piece = i - px * per_px;
                cp_async(hbase + (uint32_t)px * (uint32_t)p.halo_stride + (uint32_t)(piece * cw),
                         p.Ap + (first + px) * p.a_row_bytes + piece * cw, cw, (uint32_t)cw);
            }
            cp_async_arrive(bar(BAR_HALO));
            if (warp != WARP_PROD) {
                asm volatile("cp.async.wait_all;" ::: "memory");
                goto done;
            }
        }
        if (p.a_tma && warp != WARP_PROD) goto done;           // TMA brings both operands
        {
            Gather gt;
            gt.valid = 0u;
            const int64_t pq = (int64_t)p.P * p.Q;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int64_t m = m0 + (prow >> 2) + 32 * k;
                gt.base[k] = m;
                gt.pp[k] = gt.qq[k] = 0;
                if (m < p.M) {
                    gt.valid |= 1u << k;
                    if (p.conv) {
                        const int64_t img = m / pq;
                        const int rem = (int)(m - img * pq);
                        gt.pp[k] = rem / p.Q;
                        gt.qq[k] = rem - gt.pp[k] * p.Q;
                        gt.base[k] = img * p.H;
                    }
                }
            }
            // Ring bookkeeping (identical in every producer thread): chunks
            // rel..ci-1 are in flight; `tail` is the offset of chunk rel, `off`
            // that of chunk ci and `head` the end of chunk ci-1.
            const RingGeo ring = ring_geo(p);
            const bool a_tma = p.a_tma != 0;
            const bool a_gather = !a_tma && !p.a_halo;             // per-chunk activation gather
            int rel = 0, issued = 0, ci = 0;
            uint32_t off = 0, tail = 0, head = 0;
            bool ok = true;
#pragma unroll 1
            for (int g = 0; g < 2; ++g) {
                const GatherGroup gg{p.g[g].bits_a, p.g[g].pa >> 5, p.g[g].copy_bytes, p.g[g].a_off};
                const int nch = p.g[g].pw / 128;
                const uint32_t a_bytes = (uint32_t)p.g[g].a_bytes, w_bytes = (uint32_t)p.g[g].w_bytes;
                const uint32_t sz = a_bytes + w_bytes;
                const uint32_t tx = w_bytes + (a_tma ? a_bytes : 0u);
                const int w_x0 = p.g[g].w_off, w_dx = 16 * p.g[g].bits_w;
                const int a_x0 = p.g[g].a_off, a_dx = 16 * p.g[g].bits_a;
                if (gg.cpt > 0) gather_start_group(gt, (int)(prow & 3u), gg.cpt, p.S);
                for (int c = 0; c < nch && ok; ++c, ++ci) {
                    const int b = ci % PK_SLOTS;
                    while (rel < ci) {
                        // is [off, off + sz) clear of the chunks in flight, and is a barrier pair free?
                        bool fits;
                        if (ci - rel >= PK_SLOTS) fits = false;
                        else if (off == head) fits = head > tail || head + sz <= tail;   // tail == head: ring full
                        else fits = head > tail && sz <= tail;                           // wrapped to offset 0
                        if (fits) break;
                        // warp-uniform, so that the lanes stay converged for the gather
                        if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_PK_EMPTY + rel % PK_SLOTS), (rel / PK_SLOTS) & 1,
                                                                  abort_flag, p))) {
                            ok = false;
                            break;
                        }
                        tail = ring_next(ring, rel, tail);
                        ++rel;
                    }
                    if (!ok) break;
                    const uint32_t slot = pk_base + off;
                    if (lead) {
                        mbar_arrive_expect_tx(bar(BAR_PK_FULL + b), tx);
                        tma_load_2d(slot + a_bytes, &p.tmw[g], w_x0 + c * w_dx, n0, bar(BAR_PK_FULL + b));
                        if (a_tma) tma_load_2d(slot, &p.tma[g], a_x0 + c * a_dx, (int)m0, bar(BAR_PK_FULL + b));
                    }
                    // reconverge after the lead's copies: a diverged warp issues the gather twice
                    __syncwarp();
                    if (a_gather) {
                        gather_chunk(p, gg, gt, prow, slot);
                        cp_async_arrive(bar(BAR_PK_FULL + b));
                        gather_advance(gt, gg.cpt, p.S);
                    }
                    head = off + sz;
                    off = ring_next(ring, ci, off);
                    ++issued;
                }
            }
            // copies still in flight must land before the CTA's memory is released
            if (lead) {
                for (int ci = issued - PK_SLOTS < 0 ? 0 : issued - PK_SLOTS; ci < issued; ++ci) {
                    wait_bounded(bar(BAR_PK_FULL + ci % PK_SLOTS), (ci / PK_SLOTS) & 1, no_abort, p);
                }
            }
            asm volatile("cp.async.wait_all;" ::: "memory");
        }
    done:;
    } else if (warp == WARP_MMA) {
        // ------------------------------------------------------------------ MMA
        if (lane == 0) {
            bool ok = true;
            const bool a_in_tmem = p.a_in_tmem != 0;
            const int seg_group = p.seg_group;
            int slot = 0;
            uint32_t phase = 0;
            if (a_in_tmem && seg_group < 0) {
                // common case: no segments, activation stages in TMEM.  One tight
                // loop per group with the operand kind fixed (a per-MMA kind test
                // and the segment bookkeeping cost about a third of the issue rate)
#pragma unroll 1
                for (int g = 0; g < 2 && ok; ++g) {
                    const int nst = p.g[g].n_stages;
                    const uint32_t d = tmem_base + (uint32_t)p.acc_col[g];
                    if (p.g[g].kind == 0)
                        ok = mma_group_ta<true>(p, bar0, abort_flag, smem_u32(smem + SMEM_OP), tmem_base, d, nst, slot, phase);
                    else
                        ok = mma_group_ta<false>(p, bar0, abort_flag, smem_u32(smem + SMEM_OP), tmem_base, d, nst, slot, phase);
                }
            } else
#pragma unroll
            for (int g = 0; g < 2; ++g) {
                const int nst = p.g[g].n_stages;
                const bool f8 = p.g[g].kind == 0;
                const bool segmented = seg_group == g;
                const int seg_stages = p.g[g].seg_stages;
                const uint32_t acc_col = (uint32_t)p.acc_col[g];
                int seg = 0, in_seg = 0;
                for (int ls = 0; ls < nst && ok; ++ls) {
                    uint32_t col;
                    bool first, seg_end = false;
                    if (segmented) {
                        first = in_seg == 0;
                        seg_end = in_seg == seg_stages - 1 || ls == nst - 1;
                        col = (uint32_t)(BN + (seg & 1) * BN);
                        if (first && seg >= 2) {
                            if (!wait_bounded(bar(BAR_SLOT_FREE + (seg & 1)), ((seg >> 1) - 1) & 1, abort_flag, p)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                        }
                    } else {
                        first = ls == 0;
                        col = acc_col;
                    }
                    if (!wait_bounded(bar(BAR_OP_FULL + slot), phase, abort_flag, p)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(smem + SMEM_OP + slot * OP_STAGE_BYTES);
                    const uint32_t b_addr = a_addr + OP_A_BYTES;
                    if (a_in_tmem) {
                        // 8 TMEM columns (32 bytes of K per row) per MMA
                        const uint32_t a_t = tmem_base + (uint32_t)(A_TMEM_COL + slot * 32);
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint64_t bd = sw128_desc(b_addr + 32 * k);
                            const uint32_t acc = (first && k == 0) ? 0u : 1u;
                            if (f8) mma_f8_ta(tmem_base + col, a_t + 8 * k, bd, acc);
                            else mma_f16_ta(tmem_base + col, a_t + 8 * k, bd, acc);
                        }
                    } else {
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint64_t ad = sw128_desc(a_addr + 32 * k), bd = sw128_desc(b_addr + 32 * k);
                            const uint32_t acc = (first && k == 0) ? 0u : 1u;
                            if (f8) mma_f8(tmem_base + col, ad, bd, acc);
                            else mma_f16(tmem_base + col, ad, bd, acc);
                        }
                    }
                    mma_commit(bar(BAR_OP_EMPTY + slot));
                    if (seg_end) mma_commit(bar(BAR_SEG_FULL + (seg & 1)));
                    if (segmented && ++in_seg == seg_stages) {
                        in_seg = 0;
                        ++seg;
                    }
                    if (++slot == OP_STAGES) {
                        slot = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (ok) mma_commit(bar(BAR_ACC_FULL));
            // all issued MMAs complete before TMEM and shared memory are released
            mma_commit(bar(BAR_TEARDOWN));
            wait_bounded(bar(BAR_TEARDOWN), 0, no_abort, p);
        }
    } else if (warp < WARP_EPI) {
        // ----------------------------------------------------------- converters
        const bool a_side = warp < WARP_CVW;
        // activation rows follow the warp's TMEM lane quadrant (warp % 4)
        const uint32_t row = a_side ? (uint32_t)((warp & 3) * 32 + lane)
                                    : (uint32_t)(threadIdx.x - WARP_CVW * 32);
        const uint32_t a_tmem = (a_side && p.a_in_tmem)
                                    ? tmem_base + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)A_TMEM_COL
                                    : 0u;
        CvtCtx cx{ring_geo(p), (p.flags & SONIQ_FLAG_TEST_DROP_ARRIVE) != 0 && warp == WARP_CVA,
                  smem_u32(smem), a_tmem, pk_base, bar0, abort_flag, warp, lane, row, 0, 0, 0u};
        cx.halo = a_side && p.a_halo;
        bool halo_ok = true;
        if (cx.halo) {
            const int64_t m = m0 + row;
            const int64_t pq = (int64_t)p.P * p.Q;
            const int64_t img = m / pq;
            const int rem = (int)(m - img * pq);
            const int pp = rem / p.Q, qq = rem - (rem / p.Q) * p.Q;
            const int hp = pp * p.sh - p.ph, wq = qq * p.sw - p.pw;
            cx.hr.base = pk_base + (uint32_t)p.ring_cap;
            cx.hr.pix0 = (int32_t)((img * p.H + hp) * p.W + wq - halo_first(p, m0));
            cx.hr.mr = cx.hr.ms = 0u;
            if (m < p.M) {
                for (int t = 0; t < p.R; ++t)
                    if (hp + t >= 0 && hp + t < p.H) cx.hr.mr |= 1u << t;
                for (int t = 0; t < p.S; ++t)
                    if (wq + t >= 0 && wq + t < p.W) cx.hr.ms |= 1u << t;
            }
            halo_ok = __all_sync(0xffffffffu, wait_bounded(bar(BAR_HALO), 0, abort_flag, p));
        }
#pragma unroll 1
        for (int g = 0; g < 2 && halo_ok; ++g) {
            if (p.g[g].pw == 0) continue;
            const bool ok = a_side ? convert_group_n<true>(p, cx, g, rowsum_s, colsum_s)
                                   : convert_group_n<false>(p, cx, g, rowsum_s, colsum_s);
            if (!ok) break;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_ROWSUM));   // row and column sums are in shared memory
    } else {
        // ---------------------------------------------------- drains + epilogue
        const int quad = warp & 3;                 // TMEM lanes 32*quad .. +31
        const int row = quad * 32 + lane;
        const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16);
        bool ok = true;
        const int gs = p.seg_group;
        if (gs >= 0) {
            const uint32_t sum_col = 3 * BN;
            const int n_seg = gs == 0 ? p.g[0].n_seg : p.g[1].n_seg;
            const float seg_scale = gs == 0 ? p.g[0].acc_scale : p.g[1].acc_scale;
            for (int i = 0; i < n_seg && ok; ++i) {
                if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_SEG_FULL + (i & 1)), (i >> 1) & 1, abort_flag, p))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t ring_col = BN + (i & 1) * BN;
#pragma unroll 1
                for (int cc = 0; cc < BN / 16; ++cc) {
                    uint32_t v[16], s[16];
                    tmem_ld16(lane_base + ring_col + cc * 16, v);
                    if (i > 0) tmem_ld16(lane_base + sum_col + cc * 16, s);
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int32_t x = __float2int_rn(__uint_as_float(v[j]) * seg_scale);
                        s[j] = (uint32_t)((i > 0 ? (int32_t)s[j] : 0) + x);
                    }
                    tmem_st16(lane_base + sum_col + cc * 16, s);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(BAR_SLOT_FREE + (i & 1)));
            }
        }
    }

    // ------------------------------------------------------------- epilogue
    // Every warp but the MMA warp: warp w reads TMEM lanes 32*(w%4).. (its
    // quadrant of rows) and columns 32*((w-1)/4) .. +31, so the four warps of
    // each quadrant (one per role) share the tile's columns.
    // (With a segmented group the int32 sum is written by the epilogue warps'
    // drains, so they alone finish the tile, all columns, after their last drain.)
    const bool shared_epi = p.seg_group < 0;
    if (warp != WARP_MMA && (shared_epi || warp >= WARP_EPI)) {
        const int quad = warp & 3;                 // TMEM lanes 32*quad .. +31
        const int row = quad * 32 + lane;
        const int cc0 = shared_epi ? 2 * ((warp - 1) >> 2) : 0;   // first 16-column block of this warp
        const int cc1 = shared_epi ? cc0 + 2 : BN / 16;
        const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16);
        const int gs = p.seg_group;
        bool ok = true;
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
            int32_t corr[2];   // kind 0: the weight offset times this row's activation code sum
#pragma unroll
            for (int g = 0; g < 2; ++g) corr[g] = p.g[g].w_offset ? p.g[g].w_offset * rowsum_s[g * BM + row] : 0;
            uint32_t col[2];   // TMEM column of each group's result (the int32 sum if segmented)
#pragma unroll
            for (int g = 0; g < 2; ++g) col[g] = g == gs ? 3 * BN : p.acc_col[g];
#pragma unroll 1
            for (int cc = cc0; cc < cc1; ++cc) {
                int32_t acc[2][16];
                uint32_t v[2][16];
                tmem_ld16x2(lane_base + col[0] + cc * 16, lane_base + col[1] + cc * 16, v[0], v[1]);
#pragma unroll
                for (int g = 0; g < 2; ++g) {
                    if (p.g[g].n_stages == 0) {
#pragma unroll
                        for (int j = 0; j < 16; ++j) acc[g][j] = 0;
                        continue;
                    }
                    if (g == gs) {
#pragma unroll
                        for (int j = 0; j < 16; ++j) acc[g][j] = (int32_t)v[g][j] - corr[g];
                    } else {
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            acc[g][j] = __float2int_rn(__uint_as_float(v[g][j]) * p.g[g].acc_scale) - corr[g];
                    }
                    if (p.g[g].a_offset) {   // kind 1: undo the centring of the activations
#pragma unroll
                        for (int j = 0; j < 16; ++j) acc[g][j] += p.g[g].a_offset * colsum_s[g * BN + cc * 16 + j];
                    }
                }
                const int nb = n0 + cc * 16;
                if (m < p.M) {
                    if (p.acc_dbg != nullptr) {
#pragma unroll
                        for (int g = 0; g < 2; ++g) {
                            int32_t* dst = p.acc_dbg + ((int64_t)g * p.M + m) * p.N;
#pragma unroll
                            for (int j = 0; j < 16; ++j)
                                if (nb + j < p.N) dst[nb + j] = acc[g][j];
                        }
                    }
                    float y[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int c = cc * 16 + j;
                        y[j] = fmaf(sa[1] * sw_s[BN + c], (float)acc[1][j], sa[0] * sw_s[c] * (float)acc[0][j]);
                    }
                    const bool vec = nb + 16 <= p.N && (p.N & 7) == 0;
                    if (p.out_bf16) {
                        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.Y) + m * p.N;
                        if (vec) {
#pragma unroll
                            for (int v8 = 0; v8 < 2; ++v8) {
                                uint32_t wv[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    __nv_bfloat162 h2 = __floats2bfloat162_rn(y[v8 * 8 + 2 * e], y[v8 * 8 + 2 * e + 1]);
                                    wv[e] = *reinterpret_cast<uint32_t*>(&h2);
                                }
                                *reinterpret_cast<uint4*>(dst + nb + v8 * 8) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                            }
                        } else {
                            for (int j = 0; j < 16; ++j)
                                if (nb + j < p.N) dst[nb + j] = __float2bfloat16_rn(y[j]);
                        }
                    } else {
                        __half* dst = reinterpret_cast<__half*>(p.Y) + m * p.N;
                        if (vec) {
#pragma unroll
                            for (int v8 = 0; v8 < 2; ++v8) {
                                uint32_t wv[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    __half2 h2 = __floats2half2_rn(y[v8 * 8 + 2 * e], y[v8 * 8 + 2 * e + 1]);
                                    wv[e] = *reinterpret_cast<uint32_t*>(&h2);
                                }
                                *reinterpret_cast<uint4*>(dst + nb + v8 * 8) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                            }
                        } else {
                            for (int j = 0; j < 16; ++j)
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

// The swizzle the converters expect for packed rows of n-bit codes.
CUtensorMapSwizzle packed_swizzle(int n) {
    if (n == 2) return CU_TENSOR_MAP_SWIZZLE_32B;
    if (n == 4) return CU_TENSOR_MAP_SWIZZLE_64B;
    if (n == 8) return CU_TENSOR_MAP_SWIZZLE_128B;
    return CU_TENSOR_MAP_SWIZZLE_NONE;
}

// 2-D map over packed rows [rows][row_bytes] with a box of one 128-code chunk
// (16*n bytes) by 128 rows.
bool encode_packed(EncodeTiledFn enc, CUtensorMap* map, const uint8_t* base, int64_t row_bytes, int64_t rows,
                   int n) {
    cuuint64_t dims[2] = {(cuuint64_t)row_bytes, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
    cuuint32_t box[2] = {(cuuint32_t)(16 * n), 128u};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, packed_swizzle(n), CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Host copies of halo_first / halo_end (same arithmetic).
int64_t host_halo_first(const Params& p, int64_t m0) {
    const int64_t pq = (int64_t)p.P * p.Q;
    const int64_t img = m0 / pq;
    const int pp = (int)((m0 - img * pq) / p.Q);
    int h = pp * p.sh - p.ph;
    if (h < 0) h = 0;
    return (img * p.H + h) * p.W;
}

int64_t host_halo_end(const Params& p, int64_t m0) {
    const int64_t pq = (int64_t)p.P * p.Q;
    const int64_t m_last = (m0 + BM < p.M ? m0 + BM : p.M) - 1;
    const int64_t img = m_last / pq;
    const int pp = (int)((m_last - img * pq) / p.Q);
    int h = pp * p.sh - p.ph + p.R - 1;
    if (h > p.H - 1) h = p.H - 1;
    return (img * p.H + h) * p.W + p.W;
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
    // worst-case |product|: offset-binary weights for E4M3; centred activations
    // times signed weights for fp16
    const int64_t la = (1 << G.bits_a) - 1;
    const int64_t maxprod = out.kind == 0 ? la * ((1 << G.bits_w) - 1)
                                          : (int64_t(1) << (G.bits_a - 1)) * (int64_t(1) << (G.bits_w - 1));
    const int64_t seg_codes = maxprod > 0 ? (int64_t(1) << 24) / maxprod : (int64_t(1) << 24);
    int64_t seg_stages = seg_codes / codes_per_stage;
    if (seg_stages < 1) return false;
    if (seg_stages > out.n_stages) seg_stages = out.n_stages > 0 ? out.n_stages : 1;
    out.seg_stages = (int32_t)seg_stages;
    out.n_seg = out.n_stages > 0 ? (int32_t)((out.n_stages + seg_stages - 1) / seg_stages) : 0;
    out.w_offset = out.kind == 0 ? (1 << (G.bits_w - 1)) : 0;
    out.a_offset = out.kind == 1 ? (1 << (G.bits_a - 1)) : 0;
    out.acc_scale = out.kind == 0 ? 262144.0f : 1.0f;   // 2^18
    out.inv_levels = (float)(1.0 / ((double)la * (double)(1 << (G.bits_w - 1))));
    out.a_bytes = 128 * 16 * G.bits_a;
    out.w_bytes = 128 * 16 * G.bits_w;
    out.copy_bytes = 4;
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
    p.H = a.H; p.W = a.W; p.P = a.P; p.Q = a.Q;
    p.R = a.conv ? a.R : 1;
    p.S = a.conv ? a.S : 1;
    p.sh = a.sh; p.sw = a.sw; p.ph = a.ph; p.pw = a.pw;
    p.s_a_per_row = a.s_a_per_row;
    p.out_bf16 = a.out_bf16;
    p.flags = a.flags;
    p.timeout_ns = 2000000000LL;
    p.seg_group = p.g[0].n_seg > 1 ? 0 : (p.g[1].n_seg > 1 ? 1 : -1);
    if (p.seg_group < 0) {
        // accumulators in columns 0..255, activation stages in 256..351
        p.tmem_cols = 512;
        p.a_in_tmem = 1;
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

    // Activation chunks come by TMA when every chunk of a plain GEMM row starts
    // on a 16-byte boundary and holds data (128-code padding); else by gather.
    bool a_tma = !a.conv && (geo.a_row_bytes % 16 == 0) && ((uintptr_t)a.Ap % 16 == 0);
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = geo.g[g];
        if (G.pw == 0) continue;
        if (G.pa != G.pw || G.a_off % 16 != 0) a_tma = false;
        // widest cp.async copy that keeps every block aligned
        const int blk = 4 * G.bits_a;
        for (int w = 16; w >= 4; w /= 2) {
            if (blk % w == 0 && G.a_off % w == 0 && geo.a_row_bytes % w == 0 && (uintptr_t)a.Ap % w == 0) {
                p.g[g].copy_bytes = w;
                break;
            }
        }
    }
    p.a_tma = a_tma ? 1 : 0;

    // Convolution: load each tile's input rows once (the halo) when they fit
    // beside a ring of at least three weight chunks.
    p.ring_cap = PK_BYTES;
    if (a.conv) {
        const int64_t rb = geo.a_row_bytes;
        const uintptr_t ap = (uintptr_t)a.Ap;
        const int cw = (rb % 16 == 0 && ap % 16 == 0) ? 16 : (rb % 8 == 0 && ap % 8 == 0) ? 8
                                                      : (rb % 4 == 0 && ap % 4 == 0) ? 4 : 0;
        int64_t stride = (rb + 15) / 16 * 16;
        if ((stride / 16) % 2 == 0) stride += 16;   // odd number of 16-byte units: no bank conflicts
        int64_t max_cnt = 0;
        for (int64_t m0 = 0; m0 < a.M; m0 += BM) {
            const int64_t c = host_halo_end(p, m0) - host_halo_first(p, m0);
            if (c > max_cnt) max_cnt = c;
        }
        int64_t w_chunk = 0;
        for (int g = 0; g < 2; ++g)
            if (geo.g[g].pw > 0 && p.g[g].w_bytes > w_chunk) w_chunk = p.g[g].w_bytes;
        const int64_t ring = (PK_BYTES - max_cnt * stride) / 1024 * 1024;
        if (cw > 0 && max_cnt > 0 && ring >= 3 * w_chunk && a.R <= 32 && a.S <= 32) {
            p.a_halo = 1;
            p.halo_stride = (int32_t)stride;
            p.halo_copy = cw;
            p.ring_cap = (int32_t)ring;
            p.g[0].a_bytes = p.g[1].a_bytes = 0;   // activation codes no longer travel in the ring
        }
    }

    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return cudaErrorNotSupported;
    for (int g = 0; g < 2; ++g) {
        if (geo.g[g].pw == 0) continue;
        if (!encode_packed(enc, &p.tmw[g], a.Wp, geo.w_row_bytes, a.N, geo.g[g].bits_w))
            return cudaErrorInvalidValue;
        if (a_tma && !encode_packed(enc, &p.tma[g], a.Ap, geo.a_row_bytes, a.M, geo.g[g].bits_a))
            return cudaErrorInvalidValue;
    }
    static bool attr_done[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(mp_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_ALLOC);
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    cudaError_t ec = prefer_max_shared((const void*)mp_mma_kernel);
    if (ec != cudaSuccess) return ec;
    dim3 grid((unsigned)((a.N + BN - 1) / BN), (unsigned)((a.M + BM - 1) / BM));
    mp_mma_kernel<<<grid, NUM_THREADS, SMEM_ALLOC, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

}  // namespace soniq
