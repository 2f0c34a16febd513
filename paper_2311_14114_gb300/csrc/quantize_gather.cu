// Tiled activation quantize-and-pack with bulk-staged rows: Sec. 3
// "Enabling Low-Cost Fixed-Point Operations" step 2 (unsigned codes) with the
// channel permutation and padding of Sec. 4.1.
//
// A persistent CTA (one per SM) streams tiles of TR consecutive rows.  A
// producer warp copies each row of a tile into a ring of shared-memory stages
// with one bulk copy (rows stay in their original channel order; a 16-byte
// zero slot after every row stands in for the padding positions); a stage is
// refilled as soon as the consumer warps (up to 20, as many as the layout's
// block ranges need) have released it through its "empty" mbarrier, so no
// CTA-wide barrier sits in the tile loop.  Codes are formed one lane per
// packed position: each consumer warp owns a contiguous range of whole
// 8-block chunks of one precision group (its quantizer constants are
// warp-uniform) and, where warps are left over, a share of the tile's rows;
// it holds the staged-row byte offsets of its lanes' channels and walks its
// rows with up to 8 independent gathers per row, so every gather instruction
// reads one row (conflict-free where the permutation keeps channels in order,
// as it does within each group).  The code lands as
// one byte in a per-tile code buffer; after a warp barrier each lane packs
// whole 32-code blocks of that warp and stores them with 16-byte stores.
//
// The code of Sec. 3 step 2, u = clip(rint(RN(RN(a / s) * (2^n - 1))), 0,
// 2^n - 1): the quotient by Markstein's correction step (scales in
// [2^-60, 2^60], exact as in the other quantize kernels), IEEE division
// otherwise; the clip is taken before rounding (its bounds are integers, so
// clip and rint commute, and fmaxf maps NaN to 0 as the clip does); rint is
// the addition of 1.5 * 2^23, after which the low byte of the sum's bits is
// the integer.  Under a calibrated scale the top clip is taken on the input
// instead (a above s becomes s, whose quotient is exactly 1): +inf then
// gets the top code, where the residual step would have made it NaN.
//
// Scale modes: given scales (per tensor after the separate absmax pass, or
// calibrated), or per (row, group) maxima found from the staged rows.
#include <cuda_fp16.h>

#include "soniq_device.cuh"
#include "soniq_internal.h"
#include "tc_ptx.cuh"

namespace soniq {
namespace {

constexpr int kGatherConsumerWarps = 20;                    // at most, code-forming warps
constexpr int kGatherMinConsumerWarps = 8;                  // per-row maxima: one warp per tile row
constexpr int kGatherThreads = (kGatherConsumerWarps + 1) * 32;   // + one producer warp
constexpr int kGatherMaxRows = 8;        // rows per tile
constexpr int kGatherTileRows = 8;       // preferred rows per tile
constexpr int kGatherMaxStages = 4;      // tiles in the ring (all but one in flight)
constexpr size_t kGatherSmemBudget = 220 * 1024;

struct GatherParams {
    const uint16_t* A;
    uint8_t* Ap;
    float* s_a;              // [2] in (given scales) or [M][2] out (per row)
    const int32_t* perm;
    unsigned* err;
    long long timeout_ns;
    int64_t M;
    int32_t K;
    int32_t a_row_bytes;
    int32_t demote;          // reset the L2 eviction priority of every input line read
    int32_t tile_rows;
    int32_t stages;
    int32_t row_stride;      // bytes between staged rows (2K + 16, rounded up to 16)
    int32_t nblk0, nblk;     // 32-code blocks of group 0 / of both groups per row
    int32_t bpw;             // 32-code blocks per warp; each warp takes blocks of one group
    int32_t w0;              // block ranges 0 .. w0-1 are of group 0, w0 .. wb-1 of group 1
    int32_t wb;              // block ranges
    int32_t rg;              // row groups: warp w takes range w % wb and rows w / wb, + rg, ...
    int32_t nwc;             // consumer warps (the producer is warp nwc)
    GroupGeom g[2];
};

// Shared-memory accesses with explicit 32-bit shared addresses.  The load is
// not volatile, so the compiler may schedule the gathers of a row together;
// its address derives from a base that fresh() hands out after the stage's
// wait, which keeps it behind that wait.
__device__ __forceinline__ float lds_half(uint32_t addr) {
    uint16_t v;
    asm("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(addr));
    return __half2float(__ushort_as_half(v));
}

__device__ __forceinline__ void sts_u8(uint32_t addr, uint32_t v) {
    asm volatile("st.shared.u8 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t fresh(uint32_t v) {
    uint32_t r;
    asm volatile("mov.b32 %0, %1;" : "=r"(r) : "r"(v) : "memory");
    return r;
}

// Bits of 1.5 * 2^23 + rint(clip(RN(q * levels), 0, levels)); the low byte is the code.
__device__ __forceinline__ uint32_t code_bits(float q, float levels) {
    float t = __fmul_rn(q, levels);
    t = fminf(fmaxf(t, 0.0f), levels);
    return __float_as_uint(__fadd_rn(t, 12582912.0f));
}

// Quantizer of one (tensor or row, group): mode 1 Markstein quotient, 2 IEEE
// division, 0 every code 0 (no positive scale).
struct GConst {
    float s, r, levels;
    int mode;
};

__device__ __forceinline__ GConst gconst(float s, int bits) {
    GConst k;
    k.s = s;
    k.levels = (float)((1 << bits) - 1);
    k.mode = (s >= 0x1p-60f && s <= 0x1p60f) ? 1 : (s > 0.0f ? 2 : 0);
    k.r = k.mode == 1 ? __frcp_rn(s) : 0.0f;
    return k;
}

__device__ __forceinline__ uint32_t quant_one(float a, const GConst& k) {
    float q;
    if (k.mode == 1) {
        const float q0 = __fmul_rn(a, k.r);
        q = __fmaf_rn(__fmaf_rn(-q0, k.s, a), k.r, q0);
    } else {
        q = k.mode == 2 ? __fdiv_rn(a, k.s) : 0.0f;
    }
    return code_bits(q, k.levels);
}

// Per-group max |a| of one staged row (original channel order; grp_s holds
// 0xFFFF in the halves of group-1 channels), by one warp.
__device__ __forceinline__ void row_group_max(const uint8_t* row, const uint32_t* grp_s, int K, float& f0, float& f1) {
    const int lane = threadIdx.x & 31;
    __half2 g0 = __float2half2_rn(0.0f), g1 = g0;
    for (int v = lane; v < K / 8; v += 32) {
        const uint4 x = reinterpret_cast<const uint4*>(row)[v];
        const uint4 m = *reinterpret_cast<const uint4*>(grp_s + 4 * v);
        const uint32_t xw[4] = {x.x, x.y, x.z, x.w}, mw[4] = {m.x, m.y, m.z, m.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            // |a| (sign cleared) of the group's halves, 0 elsewhere; fp16 max drops NaN
            uint32_t a1 = xw[q] & mw[q] & 0x7FFF7FFFu, a0 = xw[q] & ~mw[q] & 0x7FFF7FFFu;
            g1 = __hmax2(g1, *reinterpret_cast<__half2*>(&a1));
            g0 = __hmax2(g0, *reinterpret_cast<__half2*>(&a0));
        }
    }
    f0 = fmaxf(__low2float(g0), __high2float(g0));
    f1 = fmaxf(__low2float(g1), __high2float(g1));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        f0 = fmaxf(f0, __shfl_xor_sync(0xffffffffu, f0, o));
        f1 = fmaxf(f1, __shfl_xor_sync(0xffffffffu, f1, o));
    }
}

}  // namespace

namespace {

// Codes of nc <= 8 consecutive 32-code blocks of one group (positions pos0 +
// 32 j of this lane) for rows rr0, rr0 + rgs, ... < nr of the tile, into the
// code buffer.  Absent blocks of a short chunk read the zero slot and skip
// their stores.  kc:
// per-row quantizers (MODE 2), kg: the group's quantizer otherwise.
template <int MODE, int RS>
__device__ __forceinline__ void codes_chunk8(uint32_t rows_ba, uint32_t codes_a, const uint32_t* offs_s, int pos0, int nc,
                                             int rr0, int rgs, int nr, uint32_t S, int npos, const GConst (*kc)[2],
                                             const GConst& kg, int g, float lv, uint32_t zero_slot) {
    // RS = 1: the warp takes every row of the tile (rr0 = 0); RS = 0: rows rr0 + k rgs
    const int rstep = RS ? RS : rgs;
    const int rfirst = RS ? 0 : rr0;
    uint32_t off[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) off[j] = j < nc ? offs_s[pos0 + 32 * j] : zero_slot;
#pragma unroll
    for (int ri = 0; ri < kGatherMaxRows; ++ri) {
        const int r = rfirst + ri * rstep;
        if (r < nr) {
            const uint32_t row = rows_ba + (uint32_t)r * S;
            const uint32_t crow = codes_a + (uint32_t)(r * npos + pos0);
            const GConst kk = MODE == 2 ? kc[r][g] : kg;
            if (kk.mode == 1 && nc == 8) {
                float a[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) a[j] = lds_half(row + off[j]);
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float x = MODE == 0 ? fmin_keep_nan(a[j], kk.s) : a[j];
                    const float q0 = __fmul_rn(x, kk.r);
                    const float q = __fmaf_rn(__fmaf_rn(-q0, kk.s, x), kk.r, q0);
                    const float u = fmaxf(__fmul_rn(q, lv), 0.0f);
                    sts_u8(crow + 32u * j, __float_as_uint(__fadd_rn(u, 12582912.0f)));
                }
            } else if (kk.mode == 1) {
                float a[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) a[j] = lds_half(row + off[j]);
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float x = MODE == 0 ? fmin_keep_nan(a[j], kk.s) : a[j];
                    const float q0 = __fmul_rn(x, kk.r);
                    const float q = __fmaf_rn(__fmaf_rn(-q0, kk.s, x), kk.r, q0);
                    const float u = fmaxf(__fmul_rn(q, lv), 0.0f);
                    const uint32_t code = __float_as_uint(__fadd_rn(u, 12582912.0f));
                    if (j < nc) sts_u8(crow + 32u * j, code);
                }
            } else {
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    if (j < nc) sts_u8(crow + 32u * j, quant_one(lds_half(row + off[j]), kk));
            }
        }
    }
}

// MODE 0: calibrated scales s_a[2] (codes clip at the top); 1: per-tensor
// scales s_a[2], the group maxima of these same values; 2: per-(row, group)
// maxima found here.  With the group maximum as the scale, |a| <= s, so the
// correctly rounded quotient is at most 1 and RN(q * levels) at most levels:
// the top clip is void in modes 1 and 2 (on the Markstein path; the IEEE
// path, taken for scales outside [2^-60, 2^60], keeps it).
template <int MODE>
__global__ void __launch_bounds__(kGatherThreads, 1) quantize_gather_kernel(const GatherParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t full_bar[kGatherMaxStages], empty_bar[kGatherMaxStages];
    __shared__ uint32_t abort_s;
    __shared__ GConst kc_s[2][kGatherMaxRows][2];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int TR = p.tile_rows, NST = p.stages, K = p.K;
    const uint32_t S = (uint32_t)p.row_stride, row_bytes = 2u * (uint32_t)K;
    const int pa0 = p.g[0].pa, npos = pa0 + p.g[1].pa;
    const int c0 = p.g[0].count, c1 = p.g[1].count;
    // shared memory: channel offsets | group masks (per row) | codes | staged rows
    uint32_t* offs_s = reinterpret_cast<uint32_t*>(smem);
    size_t o = ((size_t)npos * 4 + 15) & ~(size_t)15;
    uint32_t* grp_s = reinterpret_cast<uint32_t*>(smem + o);
    if (MODE == 2) o += ((size_t)K * 2 + 15) & ~(size_t)15;
    uint8_t* codes_s = smem + o;
    o += ((size_t)TR * npos + 15) & ~(size_t)15;
    uint8_t* rows_s = smem + o;
    const uint32_t rows_a = tc::smem_u32(rows_s);
    const uint32_t abort_flag = tc::smem_u32(&abort_s);
    const int64_t ntiles = (p.M + TR - 1) / TR;

    if (tid == 0) {
        for (int b = 0; b < NST; ++b) {
            tc::mbar_init(tc::smem_u32(&full_bar[b]), 1);
            tc::mbar_init(tc::smem_u32(&empty_bar[b]), (uint32_t)p.nwc);
        }
        tc::set_flag(abort_flag, 0);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    // launched after the previous kernel's start (launch_pdl): every global
    // access comes after this wait; one wave of CTAs, so the kernel that
    // follows may be scheduled at once
    tc::pdl_wait();
    tc::pdl_trigger();

    if (warp == p.nwc) {
        // ---- producer: one lane streams tiles into the stage ring ----
        if (lane == 0) {
            int b = 0;
            uint32_t round = 0u;
            for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x) {
                if (round > 0u &&
                    !tc::wait_bounded(tc::smem_u32(&empty_bar[b]), (round - 1u) & 1u, abort_flag, p.timeout_ns,
                                      p.err, kErrWait))
                    break;
                const int64_t m0 = t * TR;
                const int nr = p.M - m0 < TR ? (int)(p.M - m0) : TR;
                const uint32_t bar = tc::smem_u32(&full_bar[b]);
                tc::mbar_arrive_expect_tx(bar, (uint32_t)nr * row_bytes);
                for (int r = 0; r < nr; ++r)
                    tc::bulk_load(rows_a + (uint32_t)(b * TR + r) * S, p.A + (m0 + r) * K, row_bytes, bar);
                if (++b == NST) {
                    b = 0;
                    ++round;
                }
            }
        }
        return;
    }

    // ---- consumers (p.nwc warps) ----
    const int nthr_c = 32 * p.nwc;
    auto consumer_sync = [nthr_c] { asm volatile("bar.sync 1, %0;" ::"r"(nthr_c) : "memory"); };
    // offsets: the permutation's loads issued eight at a time
    for (int q0 = tid; q0 < npos; q0 += 8 * nthr_c) {
        int ch[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int q = q0 + u * nthr_c;
            int j = -1;
            if (q < pa0) j = q < c0 ? q : -1;
            else if (q < npos) j = q - pa0 < c1 ? c0 + (q - pa0) : -1;
            ch[u] = j >= 0 ? __ldg(p.perm + j) : -1;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int q = q0 + u * nthr_c;
            if (q < npos) offs_s[q] = ch[u] >= 0 ? 2u * (uint32_t)ch[u] : row_bytes;   // padding: the zero slot
        }
    }
    // the zero slot after every staged row (the bulk copies write only the row itself)
    for (int r = tid; r < NST * TR; r += nthr_c)
        *reinterpret_cast<uint4*>(rows_s + (size_t)r * S + row_bytes) = make_uint4(0u, 0u, 0u, 0u);
    if (MODE == 2) {
        for (int w = tid; w < K / 2; w += nthr_c) grp_s[w] = 0u;
        consumer_sync();
        for (int j0 = c0 + tid; j0 < K; j0 += 8 * nthr_c) {
            int ch[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) ch[u] = j0 + u * nthr_c < K ? __ldg(p.perm + j0 + u * nthr_c) : -1;
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (ch[u] >= 0) atomicOr(grp_s + (ch[u] >> 1), (ch[u] & 1) ? 0xFFFF0000u : 0x0000FFFFu);
        }
    }
    consumer_sync();

    // this warp's group, its blocks bw0 .. bw0 + nbw - 1 within the group, and
    // its rows rr0, rr0 + rg, ... of each tile (warps past wb * rg stay idle)
    const bool active = warp < p.wb * p.rg;
    const int wbi = warp % p.wb, rr0 = warp / p.wb, rgs = p.rg;
    const int g = wbi < p.w0 ? 0 : 1;
    const int bw0 = (g ? wbi - p.w0 : wbi) * p.bpw;
    const int nblk_g = g ? p.nblk - p.nblk0 : p.nblk0;
    const int nbw = active ? max(0, min(p.bpw, nblk_g - bw0)) : 0;
    const int gbase = g ? pa0 : 0;
    const int bits = p.g[g].bits_a;
    const int a_off = p.g[g].a_off;
    GConst kg;
    if (MODE != 2) kg = gconst(p.s_a[g], bits);
    const float lv = (float)((1 << bits) - 1);

    const uint8_t* A8 = reinterpret_cast<const uint8_t*>(p.A);
    const uint8_t* A_end = A8 + p.M * (int64_t)row_bytes;
    int b = 0, it = 0;
    uint32_t parity = 0u;
    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++it) {
        const int64_t m0 = t * TR;
        const int nr = p.M - m0 < TR ? (int)(p.M - m0) : TR;
        tc::wait_bounded(tc::smem_u32(&full_bar[b]), parity, abort_flag, p.timeout_ns, p.err, kErrWait);
        if (MODE == 2) consumer_sync();       // every consumer has waited: the abort test below is uniform
        if (tc::abort_raised(abort_flag)) break;
        const uint8_t* rows_b = rows_s + (size_t)(b * TR) * S;
        if (p.demote) {
            // the absmax pass kept these lines in L2 with priority; hand them back
            const uint8_t* lo = A8 + m0 * (int64_t)row_bytes;
            const uint8_t* hi = lo + (int64_t)nr * row_bytes;
            const uint8_t* l0 = reinterpret_cast<const uint8_t*>(((uintptr_t)lo + 127u) & ~(uintptr_t)127u);
            for (const uint8_t* l = l0 + 128 * tid; l < hi && l + 128 <= A_end; l += 128 * nthr_c)
                asm volatile("applypriority.global.L2::evict_normal [%0], 128;" ::"l"(l) : "memory");
        }
        GConst (*kc)[2] = kc_s[it & 1];
        if (MODE == 2) {
            if (warp < nr) {
                float f0, f1;
                row_group_max(rows_b + (size_t)warp * S, grp_s, K, f0, f1);
                if (lane == 0) {
                    p.s_a[(m0 + warp) * 2 + 0] = f0;
                    p.s_a[(m0 + warp) * 2 + 1] = f1;
                    kc[warp][0] = gconst(f0, p.g[0].bits_a);
                    kc[warp][1] = gconst(f1, p.g[1].bits_a);
                }
            }
            consumer_sync();
        }
        // ---- codes: lane per packed position; rows outer, chunks of up to 8 blocks inner ----
        const uint32_t rows_ba = fresh(rows_a + (uint32_t)(b * TR) * S);
        const uint32_t codes_a = tc::smem_u32(codes_s);
        for (int c = 0; c < nbw; c += 8) {
            const int nc = min(8, nbw - c);
            if (rgs == 1)
                codes_chunk8<MODE, 1>(rows_ba, codes_a, offs_s, gbase + (bw0 + c) * 32 + lane, nc, rr0, rgs, nr, S,
                                      npos, kc, kg, g, lv, row_bytes);
            else
                codes_chunk8<MODE, 0>(rows_ba, codes_a, offs_s, gbase + (bw0 + c) * 32 + lane, nc, rr0, rgs, nr, S,
                                      npos, kc, kg, g, lv, row_bytes);
        }
        __syncwarp();
        // this warp no longer reads the stage's rows
        if (lane == 0) tc::mbar_arrive(tc::smem_u32(&empty_bar[b]));
        // ---- pack: lane per (row, 32-code block): block lane % 8 of each chunk, rows lane / 8 and + 4 ----
        for (int c = 0; c < nbw; c += 8) {
            const int j = lane & 7;
            if (c + j < nbw) {
                const int kbg = bw0 + c + j;
#pragma unroll
                for (int h = 0; h < kGatherMaxRows / 4; ++h) {
                    const int r = rr0 + ((lane >> 3) + 4 * h) * rgs;
                    if (r < nr) {
                        const uint4* src = reinterpret_cast<const uint4*>(codes_s + (size_t)r * npos + gbase + kbg * 32);
                        const uint4 lo = src[0], hi = src[1];
                        const uint32_t ow[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
                        store_block32_n(bits, ow, p.Ap + (m0 + r) * (int64_t)p.a_row_bytes + a_off + kbg * 4 * bits);
                    }
                }
            }
        }
        __syncwarp();   // the warp's codes are packed before the next tile overwrites them
        if (++b == NST) {
            b = 0;
            parity ^= 1u;
        }
    }
}

}  // namespace

// Tiled quantize with bulk-staged rows (quantize_gather_kernel).  Needs rows
// of 16-byte-aligned 16-byte multiples (K % 8 == 0, A 16-byte aligned) and
// room for at least one row per stage; returns cudaErrorNotSupported
// otherwise.  scale_mode PER_ROW finds the scales; the others read s_a[2].
// demote: the input's L2 lines were read with an evict-last policy (the
// absmax pass), and their priority is reset as they are read here.
namespace {

struct GatherPlan {
    int32_t tile_rows, stages, row_stride, npos;
    size_t fixed, smem;
};

bool gather_plan(const LayoutGeom& geo, int32_t scale_mode, const void* A, GatherPlan* pl) {
    if (geo.K % 8 != 0 || (uintptr_t)A % 16 != 0) return false;
    if ((geo.g[0].pa + geo.g[1].pa) / 32 == 0) return false;
    pl->npos = geo.g[0].pa + geo.g[1].pa;
    pl->row_stride = ((2 * geo.K + 16) + 15) & ~15;
    const size_t budget = kGatherSmemBudget;
    pl->fixed = (((size_t)pl->npos * 4 + 15) & ~(size_t)15) +
                (scale_mode == SONIQ_SCALE_PER_ROW ? (((size_t)geo.K * 2 + 15) & ~(size_t)15) : 0) + 16;
    if (pl->fixed >= budget) return false;
    // a tile of kGatherTileRows rows with as many stages as fit (at least two),
    // else fewer rows
    const size_t per_row = (size_t)pl->row_stride;
    int64_t tr = kGatherTileRows, nst = 0;
    for (; tr >= 1; --tr) {
        const size_t codes = ((size_t)tr * pl->npos + 15) & ~(size_t)15;
        if (pl->fixed + codes >= budget) continue;
        nst = (int64_t)((budget - pl->fixed - codes) / (tr * per_row));
        if (nst > kGatherMaxStages) nst = kGatherMaxStages;
        if (nst >= 2) break;
    }
    if (tr < 1) return false;
    pl->tile_rows = (int32_t)tr;
    pl->stages = (int32_t)nst;
    pl->smem = pl->fixed + (((size_t)tr * pl->npos + 15) & ~(size_t)15) + (size_t)nst * tr * per_row;
    return pl->smem <= budget;
}

}  // namespace

bool quantize_gather_supported(const LayoutGeom& geo, int32_t scale_mode, const void* A) {
    GatherPlan pl;
    return gather_plan(geo, scale_mode, A, &pl);
}

cudaError_t launch_quantize_gather(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                   int32_t scale_mode, bool demote, float* s_a, uint8_t* Ap, cudaStream_t st) {
    GatherPlan pl;
    if (M < 1 || !gather_plan(geo, scale_mode, A, &pl)) return cudaErrorNotSupported;
    GatherParams p;
    p.A = A;
    p.Ap = Ap;
    p.s_a = s_a;
    p.perm = perm;
    p.err = device_error_word();
    if (p.err == nullptr) return cudaErrorNotSupported;
    p.timeout_ns = 2000000000LL;
    p.M = M;
    p.K = geo.K;
    p.a_row_bytes = geo.a_row_bytes;
    p.demote = demote ? 1 : 0;
    p.g[0] = geo.g[0];
    p.g[1] = geo.g[1];
    p.nblk0 = geo.g[0].pa / 32;
    p.nblk = p.nblk0 + geo.g[1].pa / 32;
    // block ranges of 8 blocks (whole 8-wide chunks), or of a multiple of 8 where
    // the row needs more ranges than there are warps; warps left over split
    // the tile's rows
    const int nblk1 = p.nblk - p.nblk0;
    for (p.bpw = 8;; p.bpw += 8) {
        p.w0 = (p.nblk0 + p.bpw - 1) / p.bpw;
        p.wb = p.w0 + (nblk1 + p.bpw - 1) / p.bpw;
        if (p.wb <= kGatherConsumerWarps) break;
    }
    p.rg = kGatherConsumerWarps / p.wb;
    if (p.rg > pl.tile_rows) p.rg = pl.tile_rows;
    // exactly the warps that take blocks, and one per tile row at least (per-row maxima)
    p.nwc = p.wb * p.rg < kGatherMinConsumerWarps ? kGatherMinConsumerWarps : p.wb * p.rg;
    p.row_stride = pl.row_stride;
    const size_t budget = kGatherSmemBudget;
    const int64_t tr = pl.tile_rows;
    const size_t smem = pl.smem;
    p.tile_rows = (int32_t)tr;
    p.stages = pl.stages;
    const int mode = scale_mode == SONIQ_SCALE_CALIBRATED ? 0 : (scale_mode == SONIQ_SCALE_PER_ROW ? 2 : 1);
    const void* fn = mode == 0 ? (const void*)quantize_gather_kernel<0>
                   : mode == 1 ? (const void*)quantize_gather_kernel<1> : (const void*)quantize_gather_kernel<2>;
    static int attr_dev[3] = {-1, -1, -1};
    int dev = 0;
    cudaGetDevice(&dev);
    if (attr_dev[mode] != dev) {
        cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)budget);
        if (e == cudaSuccess) e = prefer_max_shared(fn);
        if (e != cudaSuccess) return e;
        attr_dev[mode] = dev;
    }
    const int64_t ntiles = (M + tr - 1) / tr;
    const int64_t cap = (int64_t)num_sms();
    const int ctas = (int)(ntiles < cap ? ntiles : cap);
    const dim3 grid((unsigned)ctas), block((unsigned)(32 * (p.nwc + 1)));
    cudaError_t e = mode == 0   ? launch_pdl(quantize_gather_kernel<0>, grid, block, smem, st, p)
                    : mode == 1 ? launch_pdl(quantize_gather_kernel<1>, grid, block, smem, st, p)
                                : launch_pdl(quantize_gather_kernel<2>, grid, block, smem, st, p);
    if (e != cudaSuccess) return e;
    note_launch();
    return cudaGetLastError();
}

}  // namespace soniq
