// Quantize-and-pack kernels: Sec. 3 "Enabling Low-Cost Fixed-Point
// Operations" steps 1-3 with the channel permutation and padding of Sec. 4.1.
//
//   act_absmax_kernel     per-(tensor, group) max |a|            (step 1)
//   quantize_tiles_kernel permute, unsigned codes, pack            (steps 1-2)
//   quantize_fused_kernel per-tensor scale, codes and pack in one pass (steps 1-2)
//   weight_absmax_kernel  per-(tensor, group) max |w|             (step 1)
//   pack_weights_kernel   per-(row, group) scale, Eq. (1) codes, pack (steps 1, 3)
//
// All are HBM-streaming kernels: rows are read with 16-byte loads where the
// alignment allows, the permutation gather happens in shared memory, and one
// warp packs each 32-code block with warp-wide OR reductions.
#include <cuda_fp16.h>

#include "soniq_device.cuh"
#include "soniq_internal.h"
#include "tc_ptx.cuh"

namespace soniq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Block-wide max of two values; result valid in all threads.
__device__ __forceinline__ void block_max2(float& a, float& b, float* red /*[2][32]*/) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    a = warp_max(a);
    b = warp_max(b);
    __syncthreads();
    if (lane == 0) { red[warp] = a; red[32 + warp] = b; }
    __syncthreads();
    a = lane < nw ? red[lane] : 0.0f;
    b = lane < nw ? red[32 + lane] : 0.0f;
    a = warp_max(a);
    b = warp_max(b);
}

// ---------------------------------------------------------------------------
// Per-tensor, per-group max |x| over a [rows][K] matrix whose channel c is in
// group grp(c).  Values are non-negative, so the float bit patterns order as
// unsigned integers and atomicMax on the bits is an exact float max.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads) absmax_kernel(const T* __restrict__ X, int64_t rows,
                                                         int32_t K, const int32_t* __restrict__ perm,
                                                         int32_t count0, unsigned* __restrict__ s_bits,
                                                         int vec_ok) {
    extern __shared__ uint8_t grp[];   // group of each original channel
    __shared__ float red[64];
    for (int j = threadIdx.x; j < K; j += blockDim.x) grp[perm[j]] = (uint8_t)(j >= count0);
    __syncthreads();
    float mx0 = 0.0f, mx1 = 0.0f;
    const int64_t total = rows * (int64_t)K;
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    constexpr int V = 16 / sizeof(T);   // elements per 16-byte vector
    if (vec_ok) {
        const int64_t nvec = total / V;
        for (int64_t v = tid; v < nvec; v += stride) {
            const int64_t e = v * V;
            const int c0 = (int)(e % K);   // K % V == 0: a vector never wraps a row
            uint4 raw = __ldg(reinterpret_cast<const uint4*>(X) + v);
            const T* x = reinterpret_cast<const T*>(&raw);
#pragma unroll
            for (int i = 0; i < V; ++i) {
                float a;
                if constexpr (sizeof(T) == 2) a = fabsf(__half2float(*reinterpret_cast<const __half*>(&x[i])));
                else a = fabsf((float)x[i]);
                if (grp[c0 + i]) mx1 = fmaxf(mx1, a); else mx0 = fmaxf(mx0, a);
            }
        }
    } else {
        for (int64_t e = tid; e < total; e += stride) {
            float a;
            if constexpr (sizeof(T) == 2) a = fabsf(__half2float(*reinterpret_cast<const __half*>(&X[e])));
            else a = fabsf((float)X[e]);
            if (grp[e % K]) mx1 = fmaxf(mx1, a); else mx0 = fmaxf(mx0, a);
        }
    }
    block_max2(mx0, mx1, red);
    if (threadIdx.x == 0) {
        atomicMax(s_bits + 0, __float_as_uint(mx0));
        atomicMax(s_bits + 1, __float_as_uint(mx1));
    }
}

// ---------------------------------------------------------------------------
// fp16 activations, per-(tensor, group) max |a|.  Each thread owns a fixed
// 16-byte column of the [rows][K] matrix (8 channels) and walks rows with
// eight loads in flight, so the channel-to-group masks are computed once.
// |a| is the fp16 bit pattern with the sign cleared, split by group with
// those masks, and folded with the fp16x2 maximum, which returns the other
// operand when one is NaN, as fmaxf does.  keep_l2: the loads carry an L2
// evict-last policy, so that the quantize pass that follows finds the rows in
// L2 (it resets the lines' priority as it reads them).
// ---------------------------------------------------------------------------
constexpr int kAbsmaxThreads = 512;

__device__ __forceinline__ uint4 ld_nc_policy(const uint4* ptr, uint64_t pol) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(ptr), "l"(pol));
    return v;
}

__global__ void __launch_bounds__(kAbsmaxThreads, 4) act_absmax_kernel(const uint4* __restrict__ X, int64_t rows,
                                                                   int32_t K, const int32_t* __restrict__ perm,
                                                                   int32_t count0, int32_t keep_l2,
                                                                   unsigned* __restrict__ s_bits) {
    extern __shared__ uint8_t grp[];   // group of each original channel
    __shared__ float red[64];
    // launched after the previous kernel's start (launch_pdl): its outputs are
    // visible past this wait; one wave of CTAs, so the quantize pass that
    // follows may be scheduled at once
    tc::pdl_wait();
    tc::pdl_trigger();
    // the permutation's loads issued eight at a time
    for (int j0 = threadIdx.x; j0 < K; j0 += 8 * kAbsmaxThreads) {
        int ch[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) ch[u] = j0 + u * kAbsmaxThreads < K ? __ldg(perm + j0 + u * kAbsmaxThreads) : -1;
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (ch[u] >= 0) grp[ch[u]] = (uint8_t)(j0 + u * kAbsmaxThreads >= count0);
    }
    uint64_t pol;
    if (keep_l2) asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    else asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
    __syncthreads();
    const int KV = K >> 3;                         // 16-byte vectors per row
    const int cols = KV < kAbsmaxThreads ? KV : kAbsmaxThreads;
    const int rpar = kAbsmaxThreads / cols;        // rows in flight per CTA
    const int tc = threadIdx.x % cols, tr = threadIdx.x / cols;
    __half2 g0 = __float2half2_rn(0.0f), g1 = g0;  // group maxima, two halves each
    if (tr < rpar) {
        for (int j = tc; j < KV; j += cols) {
            uint32_t m1[4], m0[4];                 // 0x7FFF in the halves of group-1 / group-0 channels
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                m1[q] = (grp[8 * j + 2 * q] ? 0x00007FFFu : 0u) | (grp[8 * j + 2 * q + 1] ? 0x7FFF0000u : 0u);
                m0[q] = m1[q] ^ 0x7FFF7FFFu;
            }
            const int64_t rstep = (int64_t)gridDim.x * rpar;
            for (int64_t m0r = (int64_t)blockIdx.x * rpar + tr; m0r < rows; m0r += 8 * rstep) {
                uint4 v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int64_t m = m0r + u * rstep;
                    v[u] = m < rows ? ld_nc_policy(X + m * KV + j, pol) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint32_t x1 = w[q] & m1[q], x0 = w[q] & m0[q];
                        g1 = __hmax2(g1, *reinterpret_cast<__half2*>(&x1));
                        g0 = __hmax2(g0, *reinterpret_cast<__half2*>(&x0));
                    }
                }
            }
        }
    }
    float mx0 = fmaxf(__low2float(g0), __high2float(g0)), mx1 = fmaxf(__low2float(g1), __high2float(g1));
    block_max2(mx0, mx1, red);
    if (threadIdx.x == 0) {
        atomicMax(s_bits + 0, __float_as_uint(mx0));
        atomicMax(s_bits + 1, __float_as_uint(mx1));
    }
}

// Quantizes 8 halves (x) into two words of bytes: byte b of o[i] is code 4i+b.
template <bool FAST>
__device__ __forceinline__ void quarter_codes(const uint4 x, int valid, const QConst& k, uint32_t o[2]) {
    const uint32_t xw[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        uint32_t v = 0u;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&xw[2 * i + e]));
            const int c = 4 * i + 2 * e;
            const uint32_t u0 = c < valid ? act_code_q<FAST>(f.x, k.s, k.r, k.levels, k.top) : 0u;
            const uint32_t u1 = c + 1 < valid ? act_code_q<FAST>(f.y, k.s, k.r, k.levels, k.top) : 0u;
            v |= (u0 | (u1 << 8)) << (16 * e);
        }
        o[i] = v;
    }
}

// pos_s[perm[j]] = staged position of logical channel j (group 0 first, then
// group 1 from pa0), by the whole block; the permutation's loads are issued
// four at a time.
__device__ __forceinline__ void build_positions(uint16_t* pos_s, const int32_t* __restrict__ perm, int K, int c0,
                                                int pa0) {
    for (int j0 = threadIdx.x; j0 < K; j0 += 4 * blockDim.x) {
        int ch[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) ch[u] = j0 + u * (int)blockDim.x < K ? __ldg(perm + j0 + u * blockDim.x) : -1;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int j = j0 + u * (int)blockDim.x;
            if (ch[u] >= 0) pos_s[ch[u]] = (uint16_t)(j < c0 ? j : pa0 + (j - c0));
        }
    }
}

// ---------------------------------------------------------------------------
// Per-tensor scales in one pass over the input (a cooperative launch, all
// CTAs resident): each CTA stages its rows in shared memory (permuted and
// padded as above) and folds their |a| into the per-group maxima; a grid-wide
// barrier (bounded wait) makes the global maxima visible; the CTA then
// quantizes its staged rows, one thread per 32-code block.  The input is read
// from HBM once instead of twice.
// ---------------------------------------------------------------------------
struct FusedParams {
    const uint16_t* A;
    uint8_t* Ap;
    float* s_a;              // [2] out
    unsigned* bar;           // grid barrier: [0] arrivals (0 between launches), [1] generation
    float* part;             // [gridDim][2] per-CTA maxima
    unsigned* err;           // device error word
    unsigned err_bit;        // bit ORed into it when the barrier wait runs out
    int32_t drop_arrival;    // test hook: CTA 0 does not arrive at the barrier
    const int32_t* perm;
    int64_t M;
    int32_t K;
    int32_t a_row_bytes;
    int32_t vec_ok;
    int32_t rows_per_cta;
    int32_t row_halves;      // pa0 + pa1
    int32_t nblk0, nblk;
    long long timeout_ns;
    GroupGeom g[2];
};

__device__ __forceinline__ uint4 lds128q(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

// 32 staged halves at shared address `src` (padding already zero) -> 8 words of
// bytes, codes by the Markstein quotient (scales in [2^-60, 2^60]).
__device__ __forceinline__ void block_codes_fast(uint32_t src, float s, float rcp, float levels, uint32_t top,
                                                 uint32_t o[8]) {
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        const uint4 x = lds128q(src + 16u * v);
        const uint32_t xw[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            uint32_t word = 0u;
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&xw[2 * i + e]));
                const uint32_t u0 = act_code_q<true>(f.x, s, rcp, levels, top);
                const uint32_t u1 = act_code_q<true>(f.y, s, rcp, levels, top);
                word |= (u0 | (u1 << 8)) << (16 * e);
            }
            o[2 * v + i] = word;
        }
    }
}

// 32 staged halves (codes 0..31 of a block, `valid` of them real) -> 8 words of bytes.
template <bool FAST>
__device__ __forceinline__ void block_codes(const __half* src, int valid, const QConst& k, uint32_t o[8]) {
    const uint4* s4 = reinterpret_cast<const uint4*>(src);
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        uint32_t q[2];
        quarter_codes<FAST>(s4[v], valid - 8 * v, k, q);
        o[2 * v] = q[0];
        o[2 * v + 1] = q[1];
    }
}

__global__ void __launch_bounds__(1024) quantize_fused_kernel(const FusedParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    uint16_t* pos_s = reinterpret_cast<uint16_t*>(smem);
    const int pos_bytes = (p.K * 2 + 15) & ~15;
    __half* rows_s = reinterpret_cast<__half*>(smem + pos_bytes);
    __shared__ float red[64];
    __shared__ int abort_s;
    const int RH = p.row_halves;
    const int c0 = p.g[0].count, pa0 = p.g[0].pa;
    build_positions(pos_s, p.perm, p.K, c0, pa0);
    if (threadIdx.x == 0) abort_s = 0;
    __syncthreads();

    const int64_t m0 = (int64_t)blockIdx.x * p.rows_per_cta;
    const int nr = m0 >= p.M ? 0 : (p.M - m0 < p.rows_per_cta ? (int)(p.M - m0) : p.rows_per_cta);
    // ---- stage the rows; the whole tile is zeroed first so that padding slots
    // hold code 0 and do not count in the max ----
    {
        uint4* z = reinterpret_cast<uint4*>(rows_s);
        const int nz = nr * RH / 8;
        for (int i = threadIdx.x; i < nz; i += blockDim.x) z[i] = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    if (p.vec_ok) {
        // thread -> (row offset, 16-byte column), fixed: no division in the loops
        const int kv = p.K >> 3;
        const int cols = kv < (int)blockDim.x ? kv : (int)blockDim.x;
        const int rp = blockDim.x / cols;
        const int tc = threadIdx.x % cols, tr = threadIdx.x / cols;
        const uint4* src = reinterpret_cast<const uint4*>(p.A + m0 * p.K);
        if (tr < rp) {
            for (int j = tc; j < kv; j += cols) {
                const uint4 ps = *reinterpret_cast<const uint4*>(pos_s + 8 * j);
                const uint32_t pw[4] = {ps.x, ps.y, ps.z, ps.w};
                // four rows' loads in flight before their stores
                for (int r0 = tr; r0 < nr; r0 += 4 * rp) {
                    uint4 v[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int r = r0 + u * rp;
                        v[u] = r < nr ? __ldg(src + (int64_t)r * kv + j) : make_uint4(0u, 0u, 0u, 0u);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int r = r0 + u * rp;
                        if (r >= nr) break;
                        const uint32_t vw[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
                        uint16_t* dst = reinterpret_cast<uint16_t*>(rows_s) + r * RH;
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            dst[pw[q] & 0xFFFFu] = (uint16_t)(vw[q] & 0xFFFFu);
                            dst[pw[q] >> 16] = (uint16_t)(vw[q] >> 16);
                        }
                    }
                }
            }
        }
    } else {
        const uint16_t* src = p.A + m0 * p.K;
        for (int i = threadIdx.x; i < nr * p.K; i += blockDim.x) {
            const int r = i / p.K, c = i - r * p.K;
            reinterpret_cast<uint16_t*>(rows_s)[r * RH + pos_s[c]] = src[i];
        }
    }
    __syncthreads();
    // ---- per-group max |a| over the staged rows: group 0 is [0, pa0), group 1 [pa0, RH) of
    // each row; sign cleared, two halves per instruction, NaN dropped as fmaxf drops it ----
    uint32_t mx0 = 0u, mx1 = 0u;
    {
        const int vpr = RH / 8, v0 = pa0 / 8;   // 16-byte vectors per row / in group 0
        const int cols = vpr < (int)blockDim.x ? vpr : (int)blockDim.x;
        const int rp = blockDim.x / cols;
        const int tc = threadIdx.x % cols, tr = threadIdx.x / cols;
        const uint32_t rs = (uint32_t)__cvta_generic_to_shared(rows_s);
        if (tr < rp) {
            for (int v = tc; v < vpr; v += cols) {
                uint32_t m = 0u;
                for (int r = tr; r < nr; r += rp) {
                    const uint4 x = lds128q(rs + 16u * (uint32_t)(r * vpr + v));
                    const uint32_t xw[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint32_t a = xw[q] & 0x7FFF7FFFu;
                        a &= __vcmpleu2(a, 0x7C007C00u);
                        m = __vmaxu2(m, a);
                    }
                }
                if (v < v0) mx0 = __vmaxu2(mx0, m);
                else mx1 = __vmaxu2(mx1, m);
            }
        }
        mx0 = max(mx0 & 0xFFFFu, mx0 >> 16);
        mx1 = max(mx1 & 0xFFFFu, mx1 >> 16);
    }
    float f0 = __half2float(__ushort_as_half((unsigned short)mx0));
    float f1 = __half2float(__ushort_as_half((unsigned short)mx1));
    block_max2(f0, f1, red);
    // ---- grid barrier: every CTA's maxima are published before anyone reads them.
    // The last CTA to arrive resets the count and advances the generation, so the
    // barrier needs no clearing between launches ----
    if (threadIdx.x == 0) {
        p.part[2 * blockIdx.x + 0] = f0;
        p.part[2 * blockIdx.x + 1] = f1;
        const unsigned gen = *reinterpret_cast<volatile unsigned*>(p.bar + 1);
        __threadfence();
        if (!(p.drop_arrival && blockIdx.x == 0) && atomicAdd(p.bar, 1u) == gridDim.x - 1) {
            *reinterpret_cast<volatile unsigned*>(p.bar) = 0u;
            __threadfence();
            atomicAdd(p.bar + 1, 1u);
        }
        long long t0 = 0;
        for (uint32_t it = 0;; ++it) {
            if (*reinterpret_cast<volatile unsigned*>(p.bar + 1) != gen) break;
            if ((it & 63u) == 63u) {
                long long t;
                asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
                if (t0 == 0) t0 = t;
                else if (t - t0 > p.timeout_ns) {
                    atomicOr(p.err, p.err_bit);
                    abort_s = 1;
                    break;
                }
            }
        }
        __threadfence();
    }
    __syncthreads();
    if (abort_s) return;
    // every CTA folds all partial maxima (a few hundred floats from L2)
    float g0 = 0.0f, g1 = 0.0f;
    for (int i = threadIdx.x; i < (int)gridDim.x; i += blockDim.x) {
        g0 = fmaxf(g0, __ldcg(p.part + 2 * i));
        g1 = fmaxf(g1, __ldcg(p.part + 2 * i + 1));
    }
    block_max2(g0, g1, red);
    if (blockIdx.x == 0 && threadIdx.x < 2) p.s_a[threadIdx.x] = threadIdx.x ? g1 : g0;
    const float s0 = g0, s1 = g1;
    const QConst k0 = make_qconst(s0, p.g[0].bits_a), k1 = make_qconst(s1, p.g[1].bits_a);
    const bool fast = k0.mode == 1 && k1.mode == 1;   // both scales in the Markstein range
    const uint32_t rows_a = (uint32_t)__cvta_generic_to_shared(rows_s);

    // ---- quantize the staged rows: thread per (row, 32-code block) ----
    const int tasks = nr * p.nblk;
    int t = threadIdx.x;
    int r = t / p.nblk, kb = t - r * p.nblk;
    const int dr = blockDim.x / p.nblk, dk = blockDim.x - dr * p.nblk;
    for (; t < tasks; t += blockDim.x) {
        const int g = kb >= p.nblk0;
        const GroupGeom& G = p.g[g];
        const int kbg = kb - (g ? p.nblk0 : 0);
        const QConst& k = g ? k1 : k0;
        const int valid = G.count - kbg * 32;
        const __half* src = rows_s + r * RH + (g ? pa0 : 0) + kbg * 32;
        uint32_t o[8];
        if (fast) {
            const uint32_t sa = rows_a + 2u * (uint32_t)(r * RH + (g ? pa0 : 0) + kbg * 32);
            if (g) block_codes_fast(sa, k1.s, k1.r, k1.levels, k1.top, o);
            else block_codes_fast(sa, k0.s, k0.r, k0.levels, k0.top, o);
        } else if (k.mode == 1) block_codes<true>(src, valid, k, o);
        else if (k.mode == 2) block_codes<false>(src, valid, k, o);
        else {
#pragma unroll
            for (int q = 0; q < 8; ++q) o[q] = 0u;
        }
        store_block32_n(G.bits_a, o, p.Ap + (m0 + r) * (int64_t)p.a_row_bytes + G.a_off + kbg * 4 * G.bits_a);
        r += dr;
        kb += dk;
        if (kb >= p.nblk) {
            kb -= p.nblk;
            ++r;
        }
    }
}

// ---------------------------------------------------------------------------
// Weight quantize-and-pack: one CTA per output row n.  K order inside a group
// is tap-major (position p -> tap p / pa, channel p % pa), padded with code 0.
// ---------------------------------------------------------------------------
struct PackWParams {
    const float* W;
    uint8_t* Wp;
    float* s_w;
    const int32_t* perm;
    int32_t N;
    int32_t K;
    int32_t taps;
    int32_t w_row_bytes;
    int32_t per_row;
    GroupGeom g[2];
};

__global__ void __launch_bounds__(128) pack_weights_kernel(const PackWParams p) {
    __shared__ float red[64];
    __shared__ float s_sh[2];
    const int n = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const float* Wn = p.W + (int64_t)n * p.taps * p.K;

    if (p.per_row) {
        float mx[2] = {0.0f, 0.0f};
#pragma unroll
        for (int g = 0; g < 2; ++g) {
            const int cnt = p.g[g].count;
            const int64_t tot = (int64_t)cnt * p.taps;
            for (int64_t e = threadIdx.x; e < tot; e += blockDim.x) {
                const int t = (int)(e / cnt), c = (int)(e % cnt);
                mx[g] = fmaxf(mx[g], fabsf(__ldg(Wn + (int64_t)t * p.K + p.perm[p.g[g].perm_base + c])));
            }
        }
        block_max2(mx[0], mx[1], red);
        if (threadIdx.x == 0) { s_sh[0] = mx[0]; s_sh[1] = mx[1]; }
    } else if (threadIdx.x == 0) {
        // per-tensor scale, reduced into s_w[0][g] by the absmax kernel
        s_sh[0] = p.s_w[0];
        s_sh[1] = p.s_w[1];
    }
    __syncthreads();
    if (threadIdx.x < 2 && (p.per_row || n > 0)) p.s_w[(int64_t)n * 2 + threadIdx.x] = s_sh[threadIdx.x];

    uint8_t* dst_row = p.Wp + (int64_t)n * p.w_row_bytes;
#pragma unroll
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = p.g[g];
        const int nb = G.bits_w;
        const float half = (float)(1 << (nb - 1));
        const uint32_t mask = (1u << nb) - 1u;
        const float s = s_sh[g];
        const float rh = s > 0.0f ? __frcp_rn(s) * half : 0.0f;   // half is a power of two: exact
        // the estimate below needs a finite RN(1/s) * 2^(n-1): scales under about
        // 2^-121 overflow it, and their codes all take the IEEE division
        const bool est = rh <= 3.402823466e38f;
        uint32_t* dst = reinterpret_cast<uint32_t*>(dst_row + G.w_off);
        for (int kb = warp; kb < G.pw / 32; kb += nwarps) {
            const int pos = kb * 32 + lane;
            const int t = pos / G.pa, c = pos - t * G.pa;
            int32_t j = 0;
            if (t < p.taps && c < G.count && s > 0.0f) {
                // Eq. (1) from the quotient estimate w * RN(1/s), within a few ulps of
                // the correctly rounded w / s (under 3 ulps of 128 even where 1/s is
                // subnormal); |y| = |w / s| 2^(n-1) <= 128, so a y within 8 ulps of 128
                // of a half-integer redoes the IEEE division and every code is the exact
                // rule's (the conversion saturates and takes NaN to 0, as weight_code does)
                const float w = __ldg(Wn + (int64_t)t * p.K + p.perm[G.perm_base + c]);
                const float y = w * rh;
                const float k = rintf(y);
                const int32_t h = 1 << (nb - 1);
                j = (!est || fabsf(fabsf(y - k) - 0.5f) <= 8.0f * 0x1p-16f) ? weight_code(w, s, half)
                                                                            : min(max(__float2int_rz(k), -h), h - 1);
            }
            const uint32_t word = pack_block_warp((uint32_t)j & mask, nb);
            if (lane < nb) dst[kb * nb + lane] = word;
        }
    }
}

// ---------------------------------------------------------------------------
// Activation quantize-and-pack over tiles of rows (persistent CTAs of 1024
// threads).  A tile of rows is staged in shared memory already permuted and
// padded (Sec. 3 "Dynamic channel re-ordering"; the padding slots are zeroed
// once and never written again), so every 32-code block is 64 contiguous
// bytes, and one thread turns a block into its packed words (Sec. 3 step 2).
// While a tile is quantized, the next tile's input is already loading into
// registers.  Scales: given (per tensor after the max-abs pass, or
// calibrated), per row (found from the staged row), or per tensor within a
// single CTA that holds every row (tensor_in_cta, small inputs).
// ---------------------------------------------------------------------------
struct TileQuantParams {
    const uint16_t* A;
    uint8_t* Ap;
    float* s_a;
    const int32_t* perm;
    int64_t M;
    int32_t K;
    int32_t a_row_bytes;
    int32_t scale_mode;
    int32_t tensor_in_cta;
    int32_t vec_ok;          // rows load as 16-byte vectors
    int32_t tile_rows;       // rows per tile
    int32_t row_halves;      // pa0 + pa1: staged row length
    int32_t nblk0, nblk;     // 32-code blocks of group 0 / of both groups per row
    GroupGeom g[2];
};
constexpr int kTileThreads = 1024;
constexpr int kTilePrefetch = 4;   // 16-byte vectors per thread held in registers for the next tile

// Per-group max |a| of staged rows r0 .. r1-1 (sign cleared, NaN dropped as
// fmaxf drops it, two halves per instruction); block-wide, all threads.
__device__ __forceinline__ void staged_group_max(const __half* rows_s, int RH, int pa0, int r0, int r1, float* red,
                                                 float& f0, float& f1) {
    uint32_t mx0 = 0u, mx1 = 0u;
    const int vpr = RH / 8, v0 = pa0 / 8;
    const uint32_t rs = (uint32_t)__cvta_generic_to_shared(rows_s);
    for (int i = threadIdx.x; i < (r1 - r0) * vpr; i += blockDim.x) {
        const int r = r0 + i / vpr, v = i - (i / vpr) * vpr;
        const uint4 x = lds128q(rs + 16u * (uint32_t)(r * vpr + v));
        const uint32_t xw[4] = {x.x, x.y, x.z, x.w};
        uint32_t m = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t a = xw[q] & 0x7FFF7FFFu;
            a &= __vcmpleu2(a, 0x7C007C00u);
            m = __vmaxu2(m, a);
        }
        if (v < v0) mx0 = __vmaxu2(mx0, m);
        else mx1 = __vmaxu2(mx1, m);
    }
    mx0 = max(mx0 & 0xFFFFu, mx0 >> 16);
    mx1 = max(mx1 & 0xFFFFu, mx1 >> 16);
    f0 = __half2float(__ushort_as_half((unsigned short)mx0));
    f1 = __half2float(__ushort_as_half((unsigned short)mx1));
    block_max2(f0, f1, red);
}

__global__ void __launch_bounds__(kTileThreads, 1) quantize_tiles_kernel(const TileQuantParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    uint16_t* pos_s = reinterpret_cast<uint16_t*>(smem);                  // original channel -> staged position
    const int pos_bytes = (p.K * 2 + 15) & ~15;
    float* scale_s = reinterpret_cast<float*>(smem + pos_bytes);          // [tile_rows][2] (per-row scales)
    const int scale_bytes = (p.tile_rows * 8 + 15) & ~15;
    __half* rows_s = reinterpret_cast<__half*>(smem + pos_bytes + scale_bytes);
    __shared__ float red[64];
    const int RH = p.row_halves, TR = p.tile_rows;
    const int c0 = p.g[0].count, pa0 = p.g[0].pa;
    const int KV = p.K >> 3;
    const int64_t tstep = (int64_t)gridDim.x * TR;
    // staging map: vector v of a tile is row v / KV, column v % KV; this thread
    // takes v = tid + u * blockDim for u < kTilePrefetch
    const int tile_vecs = TR * KV;
    uint4 nxt[kTilePrefetch];
    auto load_tile = [&](int64_t m0) {
        const int nr = p.M - m0 < TR ? (int)(p.M - m0) : TR;
        const uint4* src = reinterpret_cast<const uint4*>(p.A + m0 * p.K);
#pragma unroll
        for (int u = 0; u < kTilePrefetch; ++u) {
            const int v = threadIdx.x + u * blockDim.x;
            if (v < tile_vecs && v < nr * KV) nxt[u] = __ldg(src + v);
        }
    };
    // the first tile's loads are in flight while the permutation table is built
    int64_t m0 = (int64_t)blockIdx.x * TR;
    if (p.vec_ok && m0 < p.M) load_tile(m0);
    build_positions(pos_s, p.perm, p.K, c0, pa0);
    {
        uint4* z = reinterpret_cast<uint4*>(rows_s);
        for (int i = threadIdx.x; i < TR * RH / 8; i += blockDim.x) z[i] = make_uint4(0u, 0u, 0u, 0u);
    }
    const bool per_row = p.scale_mode == SONIQ_SCALE_PER_ROW;
    QConst k0, k1;
    if (!per_row && !p.tensor_in_cta) {
        k0 = make_qconst(p.s_a[0], p.g[0].bits_a);
        k1 = make_qconst(p.s_a[1], p.g[1].bits_a);
    }
    __syncthreads();
    const uint32_t rows_a = (uint32_t)__cvta_generic_to_shared(rows_s);
    auto store_tile = [&](int64_t m0) {
        const int nr = p.M - m0 < TR ? (int)(p.M - m0) : TR;
#pragma unroll
        for (int u = 0; u < kTilePrefetch; ++u) {
            const int v = threadIdx.x + u * blockDim.x;
            if (v < tile_vecs && v < nr * KV) {
                const int r = v / KV, j = v - r * KV;
                const uint4 ps = *reinterpret_cast<const uint4*>(pos_s + 8 * j);
                const uint32_t pw[4] = {ps.x, ps.y, ps.z, ps.w};
                const uint32_t vw[4] = {nxt[u].x, nxt[u].y, nxt[u].z, nxt[u].w};
                uint16_t* dst = reinterpret_cast<uint16_t*>(rows_s) + r * RH;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    dst[pw[q] & 0xFFFFu] = (uint16_t)(vw[q] & 0xFFFFu);
                    dst[pw[q] >> 16] = (uint16_t)(vw[q] >> 16);
                }
            }
        }
    };
    for (; m0 < p.M; m0 += tstep) {
        const int nr = p.M - m0 < TR ? (int)(p.M - m0) : TR;
        // ---- stage this tile (from the registers), then start the next tile's loads ----
        if (p.vec_ok) {
            store_tile(m0);
            if (m0 + tstep < p.M) load_tile(m0 + tstep);
        } else {
            const uint16_t* src = p.A + m0 * p.K;
            for (int i = threadIdx.x; i < nr * p.K; i += blockDim.x) {
                const int r = i / p.K, c = i - r * p.K;
                reinterpret_cast<uint16_t*>(rows_s)[r * RH + pos_s[c]] = __ldg(src + i);
            }
        }
        __syncthreads();
        if (p.tensor_in_cta) {
            float f0, f1;
            staged_group_max(rows_s, RH, pa0, 0, nr, red, f0, f1);
            if (threadIdx.x < 2) p.s_a[threadIdx.x] = threadIdx.x ? f1 : f0;
            k0 = make_qconst(f0, p.g[0].bits_a);
            k1 = make_qconst(f1, p.g[1].bits_a);
        } else if (per_row) {
            // max |a| of each staged row and group (the group's channels are contiguous here)
            const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
            for (int r = warp; r < nr; r += nwarps) {
                const __half* row = rows_s + r * RH;
#pragma unroll
                for (int g = 0; g < 2; ++g) {
                    const int base = g ? pa0 : 0;
                    float mx = 0.0f;
                    for (int j = lane; j < p.g[g].count; j += 32) mx = fmaxf(mx, fabsf(__half2float(row[base + j])));
                    mx = warp_max(mx);
                    if (lane == 0) {
                        scale_s[2 * r + g] = mx;
                        p.s_a[(m0 + r) * 2 + g] = mx;
                    }
                }
            }
            __syncthreads();
        }
        // ---- quantize: thread per (row, 32-code block) ----
        const int tasks = nr * p.nblk;
        int t = threadIdx.x;
        int r = t / p.nblk, kb = t - r * p.nblk;
        const int dr = blockDim.x / p.nblk, dk = blockDim.x - dr * p.nblk;
        for (; t < tasks; t += blockDim.x) {
            const int g = kb >= p.nblk0;
            const GroupGeom& G = p.g[g];
            const int kbg = kb - (g ? p.nblk0 : 0);
            const QConst k = per_row ? make_qconst(scale_s[2 * r + g], G.bits_a) : (g ? k1 : k0);
            uint32_t o[8];
            if (k.mode == 1) {
                block_codes_fast(rows_a + 2u * (uint32_t)(r * RH + (g ? pa0 : 0) + kbg * 32), k.s, k.r, k.levels,
                                 k.top, o);
            } else if (k.mode == 2) {
                block_codes<false>(rows_s + r * RH + (g ? pa0 : 0) + kbg * 32, G.count - kbg * 32, k, o);
            } else {
#pragma unroll
                for (int q = 0; q < 8; ++q) o[q] = 0u;
            }
            store_block32_n(G.bits_a, o, p.Ap + (m0 + r) * (int64_t)p.a_row_bytes + G.a_off + kbg * 4 * G.bits_a);
            r += dr;
            kb += dk;
            if (kb >= p.nblk) {
                kb -= p.nblk;
                ++r;
            }
        }
        __syncthreads();   // the tile is overwritten next
    }
}

int grid_for(int64_t work_items, int per_cta) {
    int64_t ctas = (work_items + per_cta - 1) / per_cta;
    int64_t cap = (int64_t)num_sms() * 8;
    if (ctas > cap) ctas = cap;
    if (ctas < 1) ctas = 1;
    return (int)ctas;
}

}  // namespace

cudaError_t launch_act_absmax(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A,
                              int64_t M, float* s_out, bool keep_l2, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(s_out, 0, 2 * sizeof(float), st);
    if (e != cudaSuccess) return e;
    if (geo.K % 8 == 0 && (uintptr_t)A % 16 == 0) {
        const int KV = geo.K / 8;
        const int rpar = kAbsmaxThreads / (KV < kAbsmaxThreads ? KV : kAbsmaxThreads);
        // eight rows per thread in flight; a resident grid of four CTAs per SM
        int64_t ctas = (M + 8 * rpar - 1) / (8 * rpar);
        const int64_t cap = (int64_t)num_sms() * 4;
        if (ctas > cap) ctas = cap;
        if (ctas < 1) ctas = 1;
        if ((e = prefer_max_shared((const void*)act_absmax_kernel)) != cudaSuccess) return e;
        if ((e = launch_pdl(act_absmax_kernel, dim3((unsigned)ctas), dim3(kAbsmaxThreads), (size_t)geo.K, st,
                            reinterpret_cast<const uint4*>(A), M, geo.K, perm, geo.g[0].count, keep_l2 ? 1 : 0,
                            reinterpret_cast<unsigned*>(s_out))) != cudaSuccess)
            return e;
    } else {
        const int grid = grid_for(M * (int64_t)geo.K, kThreads * 4);
        absmax_kernel<__half><<<grid, kThreads, geo.K, st>>>(reinterpret_cast<const __half*>(A), M, geo.K, perm,
                                                             geo.g[0].count, reinterpret_cast<unsigned*>(s_out), 0);
    }
    note_launch();
    return cudaGetLastError();
}

// Tiled quantize (quantize_tiles_kernel).  tensor_in_cta: one CTA holds every
// row in one tile and finds the per-tensor scale itself; returns
// cudaErrorNotSupported when the rows do not fit that way.
cudaError_t launch_quantize_rows(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                 int32_t scale_mode, bool tensor_in_cta, float* s_a, uint8_t* Ap, cudaStream_t st) {
    TileQuantParams p;
    p.A = A;
    p.Ap = Ap;
    p.s_a = s_a;
    p.perm = perm;
    p.M = M;
    p.K = geo.K;
    p.a_row_bytes = geo.a_row_bytes;
    p.scale_mode = scale_mode;
    p.tensor_in_cta = tensor_in_cta ? 1 : 0;
    p.vec_ok = (geo.K % 8 == 0) && ((uintptr_t)A % 16 == 0);
    p.g[0] = geo.g[0];
    p.g[1] = geo.g[1];
    p.nblk0 = geo.g[0].pa / 32;
    p.nblk = p.nblk0 + geo.g[1].pa / 32;
    p.row_halves = geo.g[0].pa + geo.g[1].pa;
    if (p.nblk == 0) return cudaErrorNotSupported;
    const size_t pos_bytes = (size_t)((geo.K * 2 + 15) & ~15);
    const size_t row_bytes = (size_t)p.row_halves * 2;
    const size_t budget = 200 * 1024;
    // rows per tile: what the register prefetch covers (kTilePrefetch vectors per
    // thread) and shared memory holds
    const int64_t KV = geo.K / 8 > 0 ? geo.K / 8 : 1;
    int64_t tr = (int64_t)kTileThreads * kTilePrefetch / KV;
    const int64_t tr_smem = (int64_t)((budget - pos_bytes - 4096) / row_bytes);
    if (tr > tr_smem) tr = tr_smem;
    if (tr > 256) tr = 256;
    if (!p.vec_ok && tr > 64) tr = 64;
    if (tensor_in_cta) {
        // every row in the single CTA's one tile
        if (M > tr) return cudaErrorNotSupported;
        tr = M;
    }
    if (tr < 1) return cudaErrorNotSupported;
    p.tile_rows = (int32_t)tr;
    const size_t smem = pos_bytes + (size_t)((tr * 8 + 15) & ~15) + (size_t)tr * row_bytes;
    if (smem > budget) return cudaErrorNotSupported;
    static int attr_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (attr_dev != dev) {
        cudaError_t e = cudaFuncSetAttribute(quantize_tiles_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)budget);
        if (e == cudaSuccess) e = prefer_max_shared((const void*)quantize_tiles_kernel);
        if (e != cudaSuccess) return e;
        attr_dev = dev;
    }
    int64_t ctas = tensor_in_cta ? 1 : (M + tr - 1) / tr;
    const int64_t cap = (int64_t)num_sms();
    if (ctas > cap) ctas = cap;
    quantize_tiles_kernel<<<(int)ctas, kTileThreads, smem, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

// The one-pass per-tensor path, when every CTA's rows fit in shared memory
// next to a co-resident grid; returns cudaErrorNotSupported otherwise.
cudaError_t launch_quantize_fused(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                  float* s_a, uint8_t* Ap, cudaStream_t st, unsigned* bar, float* part,
                                  int max_ctas, unsigned err_bit) {
    static __thread int attr_dev = -1;
    FusedParams p;
    p.A = A;
    p.Ap = Ap;
    p.s_a = s_a;
    p.err = device_error_word();
    p.bar = bar;
    p.part = part;
    p.err_bit = err_bit;
    p.drop_arrival = 0;
    if (p.err == nullptr || p.bar == nullptr || p.part == nullptr) return cudaErrorNotSupported;
    p.perm = perm;
    p.M = M;
    p.K = geo.K;
    p.a_row_bytes = geo.a_row_bytes;
    p.vec_ok = (geo.K % 8 == 0) && ((uintptr_t)A % 16 == 0);
    p.row_halves = geo.g[0].pa + geo.g[1].pa;
    p.nblk0 = geo.g[0].pa / 32;
    p.nblk = p.nblk0 + geo.g[1].pa / 32;
    p.timeout_ns = 2000000000LL;
    p.g[0] = geo.g[0];
    p.g[1] = geo.g[1];
    if (p.nblk == 0) return cudaErrorNotSupported;
    const int threads = 1024;
    const int sms = num_sms();
    const int64_t rpc = (M + sms - 1) / sms;
    const size_t smem = (size_t)((geo.K * 2 + 15) & ~15) + (size_t)rpc * p.row_halves * 2;
    if (smem > 200 * 1024) return cudaErrorNotSupported;
    p.rows_per_cta = (int32_t)rpc;
    int dev = 0;
    cudaGetDevice(&dev);
    if (attr_dev != dev) {
        cudaError_t e = cudaFuncSetAttribute(quantize_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             200 * 1024);
        if (e != cudaSuccess) return e;
        if ((e = prefer_max_shared((const void*)quantize_fused_kernel)) != cudaSuccess) return e;
        attr_dev = dev;
    }
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, quantize_fused_kernel, threads, smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = (M + rpc - 1) / rpc;
    if (per_sm < 1 || grid > (int64_t)per_sm * sms || grid > max_ctas) return cudaErrorNotSupported;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    p.drop_arrival = take_drop_arrival() ? 1 : 0;
    e = cudaLaunchKernelEx(&cfg, quantize_fused_kernel, p);
    if (e == cudaSuccess) note_launch();
    return e;
}

cudaError_t launch_weight_absmax(const LayoutGeom& geo, const int32_t* perm, const float* W,
                                 int32_t N, float* s_out, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(s_out, 0, 2 * sizeof(float), st);
    if (e != cudaSuccess) return e;
    const int64_t rows = (int64_t)N * geo.taps;
    const int vec_ok = (geo.K % 4 == 0) && ((uintptr_t)W % 16 == 0);
    const int grid = grid_for(rows * geo.K / 4, kThreads * 4);
    absmax_kernel<float><<<grid, kThreads, geo.K, st>>>(W, rows, geo.K, perm, geo.g[0].count,
                                                        reinterpret_cast<unsigned*>(s_out), vec_ok);
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_pack_weights(const LayoutGeom& geo, const int32_t* perm, const float* W,
                                int32_t N, int32_t per_row, uint8_t* Wp, float* s_w,
                                cudaStream_t st) {
    PackWParams p;
    p.W = W;
    p.Wp = Wp;
    p.s_w = s_w;
    p.perm = perm;
    p.N = N;
    p.K = geo.K;
    p.taps = geo.taps;
    p.w_row_bytes = geo.w_row_bytes;
    p.per_row = per_row;
    p.g[0] = geo.g[0];
    p.g[1] = geo.g[1];
    pack_weights_kernel<<<N, 128, 0, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

}  // namespace soniq
