// Swap-AB tensor-core GEMM for few activation rows (decode-sized M): the
// mixed-precision integer GEMM of Sec. 3 / Sec. 4.2 (Acc_g = sum over the
// channels of group g of u * j, exact; Y = sum_g s_a s_w Acc_g / (L_w L_a))
// with the roles of the operands exchanged, so that 128 weight rows fill the
// MMA's M dimension and the M <= 32 activation rows its N dimension.
//
// At these sizes the packed weights dominate the traffic, so they are read
// once, in their packed form, and turned into tensor-pipe operands inside the
// kernel (the staged path's expansion would more than double the bytes):
//
//   warp 0        TMA: a few 128-code chunks of one group for the tile's 128
//                 weight rows and the M activation rows (one box each, rows of
//                 up to 256 bytes), per stage of a ring of raw packed bytes;
//   warps 2..17   converters: packed blocks -> operand bytes in 128-byte-
//                 swizzled K-major tiles (E4M3 for groups whose codes are at
//                 most 4 bits on both sides, fp16 otherwise);
//   warp 1        one thread issues tcgen05.mma (M = 128, N = 16 or 32) into
//                 TMEM; each exact job (a group, or a segment of one, as on the
//                 staged path) accumulates in its own region of a TMEM ring;
//   warps 18..21  drain each job to int32 registers, then apply the scales
//                 and write the outputs (thread = weight row = output column).
//
// Operand encodings (both exact on the tensor pipes):
//   E4M3 groups: activation byte u is the E4M3 value u * 2^-9, weight byte
//     j + 2^(n-1) (offset binary, 0 .. 15) likewise; the fp32 sum of their
//     products times 2^18 is sum u (j + 2^(n-1)), from which 2^(n-1) sum u is
//     taken back with the activation row's code sum.
//   fp16 groups: activations u - 2^(n_a-1), weights j; the weight row's code
//     sum times 2^(n_a-1) is added back.  Jobs are cut into segments whose
//     partial sums stay below 2^24 in magnitude.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "soniq_device.cuh"
#include "soniq_internal.h"
#include "tc_ptx.cuh"

namespace soniq {
namespace skinny {

using namespace tc;

constexpr int BM = 128;                 // weight rows per CTA: the MMA's M
constexpr int NUM_LOAD_WARPS = 1;
constexpr int NUM_CONV_WARPS = 16;
constexpr int NUM_EPI_WARPS = 4;
constexpr int WARP_LOAD = 0, WARP_MMA = NUM_LOAD_WARPS, WARP_CONV = WARP_MMA + 1,
              WARP_EPI = WARP_CONV + NUM_CONV_WARPS;
constexpr int NUM_THREADS = 32 * (WARP_EPI + NUM_EPI_WARPS);
constexpr int MAX_CONV_STAGES = 12;     // converted operand stages (ring size set per launch)
constexpr int MAX_RAW_STAGES = 8;
constexpr int TREGIONS = 8;             // TMEM ring of job accumulators
constexpr int KSTAGE = 128;             // bytes of K per converted stage: 128 E4M3 or 64 fp16 codes
constexpr int W_BYTES = BM * KSTAGE;    // 16 KB
constexpr long long kTimeoutNs = 2000000000LL;

template <int MP>
struct Geo {
    static constexpr int A_BYTES = MP * KSTAGE;
    static constexpr int CONV_SLOT = W_BYTES + A_BYTES;
    static constexpr int TCOLS = TREGIONS * MP <= 128 ? 128 : 256;   // TMEM columns allocated
    // shared memory: [conv slots][raw slots][sums][barriers][misc]
    static constexpr int SMEM_CONV = 0;
};

// barrier indices
constexpr int BAR_RAW_FULL = 0;
constexpr int BAR_RAW_EMPTY = BAR_RAW_FULL + MAX_RAW_STAGES;
constexpr int BAR_CONV_FULL = BAR_RAW_EMPTY + MAX_RAW_STAGES;
constexpr int BAR_CONV_EMPTY = BAR_CONV_FULL + MAX_CONV_STAGES;
constexpr int BAR_TM_FULL = BAR_CONV_EMPTY + MAX_CONV_STAGES;
constexpr int BAR_TM_EMPTY = BAR_TM_FULL + TREGIONS;
constexpr int BAR_SUMS = BAR_TM_EMPTY + TREGIONS;
constexpr int BAR_TEARDOWN = BAR_SUMS + 1;
constexpr int NUM_BARS = BAR_TEARDOWN + 1;

struct KParams {
    CUtensorMap tma_w[2];      // packed weight rows of group g, 4-byte elements: box {rk_g * 4 n_g, 128 rows}
    CUtensorMap tma_a[2];      // packed activation rows of group g: box {rk_g * 4 n_g, MP rows}
    const float* s_a;
    const float* s_w;
    void* Y;
    int32_t* acc_dbg;
    unsigned* err;
    int32_t M, N;
    int32_t s_a_per_row, out_bf16;
    int32_t raw_stages, raw_slot, raw_a_off;    // ring of raw packed chunks (bytes)
    int32_t conv_stages, smem_raw;              // ring of converted stages; offset of the raw ring
    int32_t smem_sums;                          // offset of the code sums
    int32_t drop_first;                         // test hook: the first chunk is never loaded
    int32_t chunks[2];         // 128-code chunks of group g
    int32_t rk[2];             // chunks per raw stage (one TMA box per operand)
    int32_t bits_a[2], bits_w[2];
    int32_t kind[2];           // 0: E4M3, 1: fp16
    int32_t center[2];         // fp16 activations are u - center
    int32_t seg_chunks[2];     // chunks per exact job
    int32_t x_w[2], x_a[2];    // byte offsets of the group in packed weight / activation rows
    float inv_levels[2];       // 1 / (L_w L_a)
    float acc_scale[2];        // TMEM value -> integer: 2^18 (E4M3) or 1
};

__host__ __device__ constexpr int jobs_of(int chunks, int seg) { return chunks > 0 ? (chunks + seg - 1) / seg : 0; }

// One converted 16-byte piece into a 128-byte-swizzled K-major tile (8-row atoms of 1024 bytes).
__device__ __forceinline__ void st_sw128(uint32_t tile, int row, int q, uint32_t a, uint32_t b, uint32_t c,
                                         uint32_t d) {
    const uint32_t addr =
        tile + (uint32_t)(row >> 3) * 1024u + (uint32_t)(row & 7) * 128u + ((((uint32_t)q) ^ (uint32_t)(row & 7)) << 4);
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

template <int N>
__device__ __forceinline__ void lds_words(uint32_t addr, uint32_t (&w)[N]) {
#pragma unroll
    for (int i = 0; i < N; ++i) asm("ld.shared.u32 %0, [%1];" : "=r"(w[i]) : "r"(addr + 4u * i));
}

// Converts block b (32 codes) of one packed row held in shared memory at
// `src` into operand bytes of `tile` row `row`.  Weights: E4M3 offset binary
// or fp16 j; activations: E4M3 u or fp16 u - center.  Returns the block's
// code sum the corrections need (weights, fp16: sum of j; activations, E4M3:
// sum of u; 0 otherwise).
template <int N>
__device__ __forceinline__ int32_t convert_block(uint32_t src, int kind, bool weight, int center, uint32_t tile0,
                                                 uint32_t tile1, int row, int b) {
    uint32_t w[N], o[8];
    lds_words<N>(src, w);
    block_to_bytes<N>(w, o);
    int32_t sum = 0;
    if (kind == 0) {
        if (weight) {
            const uint32_t flip = 0x01010101u << (N - 1);       // two's complement -> offset binary
#pragma unroll
            for (int t = 0; t < 8; ++t) o[t] ^= flip;
        } else {
#pragma unroll
            for (int t = 0; t < 8; ++t) sum = (int32_t)__dp4a(o[t], 0x01010101u, (uint32_t)sum);
        }
        st_sw128(tile0, row, 2 * b, o[0], o[1], o[2], o[3]);
        st_sw128(tile0, row, 2 * b + 1, o[4], o[5], o[6], o[7]);
    } else {
        const uint32_t flip = weight ? 0x01010101u << (N - 1) : 0u;
        const __half2 bias =
            __half2half2(__ushort_as_half((unsigned short)(0x6400u + (weight ? (1u << (N - 1)) : (uint32_t)center))));
        uint32_t h[16];
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            const uint32_t x = o[t] ^ flip;
            if (weight) sum = (int32_t)__dp4a(x, 0x01010101u, (uint32_t)sum);
            uint32_t lo, hi;
            bytes_to_magic_half2(x, lo, hi);
            h[2 * t] = half2_sub(lo, bias);
            h[2 * t + 1] = half2_sub(hi, bias);
        }
        if (weight) sum -= (1 << (N - 1)) * 32;                 // offset-binary sum -> sum of j
        // codes 32 b .. 32 b + 31: stage b / 2, 64 bytes from byte 64 (b % 2)
        const uint32_t tile = (b >> 1) ? tile1 : tile0;
        const int q0 = (b & 1) * 4;
#pragma unroll
        for (int i = 0; i < 4; ++i) st_sw128(tile, row, q0 + i, h[4 * i], h[4 * i + 1], h[4 * i + 2], h[4 * i + 3]);
    }
    return sum;
}

__device__ __forceinline__ int32_t convert_block_n(int n, uint32_t src, int kind, bool weight, int center,
                                                   uint32_t tile0, uint32_t tile1, int row, int b) {
    switch (n) {
        case 1: return convert_block<1>(src, kind, weight, center, tile0, tile1, row, b);
        case 2: return convert_block<2>(src, kind, weight, center, tile0, tile1, row, b);
        case 3: return convert_block<3>(src, kind, weight, center, tile0, tile1, row, b);
        case 4: return convert_block<4>(src, kind, weight, center, tile0, tile1, row, b);
        case 5: return convert_block<5>(src, kind, weight, center, tile0, tile1, row, b);
        case 6: return convert_block<6>(src, kind, weight, center, tile0, tile1, row, b);
        case 7: return convert_block<7>(src, kind, weight, center, tile0, tile1, row, b);
        default: return convert_block<8>(src, kind, weight, center, tile0, tile1, row, b);
    }
}

// A converter thread's fixed assignment: block b (of the 4 in a 128-code
// chunk) of weight row r0, and, for r0 < MP, of activation row r0.
struct ConvState {
    int b, r0, lane;
    bool act;
};

// Converts every chunk of group g (weights NW bits wide); false after a wait
// ran out.  rs / cs count raw chunks and converted stages across the groups.
template <int MP, int NW>
__device__ __forceinline__ bool convert_group(const KParams& p, int g, uint32_t sbase, uint32_t bar0,
                                              uint32_t abort_flag, const ConvState& cv, uint32_t& rs, uint32_t& cs,
                                              int32_t& ws, int32_t& us) {
    using G = Geo<MP>;
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    const int kind = p.kind[g], na = p.bits_a[g], center = p.center[g];
    const int per_chunk = kind == 0 ? 1 : 2;
    const uint32_t RS = (uint32_t)p.raw_stages;
    const int rk = p.rk[g];
    // raw stage rows: rk chunks of 16 NW (weights) / 16 na (activations) bytes each
    const uint32_t w_off0 = (uint32_t)(cv.r0 * rk * 16 * NW + cv.b * 4 * NW);
    const uint32_t a_off = (uint32_t)(p.raw_a_off + cv.r0 * rk * 16 * na + cv.b * 4 * na);
#pragma unroll 1
    for (int c0 = 0; c0 < p.chunks[g]; c0 += rk, ++rs) {
        const uint32_t rslot = rs % RS, rph = (rs / RS) & 1u;
        if (!__all_sync(0xffffffffu,
                        wait_bounded(bar(BAR_RAW_FULL + rslot), rph, abort_flag, kTimeoutNs, p.err, kErrWait)))
            return false;
        const uint32_t raw = sbase + (uint32_t)(p.smem_raw + rslot * p.raw_slot);
        const int nk = p.chunks[g] - c0 < rk ? p.chunks[g] - c0 : rk;
#pragma unroll 1
        for (int k = 0; k < nk; ++k, cs += per_chunk) {
            bool good = true;
            for (int h = 0; h < per_chunk && good; ++h) {
                const uint32_t cslot = (cs + h) % p.conv_stages, cph = ((cs + h) / p.conv_stages) & 1u;
                good = wait_bounded(bar(BAR_CONV_EMPTY + cslot), cph ^ 1u, abort_flag, kTimeoutNs, p.err, kErrWait);
            }
            if (!__all_sync(0xffffffffu, good)) return false;
            const uint32_t t0 = sbase + (uint32_t)(G::SMEM_CONV + (cs % p.conv_stages) * G::CONV_SLOT);
            const uint32_t t1 = sbase + (uint32_t)(G::SMEM_CONV + ((cs + 1) % p.conv_stages) * G::CONV_SLOT);
            const uint32_t kw = (uint32_t)(k * 16 * NW), ka = (uint32_t)(k * 16 * na);
            ws += convert_block<NW>(raw + w_off0 + kw, kind, true, 0, t0, t1, cv.r0, cv.b);
            if (cv.act)
                us += convert_block_n(na, raw + a_off + ka, kind, false, center, t0 + W_BYTES, t1 + W_BYTES, cv.r0,
                                      cv.b);
            fence_proxy_async_shared();
            __syncwarp();
            if (cv.lane == 0)
                for (int h = 0; h < per_chunk; ++h) mbar_arrive(bar(BAR_CONV_FULL + (cs + h) % p.conv_stages));
        }
        __syncwarp();
        if (cv.lane == 0) mbar_arrive(bar(BAR_RAW_EMPTY + rslot));
    }
    return true;
}

template <int MP>
__global__ void __launch_bounds__(NUM_THREADS, 1) skinny_mma_kernel(const __grid_constant__ KParams p) {
    using G = Geo<MP>;
    constexpr uint32_t IDESC = idesc(BM, MP);
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sbase = smem_u32(smem);
    int32_t* usum = reinterpret_cast<int32_t*>(smem + p.smem_sums);          // [2][MP]: activation code sums
    int32_t* colsum = usum + 2 * MP;                                          // [2][BM]: weight code sums
    const uint32_t bar0 = smem_u32(smem + p.smem_sums + 4 * (2 * MP + 2 * BM));
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + p.smem_sums + 4 * (2 * MP + 2 * BM) + 8 * NUM_BARS);
    const uint32_t abort_flag = smem_u32(tmem_slot + 1);
    const uint32_t no_abort = smem_u32(tmem_slot + 2);
    const int n0 = blockIdx.x * BM;
    const int RS = p.raw_stages;

    if (threadIdx.x == 0) {
        for (int i = 0; i < RS; ++i) {
            mbar_init(bar(BAR_RAW_FULL + i), 1);
            mbar_init(bar(BAR_RAW_EMPTY + i), NUM_CONV_WARPS);
        }
        for (int i = 0; i < p.conv_stages; ++i) {
            mbar_init(bar(BAR_CONV_FULL + i), NUM_CONV_WARPS);
            mbar_init(bar(BAR_CONV_EMPTY + i), 1);
        }
        for (int i = 0; i < TREGIONS; ++i) {
            mbar_init(bar(BAR_TM_FULL + i), 1);
            mbar_init(bar(BAR_TM_EMPTY + i), NUM_EPI_WARPS);
        }
        mbar_init(bar(BAR_SUMS), NUM_CONV_WARPS);
        mbar_init(bar(BAR_TEARDOWN), 1);
        set_flag(abort_flag, 0);
        set_flag(no_abort, 0);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    for (int i = threadIdx.x; i < 2 * MP + 2 * BM; i += NUM_THREADS) usum[i] = 0;
    if (warp == WARP_MMA) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(G::TCOLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == WARP_LOAD) {
        // ------------------------------------------------------------ producer
        // one raw stage: rk chunks of group g of the tile's weight rows and of the
        // activation rows, one TMA box each
        if (lane == 0) {
            uint32_t s = 0;
            bool ok = true;
#pragma unroll 1
            for (int g = 0; g < 2 && ok; ++g) {
                const int rk = p.rk[g];
                const uint32_t wbytes = (uint32_t)(BM * rk * 16 * p.bits_w[g]);
                const uint32_t abytes = (uint32_t)(MP * rk * 16 * p.bits_a[g]);
#pragma unroll 1
                for (int c = 0; c < p.chunks[g]; c += rk, ++s) {
                    const uint32_t slot = s % (uint32_t)RS, ph = (s / (uint32_t)RS) & 1u;
                    if (!wait_bounded(bar(BAR_RAW_EMPTY + slot), ph ^ 1u, abort_flag, kTimeoutNs, p.err, kErrWait)) {
                        ok = false;
                        break;
                    }
                    if (p.drop_first && s == 0) continue;   // the converters' wait for it runs out
                    const uint32_t dst = sbase + (uint32_t)(p.smem_raw + slot * p.raw_slot);
                    mbar_arrive_expect_tx(bar(BAR_RAW_FULL + slot), wbytes + abytes);
                    // 4-byte elements: x counts words
                    tma_load_2d(dst, &p.tma_w[g], (p.x_w[g] + c * 16 * p.bits_w[g]) / 4, n0, bar(BAR_RAW_FULL + slot));
                    tma_load_2d(dst + (uint32_t)p.raw_a_off, &p.tma_a[g], (p.x_a[g] + c * 16 * p.bits_a[g]) / 4, 0,
                                bar(BAR_RAW_FULL + slot));
                }
            }
            // loads still in flight land before the CTA's shared memory is released
            for (uint32_t q = s > (uint32_t)RS ? s - RS : 0u; q < s; ++q)
                if (!(p.drop_first && q == 0))
                    wait_bounded(bar(BAR_RAW_FULL + q % RS), (q / RS) & 1u, no_abort, kTimeoutNs, p.err, kErrWait);
        }
    } else if (warp == WARP_MMA) {
        // ------------------------------------------------------------------ MMA
        if (lane == 0) {
            uint32_t cs = 0, job = 0;
            bool ok = true;
            const uint64_t w_desc0 = sw128_desc(sbase + G::SMEM_CONV);
#pragma unroll 1
            for (int g = 0; g < 2 && ok; ++g) {
                const bool f8 = p.kind[g] == 0;
                const int per_chunk = f8 ? 1 : 2;                   // converted stages per raw chunk
                const int nstages = p.chunks[g] * per_chunk;
                const int per_job = p.seg_chunks[g] * per_chunk;
#pragma unroll 1
                for (int i = 0; i < nstages && ok; ++job) {
                    const uint32_t r = job % TREGIONS, use = job / TREGIONS;
                    if (!wait_bounded(bar(BAR_TM_EMPTY + r), (use & 1u) ^ 1u, abort_flag, kTimeoutNs, p.err,
                                      kErrWait)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d = tmem_base + r * MP;
                    const int jn = per_job < nstages - i ? per_job : nstages - i;
#pragma unroll 1
                    for (int q = 0; q < jn; ++q, ++i, ++cs) {
                        const uint32_t slot = cs % p.conv_stages, ph = (cs / p.conv_stages) & 1u;
                        if (!wait_bounded(bar(BAR_CONV_FULL + slot), ph, abort_flag, kTimeoutNs, p.err, kErrWait)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        // +32 bytes of K is +2 in the descriptors' start-address field
                        const uint64_t wd = w_desc0 + (uint64_t)((slot * G::CONV_SLOT) >> 4);
                        const uint64_t ad = wd + (uint64_t)(W_BYTES >> 4);
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint32_t acc = (q > 0 || k > 0) ? 1u : 0u;
                            if (f8)
                                mma_f8<IDESC>(d, wd + 2 * k, ad + 2 * k, acc);
                            else
                                mma_f16<IDESC>(d, wd + 2 * k, ad + 2 * k, acc);
                        }
                        mma_commit(bar(BAR_CONV_EMPTY + slot));
                    }
                    if (ok) mma_commit(bar(BAR_TM_FULL + r));
                }
            }
            // every issued MMA completes before TMEM and shared memory are released
            mma_commit(bar(BAR_TEARDOWN));
            wait_bounded(bar(BAR_TEARDOWN), 0u, no_abort, kTimeoutNs, p.err, kErrWait);
        }
    } else if (warp < WARP_EPI) {
        // ----------------------------------------------------------- converters
        const int t = threadIdx.x - 32 * WARP_CONV;
        ConvState cv;
        cv.b = t & 3;
        cv.r0 = t >> 2;
        cv.act = t < 4 * MP;
        cv.lane = lane;
        uint32_t rs = 0, cs = 0;
        bool ok = true;
        int32_t ws[2] = {0, 0};                   // per group: this block's share of the row's sum of j
        int32_t us[2] = {0, 0};                   // activation code sums (E4M3 groups)
#pragma unroll 1
        for (int g = 0; g < 2 && ok; ++g) {
            switch (p.bits_w[g]) {
                case 1: ok = convert_group<MP, 1>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                case 2: ok = convert_group<MP, 2>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                case 3: ok = convert_group<MP, 3>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                case 4: ok = convert_group<MP, 4>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                case 5: ok = convert_group<MP, 5>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                case 6: ok = convert_group<MP, 6>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                case 7: ok = convert_group<MP, 7>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
                default: ok = convert_group<MP, 8>(p, g, sbase, bar0, abort_flag, cv, rs, cs, ws[g], us[g]); break;
            }
        }
        // the code sums of the corrections (every thread arrives, also after a timeout)
#pragma unroll
        for (int g = 0; g < 2; ++g) {
            int32_t v = ws[g];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            if (cv.b == 0 && p.kind[g] == 1) colsum[g * BM + cv.r0] = v;
            if (cv.act && p.kind[g] == 0) atomicAdd(&usum[g * MP + cv.r0], us[g]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(BAR_SUMS));
    } else {
        // ------------------------------------------------------------- epilogue
        const int quad = warp & 3;
        const int row = quad * 32 + lane;                 // TMEM lane = weight row of the tile
        const int n = n0 + row;
        const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16);
        int32_t part[2][MP];
#pragma unroll
        for (int g = 0; g < 2; ++g)
#pragma unroll
            for (int m = 0; m < MP; ++m) part[g][m] = 0;
        uint32_t job = 0;
        bool ok = true;
#pragma unroll 1
        for (int g = 0; g < 2 && ok; ++g) {
            const int nj = jobs_of(p.chunks[g], p.seg_chunks[g]);
            const float sc = p.acc_scale[g];
#pragma unroll 1
            for (int jj = 0; jj < nj; ++jj, ++job) {
                const uint32_t r = job % TREGIONS, use = job / TREGIONS;
                if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_TM_FULL + r), use & 1u, abort_flag, kTimeoutNs,
                                                          p.err, kErrWait))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
#pragma unroll
                for (int c = 0; c < MP / 16; ++c) {
                    uint32_t v[16];
                    tmem_ld16(lane_base + r * MP + 16 * c, v);
#pragma unroll
                    for (int q = 0; q < 16; ++q) {
                        const int32_t x = __float2int_rn(__uint_as_float(v[q]) * sc);
                        if (g == 0)
                            part[0][16 * c + q] += x;
                        else
                            part[1][16 * c + q] += x;
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(BAR_TM_EMPTY + r));
            }
        }
        const bool sums_ok =
            __all_sync(0xffffffffu, wait_bounded(bar(BAR_SUMS), 0u, no_abort, kTimeoutNs, p.err, kErrWait));
        if (ok && sums_ok && n < p.N) {
            const float kw0 = __ldg(p.s_w + (int64_t)n * 2) * p.inv_levels[0];
            const float kw1 = __ldg(p.s_w + (int64_t)n * 2 + 1) * p.inv_levels[1];
            const int32_t cw0 = p.kind[0] == 1 ? p.center[0] * colsum[row] : 0;
            const int32_t cw1 = p.kind[1] == 1 ? p.center[1] * colsum[BM + row] : 0;
            const int32_t hw0 = p.kind[0] == 0 ? 1 << (p.bits_w[0] - 1) : 0;
            const int32_t hw1 = p.kind[1] == 0 ? 1 << (p.bits_w[1] - 1) : 0;
#pragma unroll
            for (int m = 0; m < MP; ++m) {
                if (m >= p.M) break;
                const int32_t a0 = part[0][m] + cw0 - hw0 * usum[m];
                const int32_t a1 = part[1][m] + cw1 - hw1 * usum[MP + m];
                const float sa0 = p.s_a_per_row ? __ldg(p.s_a + m * 2) : __ldg(p.s_a);
                const float sa1 = p.s_a_per_row ? __ldg(p.s_a + m * 2 + 1) : __ldg(p.s_a + 1);
                const float y = fmaf(sa1 * kw1, (float)a1, sa0 * kw0 * (float)a0);
                const int64_t o = (int64_t)m * p.N + n;
                if (p.out_bf16)
                    reinterpret_cast<__nv_bfloat16*>(p.Y)[o] = __float2bfloat16_rn(y);
                else
                    reinterpret_cast<__half*>(p.Y)[o] = __float2half_rn(y);
                if (p.acc_dbg != nullptr) {
                    p.acc_dbg[o] = a0;
                    p.acc_dbg[(int64_t)p.M * p.N + o] = a1;
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == WARP_MMA) {
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(G::TCOLS)
                     : "memory");
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

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

int mp_for(int64_t M) { return M <= 16 ? 16 : 32; }

struct Plan {
    int kind[2], center[2], seg_chunks[2], chunks[2], rk[2];
    int raw_slot, raw_a_off, raw_stages, conv_stages, smem_raw, smem_sums, smem_alloc;
};

// Shared memory a CTA may take (one CTA per SM).
int smem_budget(int64_t, int64_t) { return 220 * 1024; }

bool plan(const LayoutGeom& geo, int64_t M, int64_t N, Plan* pl) {
    if (geo.taps != 1 || M < 1 || M > 32) return false;
    if (geo.a_row_bytes % 16 != 0 || geo.w_row_bytes % 16 != 0) return false;
    const int MP = mp_for(M);
    int nmax_w = 1, nmax_a = 1;
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& Gg = geo.g[g];
        if (Gg.pw % 128 != 0 || Gg.pa != Gg.pw) return false;    // activation and weight chunks coincide
        if (Gg.a_off % 16 != 0 || Gg.w_off % 16 != 0) return false;
        pl->kind[g] = (Gg.bits_a <= 4 && Gg.bits_w <= 4) ? 0 : 1;
        pl->center[g] = pl->kind[g] == 1 ? (1 << (Gg.bits_a - 1)) : 0;
        pl->chunks[g] = Gg.pw / 128;
        // largest |product| of the job's encoding: exact while partial sums stay below 2^24
        const int64_t maxprod = pl->kind[g] == 0 ? (int64_t)((1 << Gg.bits_a) - 1) * ((1 << Gg.bits_w) - 1)
                                                 : (int64_t)(1 << (Gg.bits_a - 1)) * (1 << (Gg.bits_w - 1));
        const int64_t seg = ((int64_t)1 << 24) / maxprod / 128;
        if (seg < 1) return false;
        pl->seg_chunks[g] = (int)(seg < pl->chunks[g] ? seg : (pl->chunks[g] > 0 ? pl->chunks[g] : 1));
        if (pl->chunks[g] > 0) {
            if (Gg.bits_w > nmax_w) nmax_w = Gg.bits_w;
            if (Gg.bits_a > nmax_a) nmax_a = Gg.bits_a;
        }
    }
    // a raw stage is rk chunks of one group: rows of up to 256 bytes, so that
    // each TMA box row moves a few hundred bytes (boxes of 48-byte rows ran
    // far below the memory's rate)
    int wmax = 0, amax = 0;
    for (int g = 0; g < 2; ++g) {
        const int nb = geo.g[g].bits_w > geo.g[g].bits_a ? geo.g[g].bits_w : geo.g[g].bits_a;
        int rk = 16 / nb;
        if (rk > pl->chunks[g]) rk = pl->chunks[g] > 0 ? pl->chunks[g] : 1;
        pl->rk[g] = rk;
        if (pl->chunks[g] > 0) {
            const int wb = BM * rk * 16 * geo.g[g].bits_w, ab = MP * rk * 16 * geo.g[g].bits_a;
            if (wb > wmax) wmax = wb;
            if (ab > amax) amax = ab;
        }
    }
    (void)nmax_w;
    (void)nmax_a;
    pl->raw_a_off = (wmax + 127) & ~127;
    pl->raw_slot = (pl->raw_a_off + amax + 1023) & ~1023;
    const int conv_slot = W_BYTES + MP * KSTAGE;
    const int tail = 4 * (2 * MP + 2 * BM) + 8 * NUM_BARS + 16 + 1024;
    const int budget = smem_budget(M, N) - tail;
    // about 96 KB of packed bytes in flight (the loads are far from the memory's
    // rate per SM), the rest of the budget for at least 3 converted stages
    int rs = (96 * 1024 + pl->raw_slot - 1) / pl->raw_slot;
    rs = rs < 3 ? 3 : (rs > MAX_RAW_STAGES ? MAX_RAW_STAGES : rs);
    int cs = (budget - rs * pl->raw_slot) / conv_slot;
    while (cs < 4 && rs > 2) {
        --rs;
        cs = (budget - rs * pl->raw_slot) / conv_slot;
    }
    if (cs < 3) return false;
    if (cs > MAX_CONV_STAGES) cs = MAX_CONV_STAGES;
    pl->raw_stages = rs;
    pl->conv_stages = cs;
    pl->smem_raw = cs * conv_slot;
    pl->smem_sums = pl->smem_raw + rs * pl->raw_slot;
    pl->smem_alloc = pl->smem_sums + tail;
    return pl->smem_alloc <= 227 * 1024;
}

template <int MP>
cudaError_t launch_mp(const LayoutGeom& geo, const MmaArgs& a, const Plan& pl, cudaStream_t st) {
    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return cudaErrorNotSupported;
    KParams p{};
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& Gg = geo.g[g];
        const int nw = Gg.bits_w, na = Gg.bits_a;
        {
            cuuint64_t dims[2] = {(cuuint64_t)geo.w_row_bytes / 4, (cuuint64_t)a.N};
            cuuint64_t strides[1] = {(cuuint64_t)geo.w_row_bytes};
            cuuint32_t box[2] = {(cuuint32_t)(pl.rk[g] * 4 * nw), (cuuint32_t)BM};
            cuuint32_t estr[2] = {1, 1};
            if (enc(&p.tma_w[g], CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint8_t*>(a.Wp), dims, strides, box,
                    estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
                return cudaErrorInvalidValue;
        }
        {
            cuuint64_t dims[2] = {(cuuint64_t)geo.a_row_bytes / 4, (cuuint64_t)a.M};
            cuuint64_t strides[1] = {(cuuint64_t)geo.a_row_bytes};
            cuuint32_t box[2] = {(cuuint32_t)(pl.rk[g] * 4 * na), (cuuint32_t)MP};
            cuuint32_t estr[2] = {1, 1};
            if (enc(&p.tma_a[g], CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint8_t*>(a.Ap), dims, strides, box,
                    estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
                return cudaErrorInvalidValue;
        }
        p.chunks[g] = pl.chunks[g];
        p.rk[g] = pl.rk[g];
        p.bits_a[g] = na;
        p.bits_w[g] = nw;
        p.kind[g] = pl.kind[g];
        p.center[g] = pl.center[g];
        p.seg_chunks[g] = pl.seg_chunks[g];
        p.x_w[g] = Gg.w_off;
        p.x_a[g] = Gg.a_off;
        p.inv_levels[g] = (float)(1.0 / ((double)((1 << na) - 1) * (double)(1 << (nw - 1))));
        p.acc_scale[g] = pl.kind[g] == 0 ? 262144.0f : 1.0f;   // 2^18
    }
    p.s_a = a.s_a;
    p.s_w = a.s_w;
    p.Y = a.Y;
    p.acc_dbg = a.acc_dbg;
    p.err = device_error_word();
    if (p.err == nullptr) return cudaErrorUnknown;
    p.M = (int32_t)a.M;
    p.N = a.N;
    p.s_a_per_row = a.s_a_per_row;
    p.out_bf16 = a.out_bf16;
    p.raw_stages = pl.raw_stages;
    p.conv_stages = pl.conv_stages;
    p.smem_raw = pl.smem_raw;
    p.raw_slot = pl.raw_slot;
    p.raw_a_off = pl.raw_a_off;
    p.smem_sums = pl.smem_sums;
    p.drop_first = (a.flags & SONIQ_FLAG_TEST_DROP_ARRIVE) != 0 ? 1 : 0;
    cudaError_t err;
    if ((err = cudaFuncSetAttribute(skinny_mma_kernel<MP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    pl.smem_alloc)) != cudaSuccess)
        return err;
    if ((err = prefer_max_shared((const void*)skinny_mma_kernel<MP>)) != cudaSuccess) return err;
    const int grid = (a.N + BM - 1) / BM;
    skinny_mma_kernel<MP><<<grid, NUM_THREADS, pl.smem_alloc, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

}  // namespace skinny

bool skinny_supported(const LayoutGeom& geo, int64_t M, int64_t N) {
    skinny::Plan pl;
    return N >= 1 && skinny::plan(geo, M, N, &pl);
}

cudaError_t launch_skinny(const LayoutGeom& geo, const MmaArgs& a, cudaStream_t st) {
    skinny::Plan pl;
    if (a.conv || !skinny::plan(geo, a.M, a.N, &pl)) return cudaErrorNotSupported;
    if ((uintptr_t)a.Wp % 16 != 0 || (uintptr_t)a.Ap % 16 != 0) return cudaErrorNotSupported;
    return skinny::mp_for(a.M) == 16 ? skinny::launch_mp<16>(geo, a, pl, st) : skinny::launch_mp<32>(geo, a, pl, st);
}

}  // namespace soniq
