// Staged mixed-precision GEMM / implicit-GEMM convolution on the sm_103a
// tensor cores: expand the packed codes once into tensor-pipe operands in
// caller scratch, then run a persistent tcgen05 GEMM over them.
//
// What it computes (Sec. 3 "Enabling Low-Cost Fixed-Point Operations";
// Sec. 4.2): for each precision group g the exact integer dot products
//   Acc_g[m][n] = sum over k in group g of u[m][k] * j[n][k]
// and Y = sum_g s_a * s_w * Acc_g / ((2^na - 1) * 2^(nw - 1)) in fp32.
//
// Why staged.  Expanding packed codes inside the GEMM tiles (the fused
// kernel of mma_gemm.cu) repeats the expansion of every activation row once
// per column tile and of every weight row once per row tile, and that work,
// not the tensor pipe, sets its speed.  Here each code is expanded exactly
// once, by a streaming kernel, into a byte layout the MMA reads directly;
// the expanded operands (e.g. 63 MB for an 8192 x 4096 x 4096 layer) stay
// in the 129 MB L2 while the GEMM reads them.
//
// Operand encodings (all exact; one group at a time along K):
//   * groups with <= 4-bit codes on both sides: E4M3 bytes.  An activation
//     code u < 16 as a raw byte is the E4M3 value u * 2^-9; a weight code j in
//     [-8, 7] is stored sign-magnitude, the E4M3 value j * 2^-9.  The fp32
//     accumulator holds sum u*j * 2^-18 exactly (|sum| <= 65536 * 15 * 8 <
//     2^24), so the epilogue scales by 2^18.
//   * wider groups: fp16.  Activations are centred, u - 2^(na-1) (padding and
//     taps outside the image count as u = 0), weights are j; every product
//     and partial sum is an integer.  The epilogue adds back
//     2^(na-1) * C[n] with C[n] the weight row's code sum (from the expander).
//     A partial sum stays exact while |sum| <= 2^24; a group whose worst case
//     over its K range could exceed that is accumulated in segments that the
//     epilogue warps drain into int32 registers.
//
// The GEMM kernel: persistent CTAs (one per SM) walk 128 x 256 output tiles
// (N = 256 per MMA: with 128-column MMAs the per-instruction cost, not the
// tensor pipe, set the pace).
//   warp 0      TMA producer: per 128-byte K-stage, an A box (128 rows, 16 KB)
//               and a B box (256 rows, 32 KB), 128-byte swizzle, 4-stage ring
//   warp 1      TMEM owner and MMA issuer (one thread): 4 MMAs per K-stage.
//               A tile's accumulation is a sequence of jobs (a group, or one
//               exact segment of a group; the segmented group first), and job
//               k of the CTA accumulates into TMEM region k % 2 (256 columns
//               each), so the epilogue drains one region while the MMAs fill
//               the other, across tile boundaries too
//   warps 2-9   epilogue: two warps per TMEM lane quadrant, 128 columns each;
//               earlier jobs of a tile are summed into int32 registers, the
//               final job completes the outputs, which leave through shared
//               memory and TMA stores (ten warps in all, so that each thread
//               can hold 128 partial sums in registers)
// Every wait is bounded (2 s); a wait that runs out records an error bit,
// raises a CTA abort flag and the CTA winds down (copies and MMAs in flight
// are waited for, TMEM is freed).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstring>

#include "soniq_device.cuh"
#include "soniq_internal.h"
#include "tc_ptx.cuh"

namespace soniq {
namespace staged {

using namespace tc;

constexpr int BM = 128;
constexpr int BN = 256;                              // tile width (layouts without E2M1 groups)
constexpr int BN_F4 = 240;                           // tile width of layouts with E2M1 groups
constexpr int REGION = 256;                          // TMEM columns per accumulator region
constexpr int SF_COLS = 16;                          // E2M1 scale factors: region columns BN_F4 .. +15
constexpr int KSTAGE = 128;                          // bytes of K per ring stage (128-byte swizzle)
constexpr int STAGES = 3;
constexpr int A_BYTES = BM * KSTAGE;
constexpr int B_BYTES = BN * KSTAGE;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int NUM_EPI_WARPS = 8;
constexpr int WARP_TMA = 0, WARP_MMA = 1, WARP_EPI = 2;
constexpr int NUM_THREADS = (2 + NUM_EPI_WARPS) * 32;
constexpr int BAR_FULL = 0, BAR_EMPTY = STAGES, BAR_REG_FULL = 2 * STAGES, BAR_REG_EMPTY = 2 * STAGES + 2,
              BAR_TEARDOWN = 2 * STAGES + 4, NUM_BARS = 2 * STAGES + 5;
constexpr int EPI_COLS = BN / (NUM_EPI_WARPS / 4);     // columns per epilogue warp (128)
constexpr int COLS_PER_WARP = EPI_COLS * 16;            // float4 per column: s_w0', s_w1', center*C0, center*C1
constexpr int OUT_PER_WARP = 32 * EPI_COLS * 2;         // a warp's 32 x 128 outputs: two 64-column boxes, 128-byte swizzled
constexpr int SMEM_OUT = STAGES * STAGE_BYTES;
constexpr int SMEM_COLS = SMEM_OUT + NUM_EPI_WARPS * OUT_PER_WARP;
constexpr int SMEM_BAR = SMEM_COLS + NUM_EPI_WARPS * COLS_PER_WARP;
constexpr int SMEM_MISC = SMEM_BAR + NUM_BARS * 8;   // tmem base, abort flag, a zero word
constexpr int SMEM_TOTAL = SMEM_MISC + 16;
constexpr int SMEM_ALLOC = SMEM_TOTAL + 1024;        // slack for 1024-byte alignment
constexpr int PAIR_STAGES = 4;                       // ring of the 2-SM kernel (32 KB stages)

// Dynamic shared memory of the 2-SM instantiations: the ring, the output
// staging tile, the column constants, the barriers and misc words, the slack.
constexpr int pair_smem_alloc() {
    return PAIR_STAGES * (A_BYTES + BN / 2 * KSTAGE) + NUM_EPI_WARPS * OUT_PER_WARP + NUM_EPI_WARPS * COLS_PER_WARP +
           (2 * PAIR_STAGES + 5) * 8 + 16 + 1024;
}
static_assert(pair_smem_alloc() <= 227 * 1024, "the 2-SM ring fits");
constexpr uint32_t IDESC = idesc(BM, BN);
constexpr long long kTimeoutNs = 2000000000LL;

struct SGroup {
    int32_t kind;          // 0: E4M3 bytes, 1: fp16, 2: E2M1 nibbles (kind::mxf4)
    int32_t stages;        // 128-byte K-stages of the group
    int32_t x0;            // byte offset of the group in an expanded row
    int32_t seg_stages;    // K-stages per exact segment (segmented group only)
    int32_t n_seg;         // segments (1: accumulated in one piece)
    int32_t center;        // fp16 activations carry -center; the epilogue adds center * C[n]
    float acc_scale;       // 2^18 (E4M3), 1 (fp16) or 4 (E2M1)
    float inv_levels;      // 1 / ((2^na - 1) * 2^(nw - 1))
};

struct SParams {
    CUtensorMap tma_a;     // expanded activations [rows][eb]
    CUtensorMap tma_b;     // expanded weights [N][eb]
    CUtensorMap tma_b2;    // the same, 128-row boxes (each CTA of a pair loads half the tile's rows)
    CUtensorMap tma_y;     // outputs [M][N] (2-byte elements), 64 x 32 boxes, when y_tma
    const float* s_a;
    const float* s_w;
    const int32_t* colsum; // [N][2] weight code sums
    void* Y;
    int32_t* acc_dbg;
    unsigned* err;
    int64_t M;
    int32_t N;
    int32_t m_tiles, n_tiles, total_tiles;
    int32_t pair_tiles;    // CTA pairs: (m tile pair, n tile) units, m tile pairs = ceil(m_tiles / 2)
    int32_t s_a_per_row;
    int32_t out_bf16;
    int32_t seg_group;     // group accumulated in drained segments, or -1
    int32_t drop_first;    // test hook: the producer never issues the first K-stage
    int32_t y_tma;         // 1: outputs leave through shared memory and TMA stores
    int32_t write_y;       // 0: Y is not written (only the next layer's codes)
    // quantize-in-epilogue: output column j is packed position j of the next layer
    int32_t has_next;
    const float* s_next;   // the next layer's calibrated activation scales [2]
    uint8_t* Ap_next;      // its packed activation rows
    int32_t next_row_bytes;
    int32_t next_pa0;      // first packed position of its group 1
    int32_t next_count[2], next_bits[2], next_off[2];
    // scale runs along K: every job is one run of one group, scaled on its own;
    // s_a is [rows or 1][2][nb], s_w [N][2][nb]
    int32_t runs, nb;
    SGroup g[2];
};

// ---------------------------------------------------------------------------
// Expansion of packed rows into tensor-pipe operands
// ---------------------------------------------------------------------------

struct ExpandParams {
    const uint8_t* src;        // packed rows
    int64_t src_row_bytes;
    uint8_t* dst;              // expanded rows
    int64_t dst_row_bytes;
    int32_t* colsum;           // weights: [rows][2] code sums of fp16 groups (else unused)
    int64_t rows;              // output rows (conv activations: output pixels)
    int32_t is_weight;
    int32_t bits[2], kind[2], src_off[2], dst_off[2], blk_src[2], blk_dst[2], center[2];
    // implicit-GEMM convolution (activations): block kb of group g is tap kb / cpt[g],
    // channel block kb % cpt[g] of the input pixel that tap reads
    int32_t conv, H, W, P, Q, R, S, sh, sw, ph, pw;
    int32_t cpt[2];
    uint64_t cpt_magic[2];     // ceil(2^32 / cpt): tap = (kb * magic) >> 32, exact for kb < 2^32 / cpt
    int32_t vec16[2];          // source blocks of the group can be read as 16-byte vectors
    // code encoding of each group: 0 unsigned, 1 n-bit two's complement (weights,
    // signed activations), 2 one-bit +-1 (bit 1 -> +1, bit 0 -> -1, positions
    // from count[g] on -> 0)
    int32_t code_kind[2], count[2];
};

// n-bit two's-complement patterns in the bytes of x -> E4M3 sign-magnitude bytes.
template <int N>
__device__ __forceinline__ uint32_t twos_to_e4m3(uint32_t x) {
    const uint32_t neg = ((x >> (N - 1)) & 0x01010101u) * 0xFFu;   // 0xFF in negative bytes
    const uint32_t mag = ((1u << N) * 0x01010101u) - x;           // 2^N - x per byte, no borrow (x < 2^N)
    return (x & ~neg) | ((mag | 0x80808080u) & neg);
}

// This block's N packed words from src (16-byte loads when the group allows).
template <int N>
__device__ __forceinline__ void load_block_words(const uint8_t* src, bool vec16, uint32_t (&words)[N]) {
    if constexpr (N % 4 == 0) {
        if (vec16) {
#pragma unroll
            for (int i = 0; i < N; i += 4) {
                const uint4 v = __ldg(reinterpret_cast<const uint4*>(src) + i / 4);
                words[i] = v.x;
                words[i + 1] = v.y;
                words[i + 2] = v.z;
                words[i + 3] = v.w;
            }
            return;
        }
    }
#pragma unroll
    for (int i = 0; i < N; ++i) words[i] = __ldg(reinterpret_cast<const uint32_t*>(src) + i);
}

template <int N>
__device__ __forceinline__ void expand_row(const ExpandParams& p, int64_t r, int g, int lane) {
    const int kind = p.kind[g];
    const bool vec16 = p.vec16[g] != 0;
    const uint64_t magic = p.cpt_magic[g];
    uint8_t* drow = p.dst + r * p.dst_row_bytes + p.dst_off[g];
    int64_t img = 0;
    int hp = 0, wq = 0;
    if (p.conv) {
        const int64_t pq = (int64_t)p.P * p.Q;
        img = r / pq;
        const int rem = (int)(r - img * pq);
        const int pp = rem / p.Q, qq = rem - pp * p.Q;
        hp = pp * p.sh - p.ph;
        wq = qq * p.sw - p.pw;
    }
    const uint32_t flip = 0x01010101u << (N - 1);
    const int ck = p.code_kind[g];
    const __half2 bias = __half2half2(__ushort_as_half(
        (unsigned short)(0x6400u + (ck == 1 ? (1u << (N - 1)) : (uint32_t)p.center[g]))));
    int32_t csum = 0;
    for (int kb = lane; kb < p.blk_dst[g]; kb += 32) {
        const uint8_t* src = nullptr;
        if (!p.conv) {
            if (kb < p.blk_src[g]) src = p.src + r * p.src_row_bytes + p.src_off[g] + kb * 4 * N;
        } else {
            const int tap = (int)(((uint64_t)kb * magic) >> 32);
            const int cb = kb - tap * p.cpt[g];
            if (tap < p.R * p.S) {
                const int rr = tap / p.S, ss = tap - rr * p.S;
                const int h = hp + rr, w = wq + ss;
                if (h >= 0 && h < p.H && w >= 0 && w < p.W)
                    src = p.src + ((img * p.H + h) * p.W + w) * p.src_row_bytes + p.src_off[g] + cb * 4 * N;
            }
        }
        uint32_t words[N];
        if (src != nullptr) {
            load_block_words<N>(src, vec16, words);
        } else {
#pragma unroll
            for (int i = 0; i < N; ++i) words[i] = 0u;
        }
        uint32_t o[8];
        block_to_bytes<N>(words, o);
        if (kind == 2) {
            // E2M1, two codes per byte (the first in the low nibble): a code c with
            // |c| <= 4 is sign << 3 | |c|, the value c / 2
            uint32_t hw[4] = {0u, 0u, 0u, 0u};
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const uint32_t x = ck == 1 ? twos_to_e4m3<N>(o[t]) : o[t];   // sign in bit 7, magnitude below
                const uint32_t nib = ((x >> 4) & 0x08080808u) | (x & 0x07070707u);
                const uint32_t y = nib | (nib >> 4);                        // bytes 0 and 2: two codes each
                hw[t >> 1] |= (__byte_perm(y, 0u, 0x0020u) & 0xFFFFu) << (16 * (t & 1));
            }
            *reinterpret_cast<uint4*>(drow + kb * 16) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        } else if (kind == 0) {
            if (ck == 1) {
#pragma unroll
                for (int t = 0; t < 8; ++t) o[t] = twos_to_e4m3<N>(o[t]);
            } else if (ck == 2) {
                // one-bit +-1: bit 1 -> E4M3 +2^-9 (0x01), bit 0 -> -2^-9 (0x81); none past count
#pragma unroll
                for (int t = 0; t < 8; ++t) {
                    const int valid = p.count[g] - (kb * 32 + 4 * t);
                    const uint32_t keep = valid >= 4 ? 0xFFFFFFFFu : (valid <= 0 ? 0u : (1u << (8 * valid)) - 1u);
                    o[t] = (0x81818181u - (o[t] & 0x01010101u) * 0x80u) & keep;
                }
            }
            uint4* d = reinterpret_cast<uint4*>(drow + kb * 32);
            d[0] = make_uint4(o[0], o[1], o[2], o[3]);
            d[1] = make_uint4(o[4], o[5], o[6], o[7]);
        } else {
            uint32_t h[16];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                // signed codes: offset binary j + 2^(n-1); unsigned: the code u
                const uint32_t x = ck == 1 ? (o[t] ^ flip) : o[t];
                if (p.is_weight) csum += (int32_t)__dp4a(x, 0x01010101u, 0u);
                uint32_t lo, hi;
                bytes_to_magic_half2(x, lo, hi);
                h[2 * t] = half2_sub(lo, bias);
                h[2 * t + 1] = half2_sub(hi, bias);
            }
            uint4* d = reinterpret_cast<uint4*>(drow + kb * 64);
#pragma unroll
            for (int q = 0; q < 4; ++q) d[q] = make_uint4(h[4 * q], h[4 * q + 1], h[4 * q + 2], h[4 * q + 3]);
        }
    }
    if (p.is_weight && kind == 1) {
        // sum of j over the row's group: the offset-binary sum minus 2^(n-1) per code
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) csum += __shfl_xor_sync(0xffffffffu, csum, o);
        if (lane == 0) p.colsum[r * 2 + g] = csum - (1 << (N - 1)) * 32 * p.blk_dst[g];
    }
}

// Item `it` (row it / 2, group it % 2) of one operand.
__device__ __forceinline__ void expand_item(const ExpandParams& p, int64_t it, int lane) {
    const int64_t r = it >> 1;
    const int g = (int)(it & 1);
    if (p.blk_dst[g] == 0) return;
    switch (p.bits[g]) {
        case 1: expand_row<1>(p, r, g, lane); break;
        case 2: expand_row<2>(p, r, g, lane); break;
        case 3: expand_row<3>(p, r, g, lane); break;
        case 4: expand_row<4>(p, r, g, lane); break;
        case 5: expand_row<5>(p, r, g, lane); break;
        case 6: expand_row<6>(p, r, g, lane); break;
        case 7: expand_row<7>(p, r, g, lane); break;
        default: expand_row<8>(p, r, g, lane); break;
    }
}

// Both operands in one launch: items 0 .. 2 rows_a - 1 are (row, group) of the
// activations (pa), the rest of the weights (pw).
__global__ void __launch_bounds__(256, 5) expand_kernel(const __grid_constant__ ExpandParams pa,
                                                     const __grid_constant__ ExpandParams pw) {
    tc::pdl_wait();   // launched with launch_pdl: the packed rows are written before this
    const int lane = threadIdx.x & 31;
    const int64_t warp_id = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int64_t items_a = pa.rows * 2;
    for (int64_t item = warp_id; item < items_a + pw.rows * 2; item += nwarps) {
        if (item < items_a) expand_item(pa, item, lane);
        else expand_item(pw, item - items_a, lane);
    }
}

// ---------------------------------------------------------------------------
// The persistent GEMM over expanded operands
// ---------------------------------------------------------------------------

// 8 consecutive outputs of row m from column nb (one 16-byte store when aligned).
__device__ __forceinline__ void store_out8(const SParams& p, int64_t m, int nb, const float (&y)[8]) {
    const bool vec = nb + 8 <= p.N && (p.N & 7) == 0;
    uint32_t wv[4];
    if (p.out_bf16) {
        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.Y) + m * p.N;
        if (vec) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                __nv_bfloat162 h2 = __floats2bfloat162_rn(y[2 * e], y[2 * e + 1]);
                wv[e] = *reinterpret_cast<uint32_t*>(&h2);
            }
            *reinterpret_cast<uint4*>(dst + nb) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
        } else {
            for (int j = 0; j < 8; ++j)
                if (nb + j < p.N) dst[nb + j] = __float2bfloat16_rn(y[j]);
        }
    } else {
        __half* dst = reinterpret_cast<__half*>(p.Y) + m * p.N;
        if (vec) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                __half2 h2 = __floats2half2_rn(y[2 * e], y[2 * e + 1]);
                wv[e] = *reinterpret_cast<uint32_t*>(&h2);
            }
            *reinterpret_cast<uint4*>(dst + nb) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
        } else {
            for (int j = 0; j < 8; ++j)
                if (nb + j < p.N) dst[nb + j] = __float2half_rn(y[j]);
        }
    }
}

__device__ __forceinline__ void store_out16(const SParams& p, int64_t m, int nb, const float (&y)[16]) {
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

// The tile's accumulation jobs, in order: the group that needs exact
// segments (if any) first, then the other one; each segment is one job.
// Job k of the CTA accumulates into TMEM region k % 2 (256 columns), so the
// epilogue drains one region while the MMAs fill the other.
__device__ __forceinline__ int first_group(const SParams& p) { return p.seg_group == 1 ? 1 : 0; }

// Quantize-in-epilogue (Sec. 4.1, Conv2D + BatchNorm + Quantize fused): the
// next layer's packed codes of this lane's row from the fp16 outputs in the
// warp's staging tile (row `lane`, 128 columns from nc0, 64-column boxes of
// 128-byte-swizzled rows).  The columns are the next layer's packed
// positions, so each 32-column block is one packed block of its group (Sec. 3
// step 2 with the next layer's calibrated scale).  Kept out of the unrolled
// output loop, with run-time widths, so that the kernel's code stays small.
__device__ __forceinline__ void next_layer_codes(const SParams& p, uint32_t out_s, int lane, int m, int nc0) {
    const QConst kn0 = make_qconst(__ldg(p.s_next), p.next_bits[0]);
    const QConst kn1 = make_qconst(__ldg(p.s_next + 1), p.next_bits[1]);
#pragma unroll 1
    for (int b = 0; b < EPI_COLS / 32; ++b) {
        const int cb = nc0 + 32 * b;                       // first column of the block
        if (cb >= p.N) break;
        const int gn = cb >= p.next_pa0;
        const int jg = cb - (gn ? p.next_pa0 : 0);         // position within the group
        const QConst kn = gn ? kn1 : kn0;
        const int valid = (gn ? p.next_count[1] : p.next_count[0]) - jg;   // real channels in the block
        uint32_t o[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int cc = 4 * b + i;                      // 8-column chunk of the staging tile
            const uint32_t src = out_s + (uint32_t)(cc >> 3) * 4096u + (uint32_t)lane * 128u +
                                 ((((uint32_t)cc & 7u) ^ ((uint32_t)lane & 7u)) << 4);
            uint32_t h[4];
            asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(h[0]), "=r"(h[1]), "=r"(h[2]), "=r"(h[3])
                         : "r"(src)
                         : "memory");
            uint32_t u[8];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&h[e]));
                u[2 * e] = act_code_q<true>(f.x, kn.s, kn.r, kn.levels, kn.top);
                u[2 * e + 1] = act_code_q<true>(f.y, kn.s, kn.r, kn.levels, kn.top);
            }
            if (kn.mode != 1) {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&h[e]));
                    u[2 * e] = kn.mode == 0 ? 0u : act_code_q<false>(f.x, kn.s, kn.r, kn.levels, kn.top);
                    u[2 * e + 1] = kn.mode == 0 ? 0u : act_code_q<false>(f.y, kn.s, kn.r, kn.levels, kn.top);
                }
            }
#pragma unroll
            for (int q = 0; q < 8; ++q)
                if (8 * i + q >= valid) u[q] = 0u;         // padding positions hold code 0
            o[2 * i] = u[0] | (u[1] << 8) | (u[2] << 16) | (u[3] << 24);
            o[2 * i + 1] = u[4] | (u[5] << 8) | (u[6] << 16) | (u[7] << 24);
        }
        const int nb = gn ? p.next_bits[1] : p.next_bits[0];
        store_block32_rt(nb, o, p.Ap_next + m * (int64_t)p.next_row_bytes + (gn ? p.next_off[1] : p.next_off[0]) +
                                    (jg >> 5) * 4 * nb);
    }
}

// Scale runs along K (epilogue warp, one tile): every job is one run b of one
// group g, drained as its exact integer sum and added in fp32 with its own
// scale, y += s_a(g, b) s_w(n, g, b) / (La Lw) * Acc(g, b); then the tile's
// outputs.  `kw` is this warp's 128-float scratch for a run's column scales.
// With debug accumulators, acc_dbg receives [2][nb][M][N].  Returns false
// after a wait ran out.
__device__ __noinline__ bool runs_tile(const SParams& p, uint32_t sbase, uint32_t bar0, uint32_t abort_flag,
                                       uint32_t lane_base, uint32_t out_s, float* kw, int lane, int quad, int64_t m,
                                       int64_t m0, int nc0, uint32_t& job) {
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    float yr[EPI_COLS];
#pragma unroll
    for (int j = 0; j < EPI_COLS; ++j) yr[j] = 0.0f;
    const bool dbg = p.acc_dbg != nullptr && m < p.M;
    for (int g = 0; g < 2; ++g) {
        const int nrun = p.g[g].stages > 0 ? p.g[g].n_seg : 0;
        const float sc = p.g[g].acc_scale;
#pragma unroll 1
        for (int b = 0; b < nrun; ++b, ++job) {
            const uint32_t r = job & 1u, use = job >> 1;
            if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_REG_FULL + r), use & 1u, abort_flag, kTimeoutNs,
                                                      p.err, kErrWait)))
                return false;
            tc_fence_after();
            __syncwarp();
#pragma unroll
            for (int h = 0; h < EPI_COLS / 32; ++h) {
                const int c = lane + 32 * h;
                const int n = nc0 + c < p.N ? nc0 + c : p.N - 1;
                kw[c] = __ldg(p.s_w + ((int64_t)n * 2 + g) * p.nb + b) * p.g[g].inv_levels;
            }
            __syncwarp();
            const float sa = m < p.M ? __ldg(p.s_a + ((p.s_a_per_row ? m : 0) * 2 + g) * p.nb + b) : 0.0f;
            const uint32_t taddr = lane_base + r * REGION;
#pragma unroll
            for (int cc = 0; cc < EPI_COLS / 8; ++cc) {
                uint32_t v[8];
                tmem_ld8(taddr + cc * 8, v);
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const int j = cc * 8 + q;
                    const int32_t x = __float2int_rn(__uint_as_float(v[q]) * sc);
                    yr[j] = fmaf(sa * kw[j], (float)x, yr[j]);
                    if (dbg && nc0 + j < p.N)
                        p.acc_dbg[(((int64_t)g * p.nb + b) * p.M + m) * p.N + nc0 + j] = x;
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(BAR_REG_EMPTY + r));
        }
    }
    // the tile's outputs, 8 columns at a time
    if (p.y_tma) {
        if (lane == 0) bulk_wait_read0();
        __syncwarp();
    }
#pragma unroll
    for (int cc = 0; cc < EPI_COLS / 8; ++cc) {
        float y[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) y[q] = yr[cc * 8 + q];
        if (p.y_tma) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                if (p.out_bf16) {
                    __nv_bfloat162 h2 = __floats2bfloat162_rn(y[2 * e], y[2 * e + 1]);
                    w[e] = *reinterpret_cast<uint32_t*>(&h2);
                } else {
                    __half2 h2 = __floats2half2_rn(y[2 * e], y[2 * e + 1]);
                    w[e] = *reinterpret_cast<uint32_t*>(&h2);
                }
            }
            const uint32_t dst = out_s + (uint32_t)(cc >> 3) * 4096u + (uint32_t)lane * 128u +
                                 ((((uint32_t)cc & 7u) ^ ((uint32_t)lane & 7u)) << 4);
            asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(w[0]), "r"(w[1]), "r"(w[2]),
                         "r"(w[3])
                         : "memory");
        } else if (m < p.M) {
            store_out8(p, m, nc0 + cc * 8, y);
        }
    }
    if (p.y_tma) {
        fence_proxy_async_shared();
        __syncwarp();
        if (lane == 0) {
#pragma unroll
            for (int bx = 0; bx < EPI_COLS / 64; ++bx)
                tma_store_2d(&p.tma_y, nc0 + bx * 64, (int)(m0 + quad * 32), out_s + bx * 4096u);
            bulk_commit();
        }
    }
    return true;
}

// Instantiations: GENERAL = false compiles the common epilogue lean (no debug
// accumulators, outputs through TMA stores), which keeps the unrolled output
// loop small enough for the instruction cache; GENERAL = true handles the
// rest.  NEXT adds the next layer's codes (quantize-in-epilogue).
template <bool GENERAL, bool NEXT, int BNT, bool PAIR>
__global__ void __launch_bounds__(NUM_THREADS, 1) staged_mma_kernel(const __grid_constant__ SParams p) {
    // the tile width and what follows from it (BNT = 240: layouts with E2M1 groups,
    // whose block scale factors sit in the 16 TMEM columns past each region's tile)
    // PAIR: 2-SM MMAs.  CTAs run in clusters of two on a 256 x 256 tile: each
    // stages its own 128 A rows and its half of the B columns (32 KB per
    // K-stage instead of 48), the even-rank CTA issues M = 256 MMAs that read
    // both CTAs' stages, and each CTA's TMEM receives its own 128 rows.  Both
    // CTAs' operand bytes count on the issuing CTA's full barriers; its MMA
    // commits arrive on both CTAs' empty and region-full barriers; both CTAs'
    // epilogue warps arrive on its region-empty barriers.
    static_assert(!PAIR || (BNT / 2) % 8 == 0, "pairs split B boxes into halves of whole 8-row swizzle atoms");
    constexpr int BN = BNT;
    constexpr int B_BYTES = (PAIR ? BN / 2 : BN) * KSTAGE;
    constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    constexpr int EPI_COLS = BN / (NUM_EPI_WARPS / 4);
    constexpr int STAGES = PAIR ? PAIR_STAGES : staged::STAGES;
    constexpr int BAR_FULL = 0, BAR_EMPTY = STAGES, BAR_REG_FULL = 2 * STAGES, BAR_REG_EMPTY = 2 * STAGES + 2,
                  BAR_TEARDOWN = 2 * STAGES + 4, NUM_BARS = 2 * STAGES + 5;
    constexpr uint32_t IDESC2 = idesc(2 * BM, BN);
    constexpr uint32_t IDESC2_F4 = idesc_mxf4(2 * BM, BN);
    constexpr int SMEM_OUT = STAGES * STAGE_BYTES;
    constexpr int SMEM_COLS = SMEM_OUT + NUM_EPI_WARPS * OUT_PER_WARP;
    constexpr int SMEM_BAR = SMEM_COLS + NUM_EPI_WARPS * COLS_PER_WARP;
    constexpr int SMEM_MISC = SMEM_BAR + NUM_BARS * 8;
    constexpr uint32_t IDESC = idesc(BM, BN);
    constexpr uint32_t IDESC_F4 = idesc_mxf4(BM, BN);
    constexpr bool BOX8 = BN != 256;     // outputs leave in 8-column boxes (EPI_COLS is not a multiple of 64)
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sbase = smem_u32(smem);
    const uint32_t bar0 = smem_u32(smem + SMEM_BAR);
    auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + SMEM_MISC);
    const uint32_t abort_flag = smem_u32(smem + SMEM_MISC + 4);
    const uint32_t no_abort = smem_u32(smem + SMEM_MISC + 8);   // stays 0: waits that must run to completion
    const int g_first = first_group(p);
    if constexpr (PAIR) {
        // the pair instantiation works with cluster rank 1: outside a cluster
        // of two it reports the launch as invalid and does nothing
        if (cluster_size() != 2u) {
            if (threadIdx.x == 0) atomicOr(p.err, kErrWait);
            return;
        }
    }
    // the tiles this CTA walks: unit u of first_u, first_u + step_u, ... < n_units
    const uint32_t rank = PAIR ? cluster_rank() : 0u;
    const bool issuer = rank == 0u;                   // the CTA that issues the (2-SM) MMAs
    const int first_u = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
    const int step_u = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
    const int n_units = PAIR ? p.pair_tiles : p.total_tiles;
    const int mp = (p.m_tiles + 1) >> 1;
    auto tile_m = [&](int u) { return PAIR ? 2 * (u % mp) + (int)rank : u % p.m_tiles; };
    auto tile_n = [&](int u) { return PAIR ? u / mp : u / p.m_tiles; };

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(bar(BAR_FULL + i), 1);
            mbar_init(bar(BAR_EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(BAR_REG_FULL + i), 1);
            mbar_init(bar(BAR_REG_EMPTY + i), PAIR ? 2 * NUM_EPI_WARPS : NUM_EPI_WARPS);
        }
        mbar_init(bar(BAR_TEARDOWN), 1);
        set_flag(abort_flag, 0);
        set_flag(no_abort, 0);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == WARP_MMA) {
        if constexpr (PAIR) {
            // one warp of each CTA of the pair allocates, collectively
            asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(tmem_slot)),
                         "r"(512)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
        } else {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(tmem_slot)),
                         "r"(512)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    if constexpr (BN != REGION) {
        // the E2M1 block scale factors: UE8M0 2^0 in every byte of each region's
        // spare columns (one epilogue warp per TMEM lane quadrant)
        if (warp >= WARP_EPI && warp < WARP_EPI + 4) {
            const uint32_t lanes = (uint32_t)((warp & 3) * 32) << 16;
            tmem_st16(tmem_base + lanes + (uint32_t)BN_F4, 0x7F7F7F7Fu);
            tmem_st16(tmem_base + lanes + (uint32_t)(REGION + BN_F4), 0x7F7F7F7Fu);
        }
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }
    // both CTAs' barriers (and scale factors) are in place before the peer's
    // loads, arrivals or MMAs reach them
    if constexpr (PAIR) cluster_sync();
    // launched with launch_pdl: the expanded operands and weight sums are
    // written before this (the prologue above touches no global memory)
    pdl_wait();

    if (warp == WARP_TMA) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            uint32_t s = 0;
            bool ok = true;
            for (int u = first_u; u < n_units && ok; u += step_u) {
                const int m0 = tile_m(u) * BM, n0 = tile_n(u) * BN;
#pragma unroll 1
                for (int gi = 0; gi < 2 && ok; ++gi) {
                    const int g = gi == 0 ? g_first : 1 - g_first;
                    const int ns = p.g[g].stages, x0 = p.g[g].x0;
#pragma unroll 1
                    for (int i = 0; i < ns; ++i, ++s) {
                        const uint32_t slot = s % STAGES, ph = (s / STAGES) & 1u;
                        if (!wait_bounded(bar(BAR_EMPTY + slot), ph ^ 1u, abort_flag, kTimeoutNs, p.err, kErrWait)) {
                            ok = false;
                            break;
                        }
                        if (p.drop_first && s == 0) continue;   // the MMA's wait for it runs out
                        const uint32_t dst = sbase + slot * STAGE_BYTES;
                        if constexpr (PAIR) {
                            // this CTA's A rows and B half; both CTAs' bytes complete on the
                            // issuing CTA's full barrier
                            const uint32_t fb = mapa_shared(bar(BAR_FULL + slot), 0u);
                            if (issuer) mbar_arrive_expect_tx(bar(BAR_FULL + slot), 2 * STAGE_BYTES);
                            tma_load_2d_pair(dst, &p.tma_a, x0 + i * KSTAGE, m0, fb);
                            tma_load_2d_pair(dst + A_BYTES, &p.tma_b2, x0 + i * KSTAGE, n0 + (int)rank * (BN / 2), fb);
                        } else {
                            mbar_arrive_expect_tx(bar(BAR_FULL + slot), STAGE_BYTES);
                            tma_load_2d(dst, &p.tma_a, x0 + i * KSTAGE, m0, bar(BAR_FULL + slot));
                            tma_load_2d(dst + A_BYTES, &p.tma_b, x0 + i * KSTAGE, n0, bar(BAR_FULL + slot));
                        }
                    }
                }
            }
            // loads still in flight must land before the CTA's shared memory is released
            // (a pair's loads all complete on the issuing CTA's barriers; the other CTA
            // stays until the pair's final cluster barrier)
            if (!PAIR || issuer)
                for (uint32_t q = s > (uint32_t)STAGES ? s - STAGES : 0u; q < s; ++q)
                    if (!(p.drop_first && q == 0))
                        wait_bounded(bar(BAR_FULL + q % STAGES), (q / STAGES) & 1u, no_abort, kTimeoutNs, p.err,
                                     kErrWait);
        }
    } else if (warp == WARP_MMA) {
        // ------------------------------------------------------------------ MMA
        if (lane == 0 && issuer) {
            uint32_t s = 0, job = 0;
            bool ok = true;
            const uint64_t a_desc0 = KSTAGE == 128 ? sw128_desc(sbase) : sw64_desc(sbase);
            for (int u = first_u; u < n_units && ok; u += step_u) {
#pragma unroll 1
                for (int gi = 0; gi < 2 && ok; ++gi) {
                    const int g = gi == 0 ? g_first : 1 - g_first;
                    const int ns = p.g[g].stages;
                    const bool f8 = p.g[g].kind == 0, f4 = p.g[g].kind == 2;
                    const int per_job = p.g[g].n_seg > 1 ? p.g[g].seg_stages : ns;
#pragma unroll 1
                    for (int i = 0; i < ns && ok; ++job) {
                        const uint32_t r = job & 1u, use = job >> 1;
                        if (!wait_bounded(bar(BAR_REG_EMPTY + r), (use & 1u) ^ 1u, abort_flag, kTimeoutNs, p.err,
                                          kErrWait)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t d = tmem_base + r * REGION;
                        const int jn = per_job < ns - i ? per_job : ns - i;
#pragma unroll 1
                        for (int q = 0; q < jn; ++q, ++i, ++s) {
                            const uint32_t slot = s % STAGES, ph = (s / STAGES) & 1u;
                            if (!wait_bounded(bar(BAR_FULL + slot), ph, abort_flag, kTimeoutNs, p.err, kErrWait)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            // descriptors of this stage; +32 bytes of K is +2 in the start-address field
                            const uint64_t ad = a_desc0 + (uint64_t)((slot * STAGE_BYTES) >> 4);
                            const uint64_t bd = ad + (uint64_t)(A_BYTES >> 4);
                            if (PAIR && f4) {
                                // unit block scales in the spare columns of this region in both CTAs
                                const uint32_t sf = d + (uint32_t)BN_F4;
#pragma unroll
                                for (int k = 0; k < KSTAGE / 32; ++k)
                                    mma2_f4(d, ad + 2 * k, bd + 2 * k, IDESC2_F4, sf, sf + 8u, (q == 0 && k == 0) ? 0u : 1u);
                            } else if (PAIR && f8) {
#pragma unroll
                                for (int k = 0; k < KSTAGE / 32; ++k)
                                    mma2_f8<IDESC2>(d, ad + 2 * k, bd + 2 * k, (q == 0 && k == 0) ? 0u : 1u);
                            } else if (PAIR) {
#pragma unroll
                                for (int k = 0; k < KSTAGE / 32; ++k)
                                    mma2_f16<IDESC2>(d, ad + 2 * k, bd + 2 * k, (q == 0 && k == 0) ? 0u : 1u);
                            } else if (f8) {
#pragma unroll
                                for (int k = 0; k < KSTAGE / 32; ++k)
                                    mma_f8<IDESC>(d, ad + 2 * k, bd + 2 * k, (q == 0 && k == 0) ? 0u : 1u);
                            } else if (f4) {
                                // unit block scales (UE8M0 0x7F = 2^0) in this region's spare columns
                                const uint32_t sf = d + (uint32_t)BN_F4;
#pragma unroll
                                for (int k = 0; k < KSTAGE / 32; ++k)
                                    mma_f4(d, ad + 2 * k, bd + 2 * k, IDESC_F4, sf, sf + 8u,
                                           (q == 0 && k == 0) ? 0u : 1u);
                            } else {
#pragma unroll
                                for (int k = 0; k < KSTAGE / 32; ++k)
                                    mma_f16<IDESC>(d, ad + 2 * k, bd + 2 * k, (q == 0 && k == 0) ? 0u : 1u);
                            }
                            // the stage's slot is free again in both CTAs
                            if constexpr (PAIR) mma2_commit_mc(bar(BAR_EMPTY + slot), (uint16_t)0x3);
                            else mma_commit(bar(BAR_EMPTY + slot));
                        }
                        if (ok) {
                            if constexpr (PAIR) mma2_commit_mc(bar(BAR_REG_FULL + r), (uint16_t)0x3);
                            else mma_commit(bar(BAR_REG_FULL + r));
                        }
                    }
                }
            }
            // every issued MMA completes before TMEM and shared memory are released
            if constexpr (PAIR) mma2_commit(bar(BAR_TEARDOWN));
            else mma_commit(bar(BAR_TEARDOWN));
            wait_bounded(bar(BAR_TEARDOWN), 0u, no_abort, kTimeoutNs, p.err, kErrWait);
        }
    } else {
        // ------------------------------------------------------------- epilogue
        // Warp w reads TMEM lane quadrant w % 4 (rows 32*(w%4) .. +31 of the
        // tile) and the 128 columns cgrp*128 .. +127, cgrp = (w - 2) / 4.
        const int ew = warp - WARP_EPI;
        const int quad = warp & 3;
        const int cgrp = ew >> 2;
        const int row = quad * 32 + lane;
        const uint32_t lane_base = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(cgrp * EPI_COLS);
        // this warp's copy of the tile's column constants: {s_w0 * inv_levels0,
        // s_w1 * inv_levels1, center0 * C0, center1 * C1} per column
        float4* colc = reinterpret_cast<float4*>(smem + SMEM_COLS + ew * COLS_PER_WARP);
        const uint32_t out_s = sbase + (uint32_t)(SMEM_OUT + ew * OUT_PER_WARP);   // 1024-aligned
        // a drained TMEM region goes back to the CTA that issues the MMAs
        auto release_region = [&](uint32_t r) {
            if (PAIR && !issuer) mbar_arrive_cluster(mapa_shared(bar(BAR_REG_EMPTY + (int)r), 0u));
            else mbar_arrive(bar(BAR_REG_EMPTY + (int)r));
        };
        uint32_t job = 0;
        bool ok = true;
        for (int u = first_u; u < n_units && ok; u += step_u) {
            const int64_t m0 = (int64_t)tile_m(u) * BM;
            const int nc0 = tile_n(u) * BN + cgrp * EPI_COLS;    // this warp's first column
            __syncwarp();
#pragma unroll
            for (int h = 0; h < (EPI_COLS + 31) / 32; ++h) {
                const int c = lane + 32 * h;
                if (c >= EPI_COLS) break;
                const int n = nc0 + c < p.N ? nc0 + c : p.N - 1;
                float4 k;
                k.x = __ldg(p.s_w + (int64_t)n * 2) * p.g[0].inv_levels;
                k.y = __ldg(p.s_w + (int64_t)n * 2 + 1) * p.g[1].inv_levels;
                k.z = __int_as_float(p.g[0].center ? p.g[0].center * __ldg(p.colsum + (int64_t)n * 2) : 0);
                k.w = __int_as_float(p.g[1].center ? p.g[1].center * __ldg(p.colsum + (int64_t)n * 2 + 1) : 0);
                colc[c] = k;
            }
            __syncwarp();
            const int64_t m = m0 + row;
            float sa0 = 0.0f, sa1 = 0.0f;
            if (m < p.M) {
                sa0 = p.s_a_per_row ? __ldg(p.s_a + m * 2) : __ldg(p.s_a);
                sa1 = p.s_a_per_row ? __ldg(p.s_a + m * 2 + 1) : __ldg(p.s_a + 1);
            }
            if constexpr (GENERAL && BN == REGION) {
                if (p.runs) {
                    if (!runs_tile(p, sbase, bar0, abort_flag, lane_base, out_s, reinterpret_cast<float*>(colc), lane,
                                   quad, m, m0, nc0, job))
                        ok = false;
                    continue;
                }
            }
            // part: the exact accumulator of the first group (or the running
            // sum of the segments of the tile's only group)
            int32_t part[EPI_COLS];
#pragma unroll
            for (int j = 0; j < EPI_COLS; ++j) part[j] = 0;
            const int gA = g_first, gB = 1 - g_first;
            const int nA = p.g[gA].stages > 0 ? p.g[gA].n_seg : 0;
            const int nB = p.g[gB].stages > 0 ? p.g[gB].n_seg : 0;
            const int njobs = nA + nB;
            const int g_last = nB > 0 ? gB : gA;        // group of the final job
            const bool part_is_other = nA > 0 && nB > 0;
#pragma unroll 1
            for (int jj = 0; jj < njobs; ++jj, ++job) {
                const uint32_t r = job & 1u, use = job >> 1;
                if (!__all_sync(0xffffffffu, wait_bounded(bar(BAR_REG_FULL + r), use & 1u, abort_flag, kTimeoutNs,
                                                          p.err, kErrWait))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t taddr = lane_base + r * REGION;
                if (jj < njobs - 1) {
                    // accumulate: a whole first group, or a segment
                    const int gj = jj < nA ? gA : gB;
                    const float sc = p.g[gj].acc_scale;
#pragma unroll
                    for (int cc = 0; cc < EPI_COLS / 8; ++cc) {
                        uint32_t v[8];
                        tmem_ld8(taddr + cc * 8, v);
#pragma unroll
                        for (int q = 0; q < 8; ++q) part[cc * 8 + q] += __float2int_rn(__uint_as_float(v[q]) * sc);
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) release_region(r);
                    if (jj == nA - 1 && part_is_other) {
                        // the first group is complete: add back its centring
#pragma unroll
                        for (int j = 0; j < EPI_COLS; ++j) {
                            const float4 k = colc[j];
                            part[j] += __float_as_int(gA == 0 ? k.z : k.w);
                        }
                    }
                    continue;
                }
                // the final job: finish the tile's outputs, 8 columns at a time
                const float sc = p.g[g_last].acc_scale;
                const bool dbg = GENERAL && p.acc_dbg != nullptr && m < p.M;
                constexpr bool has_next = NEXT;
                const bool y_tma = GENERAL ? p.y_tma != 0 : true;
                const bool write_y = (GENERAL || NEXT) ? p.write_y != 0 : true;
                // fp16 outputs go through the staging tile for the TMA store and
                // for the next layer's quantizer
                const bool staged_out = y_tma || has_next;
                if (staged_out) {
                    // the previous tile's store must have read the staging buffer
                    if (lane == 0) bulk_wait_read0();
                    __syncwarp();
                }
#pragma unroll
                for (int cc = 0; cc < EPI_COLS / 8; ++cc) {
                    uint32_t v[8];
                    tmem_ld8(taddr + cc * 8, v);
                    const int nb = nc0 + cc * 8;
                    float y[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const int j = cc * 8 + q;
                        const float4 k = colc[j];
                        const int32_t x = __float2int_rn(__uint_as_float(v[q]) * sc) +
                                          __float_as_int(g_last == 0 ? k.z : k.w);
                        const int32_t last = part_is_other ? x : part[j] + x;     // the final job's group
                        const int32_t other = part_is_other ? part[j] : 0;
                        const int32_t a0 = g_last == 0 ? last : other;
                        const int32_t a1 = g_last == 0 ? other : last;
                        y[q] = fmaf(sa1 * k.y, (float)a1, sa0 * k.x * (float)a0);
                        if (dbg && nb + q < p.N) {
                            p.acc_dbg[m * p.N + nb + q] = a0;
                            p.acc_dbg[(p.M + m) * p.N + nb + q] = a1;
                        }
                    }
                    if (staged_out) {
                        uint32_t w[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            if (p.out_bf16) {
                                __nv_bfloat162 h2 = __floats2bfloat162_rn(y[2 * e], y[2 * e + 1]);
                                w[e] = *reinterpret_cast<uint32_t*>(&h2);
                            } else {
                                __half2 h2 = __floats2half2_rn(y[2 * e], y[2 * e + 1]);
                                w[e] = *reinterpret_cast<uint32_t*>(&h2);
                            }
                        }
                        // box cc / 8 (64 columns), row `lane`, 16-byte chunk cc % 8, 128-byte swizzle
                        // (the TMA store map's layout); with 8-column boxes, box cc of 32 x 16 bytes
                        const uint32_t dst =
                            BOX8 ? out_s + (uint32_t)cc * 512u + (uint32_t)lane * 16u
                                 : out_s + (uint32_t)(cc >> 3) * 4096u + (uint32_t)lane * 128u +
                                       ((((uint32_t)cc & 7u) ^ ((uint32_t)lane & 7u)) << 4);
                        asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(w[0]), "r"(w[1]),
                                     "r"(w[2]), "r"(w[3])
                                     : "memory");
                    }
                    if (write_y && !y_tma && m < p.M) store_out8(p, m, nb, y);
                }
                tc_fence_before();
                if (staged_out) fence_proxy_async_shared();
                __syncwarp();
                if (lane == 0) {
                    release_region(r);
                    if (y_tma && write_y) {
                        // rows and columns beyond M and N are clipped by the store
                        if constexpr (BOX8) {
#pragma unroll
                            for (int bx = 0; bx < EPI_COLS / 8; ++bx)
                                tma_store_2d(&p.tma_y, nc0 + bx * 8, (int)(m0 + quad * 32), out_s + bx * 512u);
                        } else {
#pragma unroll
                            for (int bx = 0; bx < EPI_COLS / 64; ++bx)
                                tma_store_2d(&p.tma_y, nc0 + bx * 64, (int)(m0 + quad * 32), out_s + bx * 4096u);
                        }
                        bulk_commit();
                    }
                }
                if constexpr (BN == REGION) {
                    if (has_next && m < p.M) next_layer_codes(p, out_s, lane, m, nc0);
                }
            }
        }
        if (((GENERAL || NEXT) ? p.y_tma && p.write_y : true) && lane == 0) bulk_wait0();   // stores complete before the CTA exits
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // the peer multicasts into this CTA's stages and arrives on its barriers until it is done
    if constexpr (PAIR) cluster_sync();
    if (warp == WARP_MMA) {
        if constexpr (PAIR)
            asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
        else
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
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

// 2-D map over expanded rows [rows][row_bytes] with a box of one 128-byte
// K-stage by box_rows rows, 128-byte swizzle (the layout the MMA descriptors read).
bool encode_rows(EncodeTiledFn enc, CUtensorMap* map, const uint8_t* base, int64_t row_bytes, int64_t rows,
                 int box_rows) {
    cuuint64_t dims[2] = {(cuuint64_t)row_bytes, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
    cuuint32_t box[2] = {(cuuint32_t)KSTAGE, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, KSTAGE == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int64_t align1k(int64_t x) { return (x + 1023) / 1024 * 1024; }

}  // namespace staged

bool staged_plan(const LayoutGeom& geo, StagedPlan* sp, bool allow_f4) {
    int nseg_groups = 0;
    int64_t x0 = 0;
    sp->seg_group = -1;
    sp->f4 = 0;
    const bool runs = geo.sub_k > 0;
    // E2M1 pays where its groups hold most of the K codes: the 240-column tiles
    // it needs cost the other group (measured on the 8192 x 4096 x 4096 sweep:
    // +20 % with all codes in E2M1 groups, +6 % at 75 %, -5 % at 50 %)
    if (allow_f4) {
        int64_t f4_codes = 0, all_codes = 0;
        for (int g = 0; g < 2; ++g) {
            const GroupGeom& G = geo.g[g];
            all_codes += G.pw;
            if (G.bits_a <= 2 && G.bits_w <= 2 && geo.act_kind[g] == SONIQ_ACT_UNSIGNED && !runs && G.count > 0)
                f4_codes += G.pw;
        }
        if (f4_codes * 5 < all_codes * 3) allow_f4 = false;
        // and where K is long enough for the MMAs to dominate: at K = 768 (the
        // 16384 x 768 -> 3072 MLP layer) the tile's epilogue sets the pace, and
        // the 240-column epilogue (120 columns per warp, 8-column store boxes)
        // was 10 % slower than the 256-column one
        if (all_codes < 2048) allow_f4 = false;
    }
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = geo.g[g];
        StagedGroup& S = sp->g[g];
        const int ak = geo.act_kind[g];
        S.kind = (G.bits_a <= 4 && G.bits_w <= 4) ? 0 : 1;
        // E2M1 holds 0, 0.5, 1, 1.5, 2: codes u <= 3 and |j| <= 2 are exact as code / 2
        if (allow_f4 && G.bits_a <= 2 && G.bits_w <= 2 && ak == SONIQ_ACT_UNSIGNED && !runs && G.count > 0) {
            S.kind = 2;
            sp->f4 = 1;
        }
        // E2M1 rows: two codes per byte, padded to whole 256-code stages
        const int64_t bytes = S.kind == 2 ? (((int64_t)G.pw + 255) / 256 * 256) / 2
                                          : (int64_t)G.pw * (S.kind == 0 ? 1 : 2);
        S.stages = (int32_t)(bytes / staged::KSTAGE);
        S.x0 = (int32_t)x0;
        x0 += bytes;
        // unsigned fp16 activations are centred (halving the products) unless every
        // run is scaled on its own, where the centring's weight sums would be per run
        S.center = (S.kind == 1 && ak == SONIQ_ACT_UNSIGNED && !runs) ? (1 << (G.bits_a - 1)) : 0;
        const int64_t amax = ak == SONIQ_ACT_PM1 ? 1
                                                 : (ak == SONIQ_ACT_SIGNED || S.center ? (int64_t)1 << (G.bits_a - 1)
                                                                                       : (1 << G.bits_a) - 1);
        const int64_t wmax = ak == SONIQ_ACT_PM1 ? 1 : (int64_t)1 << (G.bits_w - 1);
        const int64_t maxprod = amax * wmax;
        const int64_t codes_per_stage = S.kind == 2 ? 2 * staged::KSTAGE : (S.kind == 0 ? staged::KSTAGE : staged::KSTAGE / 2);
        int64_t seg_stages = ((int64_t)1 << 24) / maxprod / codes_per_stage;
        if (runs) {
            // one job per run; its exact sum must stay within 2^24
            if ((int64_t)geo.sub_k * maxprod > ((int64_t)1 << 24)) return false;
            seg_stages = geo.sub_k / codes_per_stage;
        }
        if (seg_stages < 1) return false;
        S.seg_stages = (int32_t)(seg_stages < S.stages ? seg_stages : (S.stages > 0 ? S.stages : 1));
        S.n_seg = S.stages > 0 ? (S.stages + S.seg_stages - 1) / S.seg_stages : 0;
        if (S.n_seg > 1 && !runs) {
            ++nseg_groups;
            sp->seg_group = g;
        }
    }
    if (nseg_groups > 1) return false;
    sp->eb = x0;
    return x0 > 0 && x0 % 128 == 0;
}

int64_t staged_scratch_bytes(const LayoutGeom& geo, int64_t rows_a, int64_t N) {
    StagedPlan sp;
    if (!staged_plan(geo, &sp)) return 0;
    return staged::align1k(rows_a * sp.eb) + staged::align1k(N * sp.eb) + staged::align1k(N * 8);
}

cudaError_t launch_staged(const LayoutGeom& geo, const MmaArgs& a, void* scratch, size_t scratch_bytes,
                          cudaStream_t st) {
    using namespace staged;
    StagedPlan sp;
    // E2M1 groups need 240-column tiles: not with a next layer (its codes are
    // packed from 64-column output boxes), nor where the narrower tiles would
    // add more than 7 % of padded columns (N = 256 would take two tiles)
    const bool f4_ok = a.next == nullptr && (int64_t)((a.N + BN_F4 - 1) / BN_F4) * BN_F4 * 100 <= (int64_t)a.N * 107;
    if (!staged_plan(geo, &sp, f4_ok)) return cudaErrorNotSupported;
    const int tile_n = sp.f4 ? BN_F4 : BN;
    const int64_t rows_a = a.M;
    if ((int64_t)scratch_bytes < staged_scratch_bytes(geo, rows_a, a.N) || scratch == nullptr ||
        (uintptr_t)scratch % 256 != 0)
        return cudaErrorNotSupported;
    uint8_t* xa = static_cast<uint8_t*>(scratch);
    uint8_t* xw = xa + align1k(rows_a * sp.eb);
    int32_t* colsum = reinterpret_cast<int32_t*>(xw + align1k((int64_t)a.N * sp.eb));
    const int taps = a.conv ? a.R * a.S : 1;

    // ---- expand activations (im2col for a convolution) and weights ----
    ExpandParams e;
    memset(&e, 0, sizeof(e));
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = geo.g[g];
        e.bits[g] = G.bits_a;
        e.kind[g] = sp.g[g].kind;
        e.src_off[g] = G.a_off;
        e.dst_off[g] = sp.g[g].x0;
        e.blk_src[g] = G.pa / 32;
        // E2M1 groups are written out to whole 256-code stages (zero codes)
        e.blk_dst[g] = (sp.g[g].kind == 2 ? (G.pw + 255) / 256 * 256 : G.pw) / 32;
        e.center[g] = sp.g[g].center;
        e.cpt[g] = G.pa / 32 > 0 ? G.pa / 32 : 1;
        e.cpt_magic[g] = (((uint64_t)1 << 32) + (uint64_t)e.cpt[g] - 1) / (uint64_t)e.cpt[g];
        e.vec16[g] = (G.a_off % 16 == 0 && geo.a_row_bytes % 16 == 0 && (uintptr_t)a.Ap % 16 == 0) ? 1 : 0;
        e.code_kind[g] = geo.act_kind[g];
        e.count[g] = G.count;
    }
    e.src = a.Ap;
    e.src_row_bytes = geo.a_row_bytes;
    e.dst = xa;
    e.dst_row_bytes = sp.eb;
    e.rows = rows_a;
    e.is_weight = 0;
    e.conv = a.conv;
    e.H = a.H; e.W = a.W; e.P = a.P; e.Q = a.Q; e.R = a.R; e.S = a.S;
    e.sh = a.sh; e.sw = a.sw; e.ph = a.ph; e.pw = a.pw;
    (void)taps;
    auto grid_for = [](int64_t items) {
        int64_t ctas = (items + 7) / 8;                        // 8 warps per CTA, one (row, group) per warp
        const int64_t cap = (int64_t)num_sms() * 16;
        return (int)(ctas < 1 ? 1 : (ctas > cap ? cap : ctas));
    };
    ExpandParams w = e;
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = geo.g[g];
        w.bits[g] = G.bits_w;
        w.src_off[g] = G.w_off;
        w.blk_src[g] = G.pw / 32;
        w.center[g] = 0;
        w.vec16[g] = (G.w_off % 16 == 0 && geo.w_row_bytes % 16 == 0 && (uintptr_t)a.Wp % 16 == 0) ? 1 : 0;
        w.code_kind[g] = geo.act_kind[g] == SONIQ_ACT_PM1 ? 2 : 1;
    }
    w.src = a.Wp;
    w.src_row_bytes = geo.w_row_bytes;
    w.dst = xw;
    w.rows = a.N;
    w.is_weight = 1;
    w.colsum = colsum;
    w.conv = 0;
    // activations and weights in one launch
    cudaError_t err = launch_pdl(expand_kernel, dim3((unsigned)grid_for(rows_a * 2 + (int64_t)a.N * 2)), dim3(256), 0,
                                 st, e, w);
    note_launch();
    if (err != cudaSuccess) return err;

    // ---- the GEMM ----
    SParams p;
    memset(&p, 0, sizeof(p));
    EncodeTiledFn enc = encode_fn();
    if (enc == nullptr) return cudaErrorNotSupported;
    if (!encode_rows(enc, &p.tma_a, xa, sp.eb, rows_a, BM) || !encode_rows(enc, &p.tma_b, xw, sp.eb, a.N, tile_n))
        return cudaErrorInvalidValue;
    p.s_a = a.s_a;
    p.s_w = a.s_w;
    p.colsum = colsum;
    p.Y = a.Y;
    p.acc_dbg = a.acc_dbg;
    p.err = device_error_word();
    if (p.err == nullptr) return cudaErrorUnknown;
    p.M = a.M;
    p.N = a.N;
    p.m_tiles = (int32_t)((a.M + BM - 1) / BM);
    p.n_tiles = (a.N + tile_n - 1) / tile_n;
    p.total_tiles = p.m_tiles * p.n_tiles;
    p.s_a_per_row = a.s_a_per_row;
    p.out_bf16 = a.out_bf16;
    p.seg_group = sp.seg_group;
    p.drop_first = (a.flags & SONIQ_FLAG_TEST_DROP_ARRIVE) != 0 ? 1 : 0;
    p.write_y = a.Y != nullptr;
    if (a.next != nullptr) {
        p.has_next = 1;
        p.s_next = a.next_s_a;
        p.Ap_next = a.next_Ap;
        p.next_row_bytes = a.next->a_row_bytes;
        p.next_pa0 = a.next->g[0].pa;
        for (int g = 0; g < 2; ++g) {
            p.next_count[g] = a.next->g[g].count;
            p.next_bits[g] = a.next->g[g].bits_a;
            p.next_off[g] = a.next->g[g].a_off;
        }
    }
    // outputs through TMA stores when the row pitch allows a tensor map (N * 2 bytes a multiple of 16)
    p.y_tma = 0;
    if (p.write_y && a.N % 8 == 0 && (uintptr_t)a.Y % 16 == 0) {
        cuuint64_t dims[2] = {(cuuint64_t)a.N, (cuuint64_t)a.M};
        cuuint64_t strides[1] = {(cuuint64_t)a.N * 2};
        // 64 x 32 boxes, 128-byte swizzled; 240-column tiles (120 columns per warp) use 8 x 32 boxes
        cuuint32_t box[2] = {sp.f4 ? 8u : 64u, 32u};
        cuuint32_t estr[2] = {1, 1};
        if (enc(&p.tma_y, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, a.Y, dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, sp.f4 ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
        p.y_tma = 1;
    }
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = geo.g[g];
        SGroup& S = p.g[g];
        S.kind = sp.g[g].kind;
        S.stages = sp.g[g].stages;
        S.x0 = sp.g[g].x0;
        S.seg_stages = sp.g[g].seg_stages;
        S.n_seg = sp.g[g].n_seg;
        S.center = sp.g[g].center;
        S.acc_scale = S.kind == 0 ? 262144.0f : (S.kind == 2 ? 4.0f : 1.0f);   // 2^18, 1, or 4 (products u j / 4)
        // decode levels: activations 2^na - 1 (unsigned), 2^(na-1) (signed) or 1 (+-1);
        // weights 2^(nw-1) or 1 (+-1)
        const int ak = geo.act_kind[g];
        const double la = ak == SONIQ_ACT_PM1 ? 1.0 : (ak == SONIQ_ACT_SIGNED ? (double)(1 << (G.bits_a - 1))
                                                                             : (double)((1 << G.bits_a) - 1));
        const double lw = ak == SONIQ_ACT_PM1 ? 1.0 : (double)(1 << (G.bits_w - 1));
        S.inv_levels = (float)(1.0 / (la * lw));
    }
    // kernel instantiation: debug accumulators, outputs that cannot leave by
    // TMA stores, or no outputs at all take the general epilogue
    p.runs = geo.sub_k > 0 ? 1 : 0;
    p.nb = geo.nb;
    const bool general = a.acc_dbg != nullptr || p.runs || (p.write_y && !p.y_tma) ||
                         (!p.write_y && !p.has_next) || p.drop_first;
    // 2-SM pairs on 256 x 256 tiles: the lean epilogue on 256-column tiles, for
    // rows of at least 3072 codes (launched as clusters of two; each CTA loads
    // 128-row halves of the B tile).  A pair waits for the slower of its two
    // epilogues before it reuses a TMEM region, so where the epilogue sets the
    // pace (short K: the K = 768 MLP layer, 123 -> 138 us as pairs; the
    // K = 2304 conv, even) and for the next-layer epilogue, whose drain is
    // longer, one CTA takes one tile.
    int64_t row_codes = 0;
    for (int g = 0; g < 2; ++g) row_codes += geo.g[g].pw;
    const bool pair = !general && !p.has_next && row_codes >= 3072;
    p.pair_tiles = ((p.m_tiles + 1) / 2) * p.n_tiles;
    if (pair && !encode_rows(enc, &p.tma_b2, xw, sp.eb, a.N, tile_n / 2)) return cudaErrorInvalidValue;
    void (*kern)(SParams) =
        sp.f4 ? (general ? staged_mma_kernel<true, false, BN_F4, false>
                 : pair  ? staged_mma_kernel<false, false, BN_F4, true>
                         : staged_mma_kernel<false, false, BN_F4, false>)
        : general ? (p.has_next ? staged_mma_kernel<true, true, BN, false> : staged_mma_kernel<true, false, BN, false>)
                  : p.has_next ? staged_mma_kernel<false, true, BN, false>
                  : pair       ? staged_mma_kernel<false, false, BN, true>
                               : staged_mma_kernel<false, false, BN, false>;
    static bool attr_done[64][8] = {};
    static int max_pairs[64][2] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    const int kidx = sp.f4 ? (pair ? 7 : 4 + (general ? 1 : 0)) : pair ? 6 : (general ? 2 : 0) + (p.has_next ? 1 : 0);
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    const int smem_alloc = pair ? pair_smem_alloc() : SMEM_ALLOC;
    cfg.blockDim = dim3(NUM_THREADS, 1, 1);
    cfg.dynamicSmemBytes = smem_alloc;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (!attr_done[dev][kidx]) {
        if ((err = cudaFuncSetAttribute((const void*)kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_alloc)) !=
            cudaSuccess)
            return err;
        if ((err = prefer_max_shared((const void*)kern)) != cudaSuccess) return err;
        if (pair) {
            // pairs that can be resident at once (one CTA per SM)
            cfg.gridDim = dim3(2 * (unsigned)num_sms() / 2, 1, 1);
            int n = 0;
            if ((err = cudaOccupancyMaxActiveClusters(&n, (const void*)kern, &cfg)) != cudaSuccess) return err;
            max_pairs[dev][sp.f4 ? 1 : 0] = n;
        }
        attr_done[dev][kidx] = true;
    }
    if (pair) {
        int pairs = max_pairs[dev][sp.f4 ? 1 : 0];
        if (pairs < 1) return cudaErrorNotSupported;
        if (pairs > p.pair_tiles) pairs = p.pair_tiles;
        cfg.gridDim = dim3(2 * (unsigned)pairs, 1, 1);
        cfg.numAttrs = 2;
        if ((err = cudaLaunchKernelEx(&cfg, kern, p)) != cudaSuccess) return err;
    } else {
        const int grid = p.total_tiles < num_sms() ? p.total_tiles : num_sms();
        if ((err = launch_pdl(kern, dim3((unsigned)grid), dim3(NUM_THREADS), (size_t)smem_alloc, st, p)) !=
            cudaSuccess)
            return err;
    }
    note_launch();
    return cudaGetLastError();
}

}  // namespace soniq
