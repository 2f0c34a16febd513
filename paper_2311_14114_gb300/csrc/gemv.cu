// Small-M mixed-precision GEMV (M <= 16): the decode-shaped case where the
// packed weight bytes streamed from HBM are the roofline (Sec. 2.4 C5).
//
// Exact integer arithmetic on CUDA cores (Sec. 4.2: unsigned x signed
// integer dot products):
//   * each CTA expands the activation codes (M rows) once into shared memory
//     as bytes, with their per-group row sums R_g[m];
//   * weight rows are contiguous in HBM; each SM takes a contiguous range of
//     them and requests all of it at once, one bulk copy per row into shared
//     memory (in rounds if the range does not fit);
//   * the sign bit of every weight code is flipped (j -> j + 2^(n-1),
//     unsigned) and dp4a(u, j + 2^(n-1)) accumulates in uint32, from the
//     packed slices directly (M <= 2) or from codes expanded to bytes;
//   * Acc_g = sum - 2^(n-1) * R_g[m], exact; the fp32 epilogue applies the
//     group scales (decode rules of Sec. 3 steps 2-3).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "soniq_device.cuh"
#include "soniq_internal.h"

namespace soniq {
namespace {

struct GemvParams {
    const uint8_t* Ap;
    const uint8_t* Wp;
    const float* s_a;
    const float* s_w;
    void* Y;
    int32_t* acc_dbg;
    int32_t M, N;
    int32_t a_row_bytes, w_row_bytes;
    int32_t s_a_per_row, out_bf16;
    GroupGeom g[2];
    int32_t a_s_off[2];   // byte offset of group g's activation bytes in shared memory
    int32_t a_m_stride[2];// bytes per activation row of group g in shared memory
    int32_t sum_off;      // per-row totals of a round [2][MT][round_rows]
    int32_t scale_off;    // weight scales of a round [round_rows][2]
    int32_t rows_cta;     // weight rows per CTA (the last CTA may have fewer)
    int32_t round_rows;   // weight rows per round through shared memory
    int32_t bar_off;      // one mbarrier per 16-row piece of a round
    int32_t buf_off;      // the round's weight rows
    int32_t wstride;      // bytes between weight rows in the buffer
    unsigned* err;        // device error word (a bounded wait ran out)
    long long timeout_ns;
};

// Activation chunk c (128 codes) of a row sits at c * A_CHUNK: 16 bytes of
// padding per chunk put the chunks of consecutive lanes on different banks.
constexpr int A_CHUNK = 144;

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

// Mask of the top code bit in every field of a w-bit slice word: flipping it
// turns n-bit two's complement j into offset binary j + 2^(n-1).
__host__ __device__ constexpr uint32_t top_bit_mask(int w) {
    return w == 8 ? 0x80808080u : w == 4 ? 0x88888888u : w == 2 ? 0xAAAAAAAAu : 0xFFFFFFFFu;
}

// Sum over a block of u * (w-bit slice field), the slice's w words at `sw`:
// field k of every byte of slice word q belongs to codes 4t..4t+3 with
// t = q*(8/w) + k, next to activation word a[t].  The field is masked in place
// rather than shifted down, so s[k] collects 2^(w*k) times its products; the
// caller shifts it down once per chunk (exact: every term carries that factor).
template <int W>
__device__ __forceinline__ void slice_dot_masked(const uint32_t* sw, const uint32_t* a, uint32_t (&s)[8 / W]) {
    constexpr int PER = 8 / W;
    constexpr uint32_t MASK = W == 8 ? 0xFFFFFFFFu : W == 4 ? 0x0F0F0F0Fu : W == 2 ? 0x03030303u : 0x01010101u;
#pragma unroll
    for (int q = 0; q < W; ++q)
#pragma unroll
        for (int k = 0; k < PER; ++k) s[k] = __dp4a(sw[q] & (MASK << (W * k)), a[q * PER + k], s[k]);
}

// One 128-code chunk (4 blocks, 16*NW bytes, in shared memory) of one weight
// row against MT rows of activation bytes (chunk-padded layout, `astride`
// bytes per row): acc[m] += sum over the chunk of u * (j + 2^(n-1)).  The
// slices of the packed codes are used directly (weights are never expanded
// to bytes); the slice holding the top code bit is flipped to offset binary.
template <int NW, int MT>
__device__ __forceinline__ void gemv_chunk_w(uint32_t (&w)[4 * NW], uint32_t a_s, int astride, int M,
                                             uint32_t (&acc)[MT]) {
    // slice widths, low bits first; the last slice holds the top bit
    constexpr int W0 = NW == 8 ? 8 : (NW & 4), W1 = NW == 8 ? 0 : (NW & 2), W2 = NW == 8 ? 0 : (NW & 1);
    constexpr int WT = W2 ? W2 : (W1 ? W1 : W0);
    constexpr int OFF1 = W0, OFF2 = W0 + W1;
    if constexpr (MT > 2) {
        // several activation rows: expand each block to bytes once, reuse it per row
        const uint32_t flip = sign_flip_mask(NW);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            uint32_t wb[8];
            block_to_bytes<NW>(w + NW * i, wb);
#pragma unroll
            for (int t = 0; t < 8; ++t) wb[t] ^= flip;
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                if (m < M) {
                    const uint32_t aa = a_s + (uint32_t)(m * astride + i * 32);
                    const uint4 x0 = lds128(aa), x1 = lds128(aa + 16);
                    // two short chains per block instead of one long one
                    uint32_t e = __dp4a(wb[0], x0.x, 0u), o = __dp4a(wb[1], x0.y, 0u);
                    e = __dp4a(wb[2], x0.z, e);
                    o = __dp4a(wb[3], x0.w, o);
                    e = __dp4a(wb[4], x1.x, e);
                    o = __dp4a(wb[5], x1.y, o);
                    e = __dp4a(wb[6], x1.z, e);
                    o = __dp4a(wb[7], x1.w, o);
                    acc[m] += e + o;
                }
            }
        }
        return;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        uint32_t* blk = w + NW * i;
        // flip the top code bit: it sits in the last slice's words
        constexpr int FIRST_TOP = NW - WT;
#pragma unroll
        for (int q = FIRST_TOP; q < NW; ++q) blk[q] ^= top_bit_mask(WT);
    }
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        if (m < M) {
            // one partial sum per slice and field position, over the chunk's four
            // blocks (independent chains); each is shifted down once at the end
            constexpr int P0 = W0 ? 8 / W0 : 1, P1 = W1 ? 8 / W1 : 1, P2 = W2 ? 8 / W2 : 1;
            uint32_t s0[P0], s1[P1], s2[P2];
#pragma unroll
            for (int k = 0; k < P0; ++k) s0[k] = 0u;
#pragma unroll
            for (int k = 0; k < P1; ++k) s1[k] = 0u;
#pragma unroll
            for (int k = 0; k < P2; ++k) s2[k] = 0u;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t aa = a_s + (uint32_t)(m * astride + i * 32);
                const uint4 x0 = lds128(aa), x1 = lds128(aa + 16);
                const uint32_t a[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
                const uint32_t* blk = w + NW * i;
                if constexpr (W0 > 0) slice_dot_masked<W0 ? W0 : 1>(blk, a, s0);
                if constexpr (W1 > 0) slice_dot_masked<W1 ? W1 : 1>(blk + W0, a, s1);
                if constexpr (W2 > 0) slice_dot_masked<W2 ? W2 : 1>(blk + W0 + W1, a, s2);
            }
            uint32_t t0 = 0u, t1 = 0u, t2 = 0u;
#pragma unroll
            for (int k = 0; k < P0; ++k) t0 += s0[k] >> (W0 * k);
#pragma unroll
            for (int k = 0; k < P1; ++k) t1 += s1[k] >> (W1 * k);
#pragma unroll
            for (int k = 0; k < P2; ++k) t2 += s2[k] >> (W2 * k);
            acc[m] += t0 + (t1 << OFF1) + (t2 << OFF2);
        }
    }
}

// The same for a chunk whose 16*NW weight bytes are in shared memory.
template <int NW, int MT>
__device__ __forceinline__ void gemv_chunk(uint32_t wsrc, uint32_t a_s, int astride, int M, uint32_t (&acc)[MT]) {
    uint32_t w[4 * NW];
#pragma unroll
    for (int q = 0; q < NW; ++q) {
        const uint4 v = lds128(wsrc + 16 * q);
        w[4 * q] = v.x;
        w[4 * q + 1] = v.y;
        w[4 * q + 2] = v.z;
        w[4 * q + 3] = v.w;
    }
    gemv_chunk_w<NW, MT>(w, a_s, astride, M, acc);
}

__device__ __forceinline__ uint32_t smem_addr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ bool gemv_wait(uint32_t bar, uint32_t parity, const GemvParams& p) {
    long long t0 = 0;
    for (uint32_t it = 0;; ++it) {
        uint32_t ok;
        // the thread sleeps in the barrier until the phase completes (or 20 us pass)
        asm volatile("{\n\t.reg .pred q;\n\tmbarrier.try_wait.parity.shared::cta.b64 q, [%1], %2, 20000;\n\tselp.u32 %0, 1, 0, q;\n\t}"
                     : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
        if (ok) return true;
        if ((it & 3u) == 3u) {
            long long t;
            asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
            if (t0 == 0) t0 = t;
            else if (t - t0 > p.timeout_ns) {
                atomicOr(p.err, 1u);
                return false;
            }
        }
    }
}

// ---- the whole share of the weight rows in flight at once ------------------
//
// One CTA per SM takes a contiguous range of weight rows.  At its start warp
// 0 issues one bulk copy per row into shared memory (rows at an odd multiple
// of 16 bytes apart), so every SM asks HBM for all of its rows at once; the
// rows land in pieces of 16, each with its own barrier, while the CTA expands
// the activation codes.  A task is one 128-code chunk of the 16 rows of a
// piece: half-warp h takes tasks h, h + 64, ... (lane = row, so weight reads
// are conflict-free and activation reads are broadcasts) as soon as their
// piece has landed, and adds its partial sums into per-row shared totals.
constexpr int kBulkMaxM = 16;

// 1024 threads (64 registers each) for up to four activation rows; 512 (128
// registers) for more, whose per-row sums and expanded blocks need the room.
template <int MT>
constexpr int bulk_threads() { return MT <= 4 ? 1024 : 512; }
constexpr int kPieceRows = 16;
constexpr int kMaxPieces = 8;

template <int MT>
__device__ __forceinline__ void bulk_task(const GemvParams& p, int g, int nw, uint32_t wsrc, uint32_t a_s,
                                          uint32_t (&acc)[MT]) {
    const int astride = p.a_m_stride[g];
    switch (nw) {
        case 1: gemv_chunk<1, MT>(wsrc, a_s, astride, p.M, acc); break;
        case 2: gemv_chunk<2, MT>(wsrc, a_s, astride, p.M, acc); break;
        case 3: gemv_chunk<3, MT>(wsrc, a_s, astride, p.M, acc); break;
        case 4: gemv_chunk<4, MT>(wsrc, a_s, astride, p.M, acc); break;
        case 5: gemv_chunk<5, MT>(wsrc, a_s, astride, p.M, acc); break;
        case 6: gemv_chunk<6, MT>(wsrc, a_s, astride, p.M, acc); break;
        case 7: gemv_chunk<7, MT>(wsrc, a_s, astride, p.M, acc); break;
        default: gemv_chunk<8, MT>(wsrc, a_s, astride, p.M, acc); break;
    }
}

template <int MT>
__global__ void __launch_bounds__(bulk_threads<MT>(), 1) gemv_bulk_kernel(const GemvParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    int32_t* rowsum = reinterpret_cast<int32_t*>(smem);                  // [2][16]
    uint32_t* acc_s = reinterpret_cast<uint32_t*>(smem + p.sum_off);     // [2][MT][round rows]
    float* sw_s = reinterpret_cast<float*>(smem + p.scale_off);          // [round rows][2] weight scales
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rows_cta = p.rows_cta, round_rows = p.round_rows;
    const int64_t n_begin = (int64_t)blockIdx.x * rows_cta;
    const int64_t n_end = n_begin + rows_cta < p.N ? n_begin + rows_cta : p.N;
    const int nch0 = p.g[0].pw / 128, nch1 = p.g[1].pw / 128, tpp = nch0 + nch1;   // tasks per piece
    const uint32_t wbuf = smem_addr(smem + p.buf_off);

    if (threadIdx.x == 0) {
        for (int i = 0; i < kMaxPieces; ++i)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(smem + p.bar_off + 8 * i)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x < 32) rowsum[threadIdx.x] = 0;
    __syncthreads();

    bool ok = true;
    int round = 0;
    for (int64_t n0 = n_begin; n0 < n_end; n0 += round_rows, ++round) {
        const int nr = (int)(n_end - n0 < round_rows ? n_end - n0 : round_rows);
        const int npieces = (nr + kPieceRows - 1) / kPieceRows;
        if (warp == 0) {
            // arm every piece's barrier before any copy can complete, then one copy per row
            if (lane < npieces) {
                const int rows = nr - lane * kPieceRows < kPieceRows ? nr - lane * kPieceRows : kPieceRows;
                const uint32_t bytes = (uint32_t)rows * (uint32_t)p.w_row_bytes;
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(
                                 smem_addr(smem + p.bar_off + 8 * lane)), "r"(bytes)
                             : "memory");
            }
            __syncwarp();
            for (int r = lane; r < nr; r += 32)
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                        wbuf + (uint32_t)(r * p.wstride)),
                    "l"(p.Wp + (n0 + r) * p.w_row_bytes), "r"((uint32_t)p.w_row_bytes),
                    "r"(smem_addr(smem + p.bar_off + 8 * (r / kPieceRows)))
                    : "memory");
        }
        for (int i = threadIdx.x; i < 2 * MT * round_rows; i += blockDim.x) acc_s[i] = 0u;
        for (int i = threadIdx.x; i < 2 * nr; i += blockDim.x) sw_s[i] = __ldg(p.s_w + n0 * 2 + i);
        if (round == 0) {
            // activation codes as bytes, chunk-padded, zero beyond PA up to the weights' PW
#pragma unroll
            for (int g = 0; g < 2; ++g) {
                const GroupGeom& G = p.g[g];
                const int nblk_a = G.pa / 32, nblk_w = G.pw / 32;
                uint8_t* a_s = smem + p.a_s_off[g];
                for (int item = threadIdx.x; item < p.M * nblk_w; item += blockDim.x) {
                    const int m = item / nblk_w, kb = item - m * nblk_w;
                    uint32_t o[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                    if (kb < nblk_a) {
                        const uint32_t* src = reinterpret_cast<const uint32_t*>(
                            p.Ap + (int64_t)m * p.a_row_bytes + G.a_off + kb * 4 * G.bits_a);
                        uint32_t w[8];
                        for (int i = 0; i < G.bits_a; ++i) w[i] = __ldg(src + i);
                        block_to_bytes_n(G.bits_a, w, o);
                        uint32_t sum = 0;
#pragma unroll
                        for (int t = 0; t < 8; ++t) sum = __dp4a(o[t], 0x01010101u, sum);
                        atomicAdd(&rowsum[g * 16 + m], (int32_t)sum);
                    }
                    uint4* d = reinterpret_cast<uint4*>(a_s + m * p.a_m_stride[g] + (kb >> 2) * A_CHUNK + (kb & 3) * 32);
                    d[0] = make_uint4(o[0], o[1], o[2], o[3]);
                    d[1] = make_uint4(o[4], o[5], o[6], o[7]);
                }
            }
        }
        __syncthreads();

        // tasks in piece order; a half-warp waits for a piece's barrier before its first task there
        const int half = threadIdx.x >> 4, nhalf = blockDim.x >> 4, r = threadIdx.x & 15;
        const int dpiece = nhalf / tpp, dj = nhalf - dpiece * tpp;   // task t -> (piece, j), stepped by nhalf
        int waited = -1;
        int piece = half / tpp, j = half - (half / tpp) * tpp;
        for (; piece < npieces && ok; piece += dpiece, j += dj) {
            if (j >= tpp) {
                j -= tpp;
                ++piece;
                if (piece >= npieces) break;
            }
            if (piece != waited) {
                ok = gemv_wait(smem_addr(smem + p.bar_off + 8 * piece), (uint32_t)(round & 1), p);
                waited = piece;
                if (!ok) break;
            }
            const int g = j < nch0 ? 0 : 1, c = g ? j - nch0 : j;
            const int row = piece * kPieceRows + r;
            if (row >= nr) continue;
            const GroupGeom& G = p.g[g];
            uint32_t acc[MT];
#pragma unroll
            for (int m = 0; m < MT; ++m) acc[m] = 0u;
            bulk_task<MT>(p, g, G.bits_w, wbuf + (uint32_t)(row * p.wstride + G.w_off + c * 16 * G.bits_w),
                          smem_addr(smem) + (uint32_t)(p.a_s_off[g] + c * A_CHUNK), acc);
#pragma unroll
            for (int m = 0; m < MT; ++m)
                if (m < p.M && acc[m] != 0u) atomicAdd(&acc_s[(g * MT + m) * round_rows + row], acc[m]);
        }
        if (__syncthreads_or(!ok)) break;

        // epilogue: one thread per (row, m)
        for (int t = threadIdx.x; t < nr * p.M; t += blockDim.x) {
            const int rr = t / p.M, m = t - rr * p.M;
            const int64_t n = n0 + rr;
            float y = 0.0f;
#pragma unroll
            for (int g = 0; g < 2; ++g) {
                const GroupGeom& G = p.g[g];
                if (G.pa == 0) continue;
                const uint32_t v = acc_s[(g * MT + m) * round_rows + rr];
                const int32_t off = 1 << (G.bits_w - 1);
                const int32_t a = (int32_t)(v - (uint32_t)(off * rowsum[g * 16 + m]));
                const float inv = 1.0f / ((float)((1 << G.bits_a) - 1) * (float)off);
                const float sw = sw_s[rr * 2 + g] * inv;
                const float sa = p.s_a_per_row ? __ldg(p.s_a + m * 2 + g) : __ldg(p.s_a + g);
                y = g == 0 ? (sa * sw) * (float)a : fmaf(sa * sw, (float)a, y);
                if (p.acc_dbg != nullptr) p.acc_dbg[((int64_t)g * p.M + m) * p.N + n] = a;
            }
            const int64_t idx = (int64_t)m * p.N + n;
            if (p.out_bf16) reinterpret_cast<__nv_bfloat16*>(p.Y)[idx] = __float2bfloat16_rn(y);
            else reinterpret_cast<__half*>(p.Y)[idx] = __float2half_rn(y);
        }
        __syncthreads();   // the buffer and the per-row totals are free for the next round
    }
    // copies of an abandoned round must land before the CTA exits
    if (!ok && threadIdx.x == 0) {
        const int64_t n0 = n_begin + (int64_t)round * round_rows;
        const int nr = (int)(n_end - n0 < round_rows ? n_end - n0 : round_rows);
        for (int k = 0; k < (nr + kPieceRows - 1) / kPieceRows; ++k)
            gemv_wait(smem_addr(smem + p.bar_off + 8 * k), (uint32_t)(round & 1), p);
    }
}

// Shared memory of the bulk kernel: row sums, per-row totals of a round,
// barriers, the activation bytes of both groups over the weights' chunks, and
// the round's weight rows.  Rows per CTA: N over the SMs; rows per round: as
// many as fit (at most kMaxPieces pieces).
size_t gemv_bulk_smem(const LayoutGeom& geo, int64_t M, int64_t N, GemvParams* p) {
    const int64_t mt = M <= 1 ? 1 : (M <= 2 ? 2 : (M <= 4 ? 4 : (M <= 8 ? 8 : 16)));   // per-row totals per activation row
    int64_t ws = geo.w_row_bytes;
    if ((ws / 16) % 2 == 0) ws += 16;
    p->wstride = (int32_t)ws;
    const int64_t nsm = num_sms() > 0 ? num_sms() : 1;
    int64_t grid = (N + kPieceRows - 1) / kPieceRows;
    if (grid > nsm) grid = nsm;
    const int64_t rows_cta = (N + grid - 1) / grid;
    size_t o = 128;
    size_t a_bytes = 0;
    for (int g = 0; g < 2; ++g) a_bytes += (size_t)M * (geo.g[g].pw / 128) * A_CHUNK;
    const size_t budget = 222 * 1024;
    // fixed: row sums, barriers, activations, alignment slack; per round row:
    // its per-row totals, its two weight scales and its weight bytes
    const size_t fixed = 128 + 8 * kMaxPieces + a_bytes + 4 * 16 + 128;
    const size_t per_row = (size_t)2 * mt * 4 + 2 * 4 + (size_t)ws;
    int64_t round = rows_cta < kPieceRows * kMaxPieces ? rows_cta : kPieceRows * kMaxPieces;
    while (round > 1 && fixed + (size_t)round * per_row > budget) --round;
    p->rows_cta = (int32_t)rows_cta;
    p->round_rows = (int32_t)round;
    p->sum_off = (int32_t)o;
    o += (size_t)2 * mt * round * 4;
    o = (o + 15) & ~(size_t)15;
    p->scale_off = (int32_t)o;
    o += (size_t)2 * round * 4;
    o = (o + 15) & ~(size_t)15;
    p->bar_off = (int32_t)o;
    o += 8 * kMaxPieces;
    o = (o + 15) & ~(size_t)15;
    for (int g = 0; g < 2; ++g) {
        const int64_t chunks = geo.g[g].pw / 128;
        p->a_s_off[g] = (int32_t)o;
        p->a_m_stride[g] = (int32_t)(chunks * A_CHUNK);
        o += (size_t)M * chunks * A_CHUNK;
        o = (o + 15) & ~(size_t)15;
    }
    o = (o + 127) & ~(size_t)127;
    p->buf_off = (int32_t)o;
    return o + (size_t)round * ws;
}

template <int MT>
cudaError_t run_bulk(const GemvParams& p, size_t smem, cudaStream_t st) {
    cudaError_t e = cudaFuncSetAttribute(gemv_bulk_kernel<MT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = prefer_max_shared((const void*)gemv_bulk_kernel<MT>);
    if (e != cudaSuccess) return e;
    const int64_t grid = (p.N + p.rows_cta - 1) / p.rows_cta;
    gemv_bulk_kernel<MT><<<(unsigned)grid, bulk_threads<MT>(), smem, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

}  // namespace

bool gemv_supported(const LayoutGeom& geo, int64_t M, int64_t N) {
    GemvParams p;
    if (M < 1 || M > kBulkMaxM || N < 1 || geo.w_row_bytes % 16 != 0) return false;
    return gemv_bulk_smem(geo, M, N, &p) <= 224 * 1024;
}

cudaError_t launch_gemv(const LayoutGeom& geo, const GemvArgs& a, cudaStream_t st) {
    GemvParams p;
    p.Ap = a.Ap;
    p.Wp = a.Wp;
    p.s_a = a.s_a;
    p.s_w = a.s_w;
    p.Y = a.Y;
    p.acc_dbg = a.acc_dbg;
    p.M = a.M;
    p.N = a.N;
    p.a_row_bytes = geo.a_row_bytes;
    p.w_row_bytes = geo.w_row_bytes;
    p.s_a_per_row = a.s_a_per_row;
    p.out_bf16 = a.out_bf16;
    p.g[0] = geo.g[0];
    p.g[1] = geo.g[1];
    if (!gemv_supported(geo, a.M, a.N)) return cudaErrorNotSupported;
    if (((uintptr_t)a.Wp & 15u) != 0) return cudaErrorNotSupported;
    p.err = device_error_word();
    if (p.err == nullptr) return cudaErrorUnknown;
    p.timeout_ns = 2000000000LL;
    const size_t smem = gemv_bulk_smem(geo, a.M, a.N, &p);
    if (a.M == 1) return run_bulk<1>(p, smem, st);
    if (a.M == 2) return run_bulk<2>(p, smem, st);
    if (a.M <= 4) return run_bulk<4>(p, smem, st);
    if (a.M <= 8) return run_bulk<8>(p, smem, st);
    return run_bulk<16>(p, smem, st);
}

}  // namespace soniq
