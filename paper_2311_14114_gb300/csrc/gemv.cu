// Small-M mixed-precision GEMV (M <= 16): the decode-shaped case where the
// packed weight bytes streamed from HBM are the roofline (Sec. 2.4 C5: one
// coalesced load per packed word).
//
// Exact integer arithmetic on CUDA cores (Sec. 4.2: unsigned x signed
// integer dot products):
//   * the activation codes (M rows) are expanded once per CTA into shared
//     memory as bytes, together with their per-group row sums R_g[m];
//   * each warp streams RT weight rows; every lane expands packed 32-code
//     blocks to bytes, flips the sign bit (j -> j + 2^(n-1), unsigned), and
//     accumulates dp4a(u, j + 2^(n-1)) in uint32;
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
    int32_t a_s_off[2];   // byte offset of group g's [M][pa] byte matrix in shared memory
};

constexpr int kThreads = 256;

template <int NB>
__device__ __forceinline__ void load_words(const uint8_t* p, uint32_t* w) {
    const uint32_t* q = reinterpret_cast<const uint32_t*>(p);
#pragma unroll
    for (int i = 0; i < NB; ++i) w[i] = __ldg(q + i);
}

// Accumulates one weight block (NW-bit codes) of RT rows against MT rows of
// activation bytes.
template <int NW, int MT, int RT>
__device__ __forceinline__ void gemv_block(const GemvParams& p, const uint8_t* const* wrow,
                                           const bool* rv, int g, int kb, const uint8_t* a_s,
                                           uint32_t (&acc)[RT][MT]) {
    uint32_t wb[RT][8];
#pragma unroll
    for (int r = 0; r < RT; ++r) {
        uint32_t w[NW];
        if (rv[r]) {
            load_words<NW>(wrow[r] + p.g[g].w_off + kb * 4 * NW, w);
        } else {
#pragma unroll
            for (int i = 0; i < NW; ++i) w[i] = 0u;
        }
        block_to_bytes<NW>(w, wb[r]);
        const uint32_t flip = sign_flip_mask(NW);
#pragma unroll
        for (int t = 0; t < 8; ++t) wb[r][t] ^= flip;
    }
    const int pa = p.g[g].pa;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
        if (m < p.M) {
            const uint4* a4 = reinterpret_cast<const uint4*>(a_s + m * pa + kb * 32);
            const uint4 x0 = a4[0], x1 = a4[1];
            const uint32_t a[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int r = 0; r < RT; ++r)
#pragma unroll
                for (int t = 0; t < 8; ++t) acc[r][m] = __dp4a(wb[r][t], a[t], acc[r][m]);
        }
    }
}

template <int MT, int RT>
__global__ void __launch_bounds__(kThreads) gemv_kernel(const GemvParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    int32_t* rowsum = reinterpret_cast<int32_t*>(smem);   // [2][16]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

    // ---- expand the activation codes of all M rows into shared memory ----
    if (threadIdx.x < 32) rowsum[threadIdx.x] = 0;
    __syncthreads();
#pragma unroll
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = p.g[g];
        const int nblk = G.pa / 32;
        uint8_t* a_s = smem + p.a_s_off[g];
        for (int item = threadIdx.x; item < p.M * nblk; item += blockDim.x) {
            const int m = item / nblk, kb = item - m * nblk;
            const uint32_t* src = reinterpret_cast<const uint32_t*>(
                p.Ap + (int64_t)m * p.a_row_bytes + G.a_off + kb * 4 * G.bits_a);
            uint32_t w[8], o[8];
            for (int i = 0; i < G.bits_a; ++i) w[i] = __ldg(src + i);
            block_to_bytes_n(G.bits_a, w, o);
            uint32_t s = 0;
#pragma unroll
            for (int t = 0; t < 8; ++t) s = __dp4a(o[t], 0x01010101u, s);
            uint4* d = reinterpret_cast<uint4*>(a_s + m * G.pa + kb * 32);
            d[0] = make_uint4(o[0], o[1], o[2], o[3]);
            d[1] = make_uint4(o[4], o[5], o[6], o[7]);
            atomicAdd(&rowsum[g * 16 + m], (int32_t)s);
        }
    }
    __syncthreads();

    // ---- stream weight rows ----
    const int total_warps = gridDim.x * (blockDim.x >> 5);
    for (int n0 = (blockIdx.x * (blockDim.x >> 5) + warp) * RT; n0 < p.N; n0 += total_warps * RT) {
        float y[RT][MT];
#pragma unroll
        for (int r = 0; r < RT; ++r)
#pragma unroll
            for (int m = 0; m < MT; ++m) y[r][m] = 0.0f;
        const uint8_t* wrow[RT];
        bool rv[RT];
#pragma unroll
        for (int r = 0; r < RT; ++r) {
            rv[r] = n0 + r < p.N;
            wrow[r] = p.Wp + (int64_t)(rv[r] ? n0 + r : 0) * p.w_row_bytes;
        }
#pragma unroll
        for (int g = 0; g < 2; ++g) {
            const GroupGeom& G = p.g[g];
            if (G.pa == 0) continue;
            uint32_t acc[RT][MT];
#pragma unroll
            for (int r = 0; r < RT; ++r)
#pragma unroll
                for (int m = 0; m < MT; ++m) acc[r][m] = 0u;
            const uint8_t* a_s = smem + p.a_s_off[g];
            const int nblk = G.pa / 32;   // blocks beyond pa hold no activation codes
            for (int kb = lane; kb < nblk; kb += 32) {
                switch (G.bits_w) {
                    case 1: gemv_block<1, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    case 2: gemv_block<2, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    case 3: gemv_block<3, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    case 4: gemv_block<4, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    case 5: gemv_block<5, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    case 6: gemv_block<6, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    case 7: gemv_block<7, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                    default: gemv_block<8, MT, RT>(p, wrow, rv, g, kb, a_s, acc); break;
                }
            }
            // warp butterfly: every lane ends with the full sums
#pragma unroll
            for (int r = 0; r < RT; ++r)
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    uint32_t v = acc[r][m];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                    acc[r][m] = v;
                }
            const int32_t off = 1 << (G.bits_w - 1);
            const float inv = 1.0f / ((float)((1 << G.bits_a) - 1) * (float)off);
#pragma unroll
            for (int r = 0; r < RT; ++r) {
                if (!rv[r]) continue;
                const int n = n0 + r;
                const float sw = __ldg(p.s_w + (int64_t)n * 2 + g) * inv;
#pragma unroll
                for (int m = 0; m < MT; ++m) {
                    if (m < p.M) {
                        const int32_t a = (int32_t)(acc[r][m] - (uint32_t)(off * rowsum[g * 16 + m]));
                        const float sa = p.s_a_per_row ? __ldg(p.s_a + m * 2 + g) : __ldg(p.s_a + g);
                        y[r][m] = fmaf(sa * sw, (float)a, y[r][m]);
                        if (p.acc_dbg != nullptr && lane == ((r * MT + m) & 31))
                            p.acc_dbg[((int64_t)g * p.M + m) * p.N + n] = a;
                    }
                }
            }
        }
#pragma unroll
        for (int r = 0; r < RT; ++r) {
            if (!rv[r]) continue;
#pragma unroll
            for (int m = 0; m < MT; ++m) {
                if (m < p.M && lane == ((r * MT + m) & 31)) {
                    const int64_t idx = (int64_t)m * p.N + n0 + r;
                    if (p.out_bf16) reinterpret_cast<__nv_bfloat16*>(p.Y)[idx] = __float2bfloat16_rn(y[r][m]);
                    else reinterpret_cast<__half*>(p.Y)[idx] = __float2half_rn(y[r][m]);
                }
            }
        }
    }
}

size_t gemv_smem(const LayoutGeom& geo, int64_t M, int32_t* off) {
    size_t o = 128;   // row sums [2][16]
    for (int g = 0; g < 2; ++g) {
        off[g] = (int32_t)o;
        o += (size_t)M * geo.g[g].pa;
        o = (o + 15) & ~(size_t)15;
    }
    return o;
}

template <int MT, int RT>
cudaError_t run(const GemvParams& p, size_t smem, cudaStream_t st) {
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(gemv_kernel<MT, RT>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    int per_sm = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gemv_kernel<MT, RT>,
                                                                   kThreads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorNotSupported;
    const int rows_per_cta = (kThreads / 32) * RT;
    int grid = (p.N + rows_per_cta - 1) / rows_per_cta;
    const int cap = num_sms() * per_sm;
    if (grid > cap) grid = cap;
    gemv_kernel<MT, RT><<<grid, kThreads, smem, st>>>(p);
    note_launch();
    return cudaGetLastError();
}

}  // namespace

bool gemv_supported(const LayoutGeom& geo, int64_t M) {
    int32_t off[2];
    return M >= 1 && M <= 16 && gemv_smem(geo, M, off) <= 200 * 1024;
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
    if (!gemv_supported(geo, a.M)) return cudaErrorNotSupported;
    const size_t smem = gemv_smem(geo, a.M, p.a_s_off);
    if (a.M == 1) return run<1, 4>(p, smem, st);
    if (a.M <= 2) return run<2, 4>(p, smem, st);
    if (a.M <= 4) return run<4, 4>(p, smem, st);
    if (a.M <= 8) return run<8, 2>(p, smem, st);
    return run<16, 2>(p, smem, st);
}

}  // namespace soniq
