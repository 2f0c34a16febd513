// Quantize and pack for the layout variants (linear layers):
//   * signed activations: Eq. (1) applied to the activation, codes in
//     [-2^(n-1), 2^(n-1) - 1] stored as n-bit two's complement (the
//     transformer-layer reading of Sec. 3);
//   * one-bit +-1 groups (Sec. 4.2, XNOR and POPCOUNT for one-bit channels):
//     code +1 for x >= 0 and -1 otherwise on both sides, stored as the bit
//     (code + 1) / 2;
//   * scale runs along K: a group's packed positions are cut into runs of
//     sub_k, each with its own max-abs scale (the fine scale groups of the
//     evaluation setup); scale arrays are [rows or 1][2][nb].
// The default path's kernels stay as they are; these kernels favour plain,
// checkable indexing over speed.
#include <cuda_fp16.h>
#include <stdint.h>

#include "soniq_device.cuh"
#include "soniq_internal.h"

namespace soniq {
namespace {

constexpr int kAbsmaxThreads = 256;
constexpr int kMaxRuns = 512;   // 65536 / 128

template <typename T>
__device__ __forceinline__ float load_x(const T* X, int64_t i);
template <>
__device__ __forceinline__ float load_x<uint16_t>(const uint16_t* X, int64_t i) {
    return __half2float(__ushort_as_half(X[i]));
}
template <>
__device__ __forceinline__ float load_x<float>(const float* X, int64_t i) {
    return X[i];
}

struct VGeo {
    int32_t K, count0, count1, sub_k, nb;
    int32_t bits[2];
    int32_t kind[2];        // 0 unsigned, 1 signed (Eq. (1)), 2 +-1
    int32_t off[2];         // byte offset of group g in a packed row
    int32_t blocks[2];      // 32-code blocks of group g in a packed row
    int32_t row_bytes;
};

__device__ __forceinline__ int run_of(int j, int sub_k) { return sub_k > 0 ? j / sub_k : 0; }

// Max |x| per (group, run) of each row (per_row) or of all rows; s must be
// zero before a per-tensor launch (maxima are merged with atomicMax on the
// bit patterns, which order non-negative floats and infinity; NaN, whose
// patterns lie above infinity's, is skipped as the other max-abs passes skip it).
template <typename T>
__global__ void __launch_bounds__(kAbsmaxThreads) variant_absmax_kernel(const T* X, int64_t rows, const int32_t* perm,
                                                                        VGeo v, int per_row, float* s) {
    __shared__ unsigned smax[2 * kMaxRuns];
    const int nkeys = 2 * v.nb;
    for (int i = threadIdx.x; i < nkeys; i += blockDim.x) smax[i] = 0u;
    __syncthreads();
    for (int64_t m = blockIdx.x; m < rows; m += gridDim.x) {
        for (int p = threadIdx.x; p < v.K; p += blockDim.x) {
            const int g = p < v.count0 ? 0 : 1;
            const int j = g == 0 ? p : p - v.count0;
            const float a = fabsf(load_x<T>(X, m * v.K + perm[p]));
            if (a == a) atomicMax(&smax[g * v.nb + run_of(j, v.sub_k)], __float_as_uint(a));
        }
        if (per_row) {
            __syncthreads();
            for (int i = threadIdx.x; i < nkeys; i += blockDim.x) {
                s[m * nkeys + i] = __uint_as_float(smax[i]);
                smax[i] = 0u;
            }
            __syncthreads();
        }
    }
    if (!per_row) {
        __syncthreads();
        for (int i = threadIdx.x; i < nkeys; i += blockDim.x)
            if (smax[i] != 0u) atomicMax(reinterpret_cast<unsigned*>(s) + i, smax[i]);
    }
}

// One warp per (row, group, 32-code block): lane i takes code i of the block.
template <typename T>
__global__ void __launch_bounds__(256) variant_codes_kernel(const T* X, int64_t rows, const int32_t* perm, VGeo v,
                                                            const float* s, int per_row, int is_weight,
                                                            uint8_t* out) {
    const int lane = threadIdx.x & 31;
    const int64_t nblk = (int64_t)v.blocks[0] + v.blocks[1];
    const int64_t items = rows * nblk;
    const int64_t warp0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t it = warp0; it < items; it += nwarps) {
        const int64_t m = it / nblk;
        int blk = (int)(it - m * nblk);
        const int g = blk < v.blocks[0] ? 0 : 1;
        if (g == 1) blk -= v.blocks[0];
        const int n = v.bits[g];
        const int count = g == 0 ? v.count0 : v.count1;
        const int base = g == 0 ? 0 : v.count0;
        const int j = blk * 32 + lane;
        uint32_t pattern = 0u;
        if (j < count) {
            const float x = load_x<T>(X, m * v.K + perm[base + j]);
            const float sc = s[((per_row ? m : 0) * 2 + g) * v.nb + run_of(j, v.sub_k)];
            if (v.kind[g] == 2) {
                pattern = x >= 0.0f ? 1u : 0u;
            } else if (v.kind[g] == 1 || is_weight) {
                pattern = (uint32_t)weight_code(x, sc, (float)(1 << (n - 1))) & ((1u << n) - 1u);
            } else {
                pattern = act_code(x, sc, (float)((1 << n) - 1));
            }
        }
        const uint32_t word = pack_block_warp(pattern, n);
        if (lane < n)
            reinterpret_cast<uint32_t*>(out + m * v.row_bytes + v.off[g] + (int64_t)blk * 4 * n)[lane] = word;
    }
}

VGeo make_vgeo(const LayoutGeom& geo, bool weight) {
    VGeo v{};
    v.K = geo.K;
    v.count0 = geo.g[0].count;
    v.count1 = geo.g[1].count;
    v.sub_k = geo.sub_k;
    v.nb = geo.nb;
    for (int g = 0; g < 2; ++g) {
        const GroupGeom& G = geo.g[g];
        v.bits[g] = weight ? G.bits_w : G.bits_a;
        v.kind[g] = weight ? (geo.act_kind[g] == 2 ? 2 : 1) : geo.act_kind[g];
        v.off[g] = weight ? G.w_off : G.a_off;
        v.blocks[g] = (weight ? G.pw : G.pa) / 32;
    }
    v.row_bytes = weight ? geo.w_row_bytes : geo.a_row_bytes;
    return v;
}

template <typename T>
cudaError_t run_variant(const LayoutGeom& geo, const int32_t* perm, const T* X, int64_t rows, bool weight,
                        int32_t scale_mode, float* s, uint8_t* out, cudaStream_t st) {
    const VGeo v = make_vgeo(geo, weight);
    const int per_row = scale_mode == SONIQ_SCALE_PER_ROW;
    cudaError_t e = cudaSuccess;
    if (scale_mode != SONIQ_SCALE_CALIBRATED) {
        if (!per_row && (e = cudaMemsetAsync(s, 0, sizeof(float) * 2 * v.nb, st)) != cudaSuccess) return e;
        const int64_t cap = (int64_t)num_sms() * 8;
        const int grid = (int)(rows < cap ? rows : cap);
        variant_absmax_kernel<T><<<grid, kAbsmaxThreads, 0, st>>>(X, rows, perm, v, per_row, s);
        note_launch();
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    const int64_t items = rows * ((int64_t)v.blocks[0] + v.blocks[1]);
    const int64_t ctas = (items + 7) / 8;
    const int64_t cap = (int64_t)num_sms() * 16;
    variant_codes_kernel<T><<<(int)(ctas < cap ? ctas : cap), 256, 0, st>>>(X, rows, perm, v, s, per_row,
                                                                           weight ? 1 : 0, out);
    note_launch();
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_variant_quantize_act(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A, int64_t M,
                                        int32_t scale_mode, float* s_a, uint8_t* Ap, cudaStream_t st) {
    return run_variant<uint16_t>(geo, perm, A, M, false, scale_mode, s_a, Ap, st);
}

cudaError_t launch_variant_pack_weights(const LayoutGeom& geo, const int32_t* perm, const float* W, int32_t N,
                                        float* s_w, uint8_t* Wp, cudaStream_t st) {
    return run_variant<float>(geo, perm, W, N, true, SONIQ_SCALE_PER_ROW, s_w, Wp, st);
}

}  // namespace soniq
