// Quantize-and-pack kernels: Sec. 3 "Enabling Low-Cost Fixed-Point
// Operations" steps 1-3 with the channel permutation and padding of Sec. 4.1.
//
//   act_absmax_kernel     per-(tensor, group) max |a|            (step 1)
//   quantize_act_kernel   gather by perm, unsigned codes, pack    (steps 1-2)
//   weight_absmax_kernel  per-(tensor, group) max |w|             (step 1)
//   pack_weights_kernel   per-(row, group) scale, Eq. (1) codes, pack (steps 1, 3)
//
// All are HBM-streaming kernels: rows are read with 16-byte loads where the
// alignment allows, the permutation gather happens in shared memory, and one
// warp packs each 32-code block with warp-wide OR reductions.
#include <cuda_fp16.h>

#include "soniq_device.cuh"
#include "soniq_internal.h"

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
// Activation quantize-and-pack.  One warp per row: the fp16 row is staged in
// shared memory with 16-byte loads, then each 32-code block is gathered
// through perm, quantized (Sec. 3 step 2) and packed by the warp.
// ---------------------------------------------------------------------------
struct QuantActParams {
    const uint16_t* A;
    uint8_t* Ap;
    float* s_a;
    const int32_t* perm;
    int64_t M;
    int32_t K;
    int32_t a_row_bytes;
    int32_t scale_mode;
    int32_t vec_ok;
    int32_t warps;           // rows staged per CTA
    GroupGeom g[2];
};

__global__ void __launch_bounds__(kThreads) quantize_act_kernel(const QuantActParams p) {
    extern __shared__ __align__(16) uint8_t smem[];
    uint16_t* perm_s = reinterpret_cast<uint16_t*>(smem);                 // K entries
    const int perm_bytes = (p.K * 2 + 15) & ~15;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __half* row_s = reinterpret_cast<__half*>(smem + perm_bytes) + (int64_t)warp * p.K;

    for (int j = threadIdx.x; j < p.K; j += blockDim.x) perm_s[j] = (uint16_t)p.perm[j];
    __syncthreads();

    float tensor_s[2] = {0.0f, 0.0f};
    if (p.scale_mode != SONIQ_SCALE_PER_ROW) { tensor_s[0] = p.s_a[0]; tensor_s[1] = p.s_a[1]; }

    for (int64_t m = (int64_t)blockIdx.x * p.warps + warp; m < p.M; m += (int64_t)gridDim.x * p.warps) {
        const uint16_t* src = p.A + m * p.K;
        if (p.vec_ok) {
            const uint4* s4 = reinterpret_cast<const uint4*>(src);
            uint4* d4 = reinterpret_cast<uint4*>(row_s);
            for (int v = lane; v < p.K / 8; v += 32) d4[v] = __ldg(s4 + v);
        } else {
            for (int c = lane; c < p.K; c += 32)
                row_s[c] = *reinterpret_cast<const __half*>(src + c);
        }
        __syncwarp();

        float s[2] = {tensor_s[0], tensor_s[1]};
        if (p.scale_mode == SONIQ_SCALE_PER_ROW) {
#pragma unroll
            for (int g = 0; g < 2; ++g) {
                float mx = 0.0f;
                for (int j = lane; j < p.g[g].count; j += 32)
                    mx = fmaxf(mx, fabsf(__half2float(row_s[perm_s[p.g[g].perm_base + j]])));
                s[g] = warp_max(mx);
            }
            if (lane < 2) p.s_a[m * 2 + lane] = s[lane];
        }

        uint8_t* dst_row = p.Ap + m * (int64_t)p.a_row_bytes;
#pragma unroll
        for (int g = 0; g < 2; ++g) {
            const GroupGeom& G = p.g[g];
            const int n = G.bits_a;
            const float levels = (float)((1 << n) - 1);
            const int nblk = G.pa / 32;
            uint32_t* dst = reinterpret_cast<uint32_t*>(dst_row + G.a_off);
            for (int kb = 0; kb < nblk; ++kb) {
                const int c = kb * 32 + lane;
                uint32_t u = 0u;
                if (c < G.count) u = act_code(__half2float(row_s[perm_s[G.perm_base + c]]), s[g], levels);
                const uint32_t word = pack_block_warp(u, n);
                if (lane < n) dst[kb * n + lane] = word;
            }
        }
        __syncwarp();
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
        uint32_t* dst = reinterpret_cast<uint32_t*>(dst_row + G.w_off);
        for (int kb = warp; kb < G.pw / 32; kb += nwarps) {
            const int pos = kb * 32 + lane;
            const int t = pos / G.pa, c = pos - t * G.pa;
            int32_t j = 0;
            if (t < p.taps && c < G.count)
                j = weight_code(__ldg(Wn + (int64_t)t * p.K + p.perm[G.perm_base + c]), s, half);
            const uint32_t word = pack_block_warp((uint32_t)j & mask, nb);
            if (lane < nb) dst[kb * nb + lane] = word;
        }
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
                              int64_t M, float* s_out, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(s_out, 0, 2 * sizeof(float), st);
    if (e != cudaSuccess) return e;
    const int vec_ok = (geo.K % 8 == 0) && ((uintptr_t)A % 16 == 0);
    const int grid = grid_for(M * (int64_t)geo.K / 8, kThreads * 4);
    absmax_kernel<__half><<<grid, kThreads, geo.K, st>>>(reinterpret_cast<const __half*>(A), M,
                                                         geo.K, perm, geo.g[0].count,
                                                         reinterpret_cast<unsigned*>(s_out), vec_ok);
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_quantize_act(const LayoutGeom& geo, const int32_t* perm, const uint16_t* A,
                                int64_t M, int32_t scale_mode, float* s_a, uint8_t* Ap,
                                cudaStream_t st) {
    QuantActParams p;
    p.A = A;
    p.Ap = Ap;
    p.s_a = s_a;
    p.perm = perm;
    p.M = M;
    p.K = geo.K;
    p.a_row_bytes = geo.a_row_bytes;
    p.scale_mode = scale_mode;
    p.vec_ok = (geo.K % 8 == 0) && ((uintptr_t)A % 16 == 0);
    p.g[0] = geo.g[0];
    p.g[1] = geo.g[1];
    const int perm_bytes = (geo.K * 2 + 15) & ~15;
    // rows staged per CTA: as many warps as fit in 96 KB of shared memory
    int warps = (96 * 1024 - perm_bytes) / (geo.K * 2);
    if (warps > kThreads / 32) warps = kThreads / 32;
    if (warps < 1) warps = 1;
    p.warps = warps;
    const size_t smem = (size_t)perm_bytes + (size_t)warps * geo.K * 2;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(quantize_act_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    const int grid = grid_for(M, warps * 4);
    quantize_act_kernel<<<grid, warps * 32, smem, st>>>(p);
    note_launch();
    return cudaGetLastError();
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
