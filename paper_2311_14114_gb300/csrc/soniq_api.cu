// C-ABI entry points of the SONIQ library: argument validation (host only,
// before any CUDA call), layout geometry, dispatch to the kernels and the
// device-side error word that bounded waits report into.
#include <atomic>
#include <cstring>
#include <vector>

#include <mutex>
#include <set>
#include <utility>

#include "soniq_internal.h"

namespace soniq {

namespace {

// One word per device: kernels atomically OR error bits into it when a
// bounded wait runs out (kErrWait, kErrQuantBarrier, kErrOneshotBarrier);
// soniq_sync_status reads and clears it.
__device__ unsigned g_error_word;

// Working memory of soniq_quantize_act_oneshot, the entry point that takes no
// scratch from its caller: a grid barrier (arrival count, generation; zero
// when the module loads and left at zero by every completed call) and the
// per-CTA maxima of at most kOneShotMaxCtas CTAs (8 KB in all).  Host code
// reaches it only through the address cudaGetSymbolAddress returns.
constexpr int kOneShotMaxCtas = 1024;
static __device__ __align__(256) unsigned g_oneshot_barrier[2];
static __device__ __align__(256) float g_oneshot_partials[2 * kOneShotMaxCtas];

// Test hook (soniq_test_drop_barrier_arrival): the next one-pass quantize
// launch drops one grid-barrier arrival.
std::atomic<int> g_drop_arrival{0};

std::atomic<int64_t> g_launches{0};

constexpr int kMaxDevices = 64;
unsigned* g_err_addr[kMaxDevices] = {};
int g_sms[kMaxDevices] = {};

int64_t roundup(int64_t x, int64_t u) { return (x + u - 1) / u * u; }

bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

int current_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
    return dev;
}

soniq_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return SONIQ_OK;
    if (e == cudaErrorNotSupported) return SONIQ_ERR_UNSUPPORTED;
    return SONIQ_ERR_CUDA;
}

}  // namespace

unsigned* device_error_word() {
    const int dev = current_device();
    if (dev < 0) return nullptr;
    if (g_err_addr[dev] == nullptr) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
        g_err_addr[dev] = static_cast<unsigned*>(p);
    }
    return g_err_addr[dev];
}

// Device addresses of the one-shot scratch, resolved once per device at first
// use; false if the runtime cannot resolve them.
bool oneshot_scratch(unsigned** bar, float** part) {
    static std::mutex mu;
    static unsigned* bars[64] = {};
    static float* parts[64] = {};
    const int dev = current_device();
    if (dev < 0 || dev >= 64) return false;
    std::lock_guard<std::mutex> lock(mu);
    if (bars[dev] == nullptr) {
        void* b = nullptr;
        void* q = nullptr;
        if (cudaGetSymbolAddress(&b, g_oneshot_barrier) != cudaSuccess) return false;
        if (cudaGetSymbolAddress(&q, g_oneshot_partials) != cudaSuccess) return false;
        bars[dev] = static_cast<unsigned*>(b);
        parts[dev] = static_cast<float*>(q);
    }
    *bar = bars[dev];
    *part = parts[dev];
    return true;
}

bool take_drop_arrival() { return g_drop_arrival.exchange(0) != 0; }

void note_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

cudaError_t prefer_max_shared(const void* func) {
    static std::mutex mu;
    static std::set<std::pair<int, const void*>> done;
    const int dev = current_device();
    std::lock_guard<std::mutex> lock(mu);
    if (done.count({dev, func})) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(func, cudaFuncAttributePreferredSharedMemoryCarveout,
                                         (int)cudaSharedmemCarveoutMaxShared);
    if (e == cudaSuccess) done.insert({dev, func});
    return e;
}

int num_sms() {
    const int dev = current_device();
    if (dev < 0) return 148;
    if (g_sms[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        g_sms[dev] = v > 0 ? v : 148;
    }
    return g_sms[dev];
}

soniq_status make_geom(const soniq_layout* L, int32_t taps, LayoutGeom* geo) {
    if (L == nullptr || geo == nullptr) return SONIQ_ERR_INVALID_ARG;
    if (L->K < 1 || L->K > 65536) return L->K < 1 ? SONIQ_ERR_INVALID_ARG : SONIQ_ERR_UNSUPPORTED;
    if (L->n_groups != 1 && L->n_groups != 2) return SONIQ_ERR_INVALID_ARG;
    if (L->pad_unit != 32 && L->pad_unit != 128) return SONIQ_ERR_INVALID_ARG;
    if (taps < 1 || taps > 4096) return SONIQ_ERR_INVALID_ARG;
    if (L->count[0] < 0 || L->count[1] < 0 || (int64_t)L->count[0] + L->count[1] != L->K)
        return SONIQ_ERR_INVALID_ARG;
    if (L->n_groups == 1 && L->count[1] != 0) return SONIQ_ERR_INVALID_ARG;
    geo->K = L->K;
    geo->taps = taps;
    int64_t a_off = 0, w_off = 0;
    for (int g = 0; g < 2; ++g) {
        GroupGeom& G = geo->g[g];
        const bool used = g < L->n_groups;
        const int bw = used ? L->bits_w[g] : 1;
        const int ba = used ? L->bits_a[g] : 1;
        if (bw < 1 || bw > 8 || ba < 1 || ba > 8) return SONIQ_ERR_INVALID_ARG;
        G.count = used ? L->count[g] : 0;
        G.bits_a = ba;
        G.bits_w = bw;
        G.pa = (int32_t)roundup(G.count, L->pad_unit);
        G.pw = (int32_t)roundup((int64_t)taps * G.pa, 128);
        G.a_off = (int32_t)a_off;
        G.w_off = (int32_t)w_off;
        G.perm_base = g == 0 ? 0 : L->count[0];
        a_off += (int64_t)G.pa / 32 * 4 * ba;
        w_off += (int64_t)G.pw / 32 * 4 * bw;
    }
    if (a_off > (1 << 30) || w_off > (1 << 30)) return SONIQ_ERR_UNSUPPORTED;
    geo->a_row_bytes = (int32_t)a_off;
    geo->w_row_bytes = (int32_t)w_off;
    // variants
    geo->variant = 0;
    for (int g = 0; g < 2; ++g) {
        const int k = L->act_kind[g];
        if (k != SONIQ_ACT_UNSIGNED && k != SONIQ_ACT_SIGNED && k != SONIQ_ACT_PM1) return SONIQ_ERR_INVALID_ARG;
        if (k == SONIQ_ACT_PM1 && g < L->n_groups && (L->bits_a[g] != 1 || L->bits_w[g] != 1))
            return SONIQ_ERR_INVALID_ARG;
        geo->act_kind[g] = g < L->n_groups ? k : SONIQ_ACT_UNSIGNED;
        if (geo->act_kind[g] != SONIQ_ACT_UNSIGNED) geo->variant = 1;
    }
    if (L->sub_k < 0 || (L->sub_k > 0 && L->sub_k % 128 != 0)) return SONIQ_ERR_INVALID_ARG;
    geo->sub_k = L->sub_k;
    geo->nb = 1;
    if (L->sub_k > 0) {
        geo->variant = 1;
        const int32_t pmax = geo->g[0].pa > geo->g[1].pa ? geo->g[0].pa : geo->g[1].pa;
        geo->nb = (pmax + L->sub_k - 1) / L->sub_k;
        if (geo->nb < 1) geo->nb = 1;
    }
    // the variants are implemented for linear layers with 128-code groups
    if (geo->variant && (taps != 1 || L->pad_unit != 128)) return SONIQ_ERR_UNSUPPORTED;
    return SONIQ_OK;
}

}  // namespace soniq

using namespace soniq;

namespace {

cudaStream_t as_stream(soniq_stream_t s) { return reinterpret_cast<cudaStream_t>(s); }

// The staged path pays for its expansion passes and a persistent launch; below
// about 2^30 multiply-adds the fused kernel is faster (measured: a 64 x 512 x
// 512 layer 37 vs 17 us, decode M = 16 x 11008 x 4096 62 vs 41.5 us), unless
// the call needs an epilogue only the staged kernel has.
bool staged_worthwhile(const LayoutGeom& geo, int64_t M, int64_t N, uint32_t flags) {
    if (flags & SONIQ_FLAG_FORCE_STAGED) return true;
    return (double)M * (double)N * (double)geo.K * (double)geo.taps >= 1073741824.0;
}

// The kernel soniq_mp_gemm runs: a SONIQ_PATH_* value, -1 when the
// tensor-core kernel would be chosen but cannot take the layout (mma_check
// says why), -2 when the GEMV was forced but cannot take the shape.
int gemm_path(const LayoutGeom& geo, int64_t M, int32_t N, uint32_t flags, size_t scratch_bytes) {
    // the layout variants run on the staged path only
    if (geo.variant) {
        if (flags & (SONIQ_FLAG_FORCE_GEMV | SONIQ_FLAG_FORCE_FUSED | SONIQ_FLAG_FORCE_SKINNY)) return -2;
        const int64_t need = staged_scratch_bytes(geo, M, N);
        return need > 0 && (int64_t)scratch_bytes >= need ? SONIQ_PATH_TENSOR_STAGED : -2;
    }
    // up to SONIQ_GEMV_MAX_M rows the CUDA-core GEMV is faster; above, the tensor-core
    // kernels (whose time hardly grows with M below 128) overtake it
    const bool want_gemv =
        (flags & SONIQ_FLAG_FORCE_GEMV) ||
        (M <= SONIQ_GEMV_MAX_M && !(flags & (SONIQ_FLAG_FORCE_MMA | SONIQ_FLAG_FORCE_SKINNY)));
    if (want_gemv && gemv_supported(geo, M, N)) return SONIQ_PATH_GEMV;
    if (flags & SONIQ_FLAG_FORCE_GEMV) return -2;
    const bool pinned = (flags & (SONIQ_FLAG_FORCE_FUSED | SONIQ_FLAG_FORCE_STAGED)) != 0;
    if ((flags & SONIQ_FLAG_FORCE_SKINNY) || (!pinned && M <= SONIQ_SKINNY_MAX_M)) {
        if (skinny_supported(geo, M, N)) return SONIQ_PATH_TENSOR_SKINNY;
        if (flags & SONIQ_FLAG_FORCE_SKINNY) return -2;
    }
    if (!(flags & SONIQ_FLAG_FORCE_FUSED) && staged_worthwhile(geo, M, N, flags)) {
        const int64_t need = staged_scratch_bytes(geo, M, N);
        if (need > 0 && (int64_t)scratch_bytes >= need) return SONIQ_PATH_TENSOR_STAGED;
    }
    if (mma_check(geo) != SONIQ_OK) return -1;
    return SONIQ_PATH_TENSOR;
}

// Checks a quantize-in-epilogue descriptor against this call's output width N.
soniq_status check_next(const soniq_next_layer* next, int64_t N, int32_t out_dtype, LayoutGeom* geo_next) {
    if (next->layout == nullptr || next->s_a == nullptr || next->Ap == nullptr) return SONIQ_ERR_INVALID_ARG;
    soniq_status st = make_geom(next->layout, 1, geo_next);
    if (st != SONIQ_OK) return st;
    if (out_dtype != SONIQ_OUT_F16) return SONIQ_ERR_INVALID_ARG;   // the next layer reads fp16 activations
    if ((int64_t)geo_next->g[0].pa + geo_next->g[1].pa != N) return SONIQ_ERR_INVALID_ARG;
    if (!aligned(next->s_a, 4) || !aligned(next->Ap, 4)) return SONIQ_ERR_ALIGNMENT;
    return SONIQ_OK;
}

// Rows of a GEMM (output pixels of a convolution) the kernels address: their
// tile and TMA row coordinates are 32-bit.
constexpr int64_t kMaxRows = 2147483647;

// Taps, output size and output rows of a convolution, in 64-bit arithmetic:
// SONIQ_ERR_INVALID_ARG for a malformed geometry (the filter larger than the
// padded image included), SONIQ_ERR_UNSUPPORTED beyond the addressable sizes.
soniq_status conv_geometry(const soniq_conv_desc* cd, int32_t* taps, int32_t* P, int32_t* Q, int64_t* rows) {
    if (cd == nullptr || cd->R < 1 || cd->S < 1 || cd->stride_h < 1 || cd->stride_w < 1 || cd->pad_h < 0 ||
        cd->pad_w < 0 || cd->batch < 0 || cd->H < 1 || cd->W < 1 || cd->C_out < 0)
        return SONIQ_ERR_INVALID_ARG;
    const int64_t hp = (int64_t)cd->H + 2 * (int64_t)cd->pad_h, wp = (int64_t)cd->W + 2 * (int64_t)cd->pad_w;
    if (hp < cd->R || wp < cd->S) return SONIQ_ERR_INVALID_ARG;
    const int64_t t = (int64_t)cd->R * cd->S;
    const int64_t p = (hp - cd->R) / cd->stride_h + 1, q = (wp - cd->S) / cd->stride_w + 1;
    if (t > kMaxRows || p > kMaxRows || q > kMaxRows || p * q > kMaxRows || (int64_t)cd->batch * (p * q) > kMaxRows)
        return SONIQ_ERR_UNSUPPORTED;
    *taps = (int32_t)t;
    *P = (int32_t)p;
    *Q = (int32_t)q;
    *rows = (int64_t)cd->batch * p * q;
    return SONIQ_OK;
}

soniq_status check_scale_mode_act(int32_t mode) {
    return (mode == SONIQ_SCALE_PER_TENSOR || mode == SONIQ_SCALE_PER_ROW || mode == SONIQ_SCALE_CALIBRATED)
               ? SONIQ_OK
               : SONIQ_ERR_INVALID_ARG;
}

}  // namespace

extern "C" {

int32_t soniq_abi_version(void) { return SONIQ_ABI_VERSION; }

const char* soniq_status_string(soniq_status s) {
    switch (s) {
        case SONIQ_OK: return "ok";
        case SONIQ_ERR_INVALID_ARG: return "invalid argument";
        case SONIQ_ERR_UNSUPPORTED: return "unsupported configuration";
        case SONIQ_ERR_ALIGNMENT: return "misaligned pointer";
        case SONIQ_ERR_CUDA: return "CUDA error";
        case SONIQ_ERR_TIMEOUT: return "device wait timed out";
    }
    return "unknown status";
}

int64_t soniq_group_codes(const soniq_layout* L, int32_t group, int32_t is_weight, int32_t taps) {
    LayoutGeom geo;
    if (group < 0 || group > 1) return -1;
    if (make_geom(L, is_weight ? taps : 1, &geo) != SONIQ_OK) return -1;
    return is_weight ? geo.g[group].pw : geo.g[group].pa;
}

int64_t soniq_packed_row_bytes(const soniq_layout* L, int32_t is_weight, int32_t taps) {
    LayoutGeom geo;
    if (make_geom(L, is_weight ? taps : 1, &geo) != SONIQ_OK) return -1;
    return is_weight ? geo.w_row_bytes : geo.a_row_bytes;
}

int32_t soniq_scale_runs(const soniq_layout* L) {
    LayoutGeom geo;
    if (make_geom(L, 1, &geo) != SONIQ_OK) return -1;
    return geo.nb;
}

soniq_status soniq_validate_layout(const soniq_layout* L, const int32_t* perm_host) {
    LayoutGeom geo;
    soniq_status st = make_geom(L, 1, &geo);
    if (st != SONIQ_OK) return st;
    if (perm_host != nullptr) {
        std::vector<unsigned char> seen((size_t)L->K, 0);
        for (int32_t j = 0; j < L->K; ++j) {
            const int32_t c = perm_host[j];
            if (c < 0 || c >= L->K || seen[(size_t)c]) return SONIQ_ERR_INVALID_ARG;
            seen[(size_t)c] = 1;
        }
    }
    return SONIQ_OK;
}

int64_t soniq_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

soniq_status soniq_pack_weights(const soniq_layout* L, const float* W, int32_t N, int32_t taps,
                                int32_t scale_mode, uint8_t* Wp, float* s_w, soniq_stream_t stream) {
    LayoutGeom geo;
    soniq_status st = make_geom(L, taps, &geo);
    if (st != SONIQ_OK) return st;
    if (N < 0) return SONIQ_ERR_INVALID_ARG;
    if (scale_mode != SONIQ_SCALE_PER_ROW && scale_mode != SONIQ_SCALE_PER_TENSOR) return SONIQ_ERR_INVALID_ARG;
    if (N == 0) return SONIQ_OK;
    if (W == nullptr || Wp == nullptr || s_w == nullptr || L->perm == nullptr) return SONIQ_ERR_INVALID_ARG;
    if (!aligned(W, 4) || !aligned(Wp, 16) || !aligned(s_w, 4)) return SONIQ_ERR_ALIGNMENT;
    cudaStream_t s = as_stream(stream);
    if (geo.variant) {
        if (scale_mode != SONIQ_SCALE_PER_ROW) return SONIQ_ERR_UNSUPPORTED;
        return cuda_status(launch_variant_pack_weights(geo, L->perm, W, N, s_w, Wp, s));
    }
    if (scale_mode == SONIQ_SCALE_PER_TENSOR) {
        cudaError_t e = launch_weight_absmax(geo, L->perm, W, N, s_w, s);
        if (e != cudaSuccess) return cuda_status(e);
    }
    return cuda_status(launch_pack_weights(geo, L->perm, W, N, scale_mode == SONIQ_SCALE_PER_ROW, Wp, s_w, s));
}

int64_t soniq_quantize_act_scratch_bytes(const soniq_layout* L, int64_t M, int32_t scale_mode) {
    LayoutGeom geo;
    if (make_geom(L, 1, &geo) != SONIQ_OK || M < 0 || check_scale_mode_act(scale_mode) != SONIQ_OK) return -1;
    return scale_mode == SONIQ_SCALE_PER_TENSOR && M > 0 ? kQuantScratchBytes : 0;
}

soniq_status soniq_quantize_act(const soniq_layout* L, const void* A, int64_t M, int32_t scale_mode,
                                float* s_a, uint8_t* Ap, void* scratch, size_t scratch_bytes,
                                soniq_stream_t stream) {
    LayoutGeom geo;
    soniq_status st = make_geom(L, 1, &geo);
    if (st != SONIQ_OK) return st;
    if (L->K > 32768) return SONIQ_ERR_UNSUPPORTED;
    if (M < 0) return SONIQ_ERR_INVALID_ARG;
    if ((st = check_scale_mode_act(scale_mode)) != SONIQ_OK) return st;
    if (M == 0) return SONIQ_OK;
    if (A == nullptr || s_a == nullptr || Ap == nullptr || L->perm == nullptr) return SONIQ_ERR_INVALID_ARG;
    if (!aligned(A, 2) || !aligned(Ap, 4) || !aligned(s_a, 4) || (scratch != nullptr && !aligned(scratch, 16)))
        return SONIQ_ERR_ALIGNMENT;
    cudaStream_t s = as_stream(stream);
    const uint16_t* A16 = static_cast<const uint16_t*>(A);
    if (geo.variant) return cuda_status(launch_variant_quantize_act(geo, L->perm, A16, M, scale_mode, s_a, Ap, s));
    if (scale_mode == SONIQ_SCALE_PER_TENSOR) {
        // a small input (up to 16K values): one CTA finds the scale and quantizes, no scratch needed
        if (M * (int64_t)L->K <= 16384) {
            cudaError_t e0 = launch_quantize_rows(geo, L->perm, A16, M, scale_mode, true, s_a, Ap, s);
            if (e0 == cudaSuccess) return SONIQ_OK;
            if (e0 != cudaErrorNotSupported) return cuda_status(e0);
        }
        if (scratch != nullptr && scratch_bytes >= (size_t)kQuantScratchBytes) {
            // one pass: barrier words at the start of the scratch, per-CTA maxima after 256 bytes
            unsigned* bar = static_cast<unsigned*>(scratch);
            float* part = reinterpret_cast<float*>(static_cast<uint8_t*>(scratch) + 256);
            cudaError_t e = launch_quantize_fused(geo, L->perm, A16, M, s_a, Ap, s, bar, part, kMaxGridPartials,
                                                  kErrQuantBarrier);
            if (e == cudaSuccess) return SONIQ_OK;
            if (e != cudaErrorNotSupported) return cuda_status(e);
        }
    }
    const bool gather = quantize_gather_supported(geo, scale_mode, A);
    bool demote = false;
    if (scale_mode == SONIQ_SCALE_PER_TENSOR) {
        // two passes; an input that fits in L2 with room to spare stays there between them
        demote = gather && M * (int64_t)L->K * 2 <= kKeepInL2Bytes;
        cudaError_t e = launch_act_absmax(geo, L->perm, A16, M, s_a, demote, s);
        if (e != cudaSuccess) return cuda_status(e);
    }
    if (gather) return cuda_status(launch_quantize_gather(geo, L->perm, A16, M, scale_mode, demote, s_a, Ap, s));
    return cuda_status(launch_quantize_rows(geo, L->perm, A16, M, scale_mode, false, s_a, Ap, s));
}

soniq_status soniq_quantize_act_oneshot(const soniq_layout* L, const void* A, int64_t M, float* s_a, uint8_t* Ap,
                                        soniq_stream_t stream) {
    LayoutGeom geo;
    soniq_status st = make_geom(L, 1, &geo);
    if (st != SONIQ_OK) return st;
    if (geo.variant) return SONIQ_ERR_UNSUPPORTED;
    if (L->K > 32768) return SONIQ_ERR_UNSUPPORTED;
    if (M < 0) return SONIQ_ERR_INVALID_ARG;
    if (M == 0) return SONIQ_OK;
    if (A == nullptr || s_a == nullptr || Ap == nullptr || L->perm == nullptr) return SONIQ_ERR_INVALID_ARG;
    if (!aligned(A, 2) || !aligned(Ap, 4) || !aligned(s_a, 4)) return SONIQ_ERR_ALIGNMENT;
    unsigned* bar = nullptr;
    float* part = nullptr;
    if (!oneshot_scratch(&bar, &part)) return SONIQ_ERR_CUDA;
    const cudaError_t e = launch_quantize_fused(geo, L->perm, static_cast<const uint16_t*>(A), M, s_a, Ap,
                                                as_stream(stream), bar, part, kOneShotMaxCtas, kErrOneshotBarrier);
    if (e == cudaErrorNotSupported) return SONIQ_ERR_UNSUPPORTED;   // rows do not fit on chip: no fallback
    return cuda_status(e);
}

soniq_status soniq_mp_gemm(const soniq_layout* L, const uint8_t* Ap, const float* s_a, int32_t scale_mode,
                           int64_t M, const uint8_t* Wp, const float* s_w, int32_t N, void* Y,
                           int32_t out_dtype, int32_t* acc_dbg, uint32_t flags, void* scratch,
                           size_t scratch_bytes, const soniq_next_layer* next, soniq_stream_t stream) {
    LayoutGeom geo;
    soniq_status st = make_geom(L, 1, &geo);
    if (st != SONIQ_OK) return st;
    if (M < 0 || N < 0) return SONIQ_ERR_INVALID_ARG;
    if (M > kMaxRows) return SONIQ_ERR_UNSUPPORTED;
    if ((st = check_scale_mode_act(scale_mode)) != SONIQ_OK) return st;
    if (out_dtype != SONIQ_OUT_F16 && out_dtype != SONIQ_OUT_BF16) return SONIQ_ERR_INVALID_ARG;
    if ((flags & SONIQ_FLAG_FORCE_GEMV) && (flags & SONIQ_FLAG_FORCE_MMA)) return SONIQ_ERR_INVALID_ARG;
    if ((flags & SONIQ_FLAG_FORCE_FUSED) && (flags & SONIQ_FLAG_FORCE_STAGED)) return SONIQ_ERR_INVALID_ARG;
    if ((flags & SONIQ_FLAG_FORCE_SKINNY) && (flags & (SONIQ_FLAG_FORCE_FUSED | SONIQ_FLAG_FORCE_STAGED |
                                                      SONIQ_FLAG_FORCE_GEMV)))
        return SONIQ_ERR_INVALID_ARG;
    LayoutGeom geo_next;
    if (next != nullptr && (st = check_next(next, N, out_dtype, &geo_next)) != SONIQ_OK) return st;
    if (next != nullptr && (geo.variant || geo_next.variant)) return SONIQ_ERR_UNSUPPORTED;
    if (M == 0 || N == 0) return SONIQ_OK;
    if (Ap == nullptr || s_a == nullptr || Wp == nullptr || s_w == nullptr || (Y == nullptr && next == nullptr))
        return SONIQ_ERR_INVALID_ARG;
    if (!aligned(Ap, 4) || !aligned(Wp, 16) || !aligned(Y, 16) || !aligned(s_a, 4) || !aligned(s_w, 4) ||
        (acc_dbg != nullptr && !aligned(acc_dbg, 4)))
        return SONIQ_ERR_ALIGNMENT;
    // K <= 65536 keeps |Acc| < 2^31 and the GEMV's unsigned offset sums below 2^32
    const int per_row = scale_mode == SONIQ_SCALE_PER_ROW;
    cudaStream_t s = as_stream(stream);
    if (next != nullptr)
        flags = (flags & ~(uint32_t)(SONIQ_FLAG_FORCE_GEMV | SONIQ_FLAG_FORCE_SKINNY)) | SONIQ_FLAG_FORCE_MMA |
                SONIQ_FLAG_FORCE_STAGED;
    const int path = gemm_path(geo, M, N, flags, scratch != nullptr ? scratch_bytes : 0);
    if (next != nullptr && path != SONIQ_PATH_TENSOR_STAGED) return SONIQ_ERR_UNSUPPORTED;
    if (path < 0) return path == -2 ? SONIQ_ERR_UNSUPPORTED : mma_check(geo);
    if (path == SONIQ_PATH_GEMV) {
        GemvArgs a{Ap, Wp, s_a, s_w, Y, acc_dbg, (int32_t)M, N, per_row, out_dtype == SONIQ_OUT_BF16};
        return cuda_status(launch_gemv(geo, a, s));
    }
    if (path == SONIQ_PATH_TENSOR_STAGED && !aligned(scratch, 256)) return SONIQ_ERR_ALIGNMENT;
    MmaArgs a{};
    a.Ap = Ap;
    a.Wp = Wp;
    a.s_a = s_a;
    a.s_w = s_w;
    a.Y = Y;
    a.acc_dbg = acc_dbg;
    a.M = M;
    a.N = N;
    a.s_a_per_row = per_row;
    a.out_bf16 = out_dtype == SONIQ_OUT_BF16;
    a.flags = flags;
    a.conv = 0;
    if (next != nullptr) {
        a.next = &geo_next;
        a.next_s_a = next->s_a;
        a.next_Ap = next->Ap;
    }
    if (path == SONIQ_PATH_TENSOR_STAGED) return cuda_status(launch_staged(geo, a, scratch, scratch_bytes, s));
    if (path == SONIQ_PATH_TENSOR_SKINNY) return cuda_status(launch_skinny(geo, a, s));
    return cuda_status(launch_mma(geo, a, s));
}

soniq_status soniq_mp_conv2d(const soniq_layout* L, const soniq_conv_desc* cd, const uint8_t* Xp,
                             const float* s_a, int32_t scale_mode, const uint8_t* Wp, const float* s_w,
                             void* Y, int32_t out_dtype, int32_t* acc_dbg, uint32_t flags,
                             void* scratch, size_t scratch_bytes, const soniq_next_layer* next,
                             soniq_stream_t stream) {
    int32_t taps = 0, P = 0, Q = 0;
    int64_t M = 0;
    soniq_status st = conv_geometry(cd, &taps, &P, &Q, &M);
    if (st != SONIQ_OK) return st;
    LayoutGeom geo;
    if ((st = make_geom(L, taps, &geo)) != SONIQ_OK) return st;
    if (geo.variant) return SONIQ_ERR_UNSUPPORTED;   // the layout variants are for linear layers
    if (scale_mode != SONIQ_SCALE_PER_TENSOR && scale_mode != SONIQ_SCALE_CALIBRATED) return SONIQ_ERR_INVALID_ARG;
    if (out_dtype != SONIQ_OUT_F16 && out_dtype != SONIQ_OUT_BF16) return SONIQ_ERR_INVALID_ARG;
    LayoutGeom geo_next;
    if (next != nullptr && (st = check_next(next, cd->C_out, out_dtype, &geo_next)) != SONIQ_OK) return st;
    if (next != nullptr) flags |= SONIQ_FLAG_FORCE_STAGED;
    if (M == 0 || cd->C_out == 0) return SONIQ_OK;
    if (Xp == nullptr || s_a == nullptr || Wp == nullptr || s_w == nullptr || (Y == nullptr && next == nullptr))
        return SONIQ_ERR_INVALID_ARG;
    if (!aligned(Xp, 4) || !aligned(Wp, 16) || !aligned(Y, 16) || !aligned(s_a, 4) || !aligned(s_w, 4) ||
        (acc_dbg != nullptr && !aligned(acc_dbg, 4)))
        return SONIQ_ERR_ALIGNMENT;
    const bool staged = !(flags & SONIQ_FLAG_FORCE_FUSED) && scratch != nullptr &&
                        staged_worthwhile(geo, M, cd->C_out, flags) && staged_scratch_bytes(geo, M, cd->C_out) > 0 &&
                        (int64_t)scratch_bytes >= staged_scratch_bytes(geo, M, cd->C_out);
    if (staged && !aligned(scratch, 256)) return SONIQ_ERR_ALIGNMENT;
    if (next != nullptr && !staged) return SONIQ_ERR_UNSUPPORTED;
    if (!staged && (st = mma_check(geo)) != SONIQ_OK) return st;
    MmaArgs a{};
    a.Ap = Xp;
    a.Wp = Wp;
    a.s_a = s_a;
    a.s_w = s_w;
    a.Y = Y;
    a.acc_dbg = acc_dbg;
    a.M = M;
    a.N = cd->C_out;
    a.s_a_per_row = 0;
    a.out_bf16 = out_dtype == SONIQ_OUT_BF16;
    a.flags = flags;
    a.conv = 1;
    a.H = cd->H;
    a.W = cd->W;
    a.P = P;
    a.Q = Q;
    a.R = cd->R;
    a.S = cd->S;
    a.sh = cd->stride_h;
    a.sw = cd->stride_w;
    a.ph = cd->pad_h;
    a.pw = cd->pad_w;
    if (next != nullptr) {
        a.next = &geo_next;
        a.next_s_a = next->s_a;
        a.next_Ap = next->Ap;
    }
    if (staged) return cuda_status(launch_staged(geo, a, scratch, scratch_bytes, as_stream(stream)));
    return cuda_status(launch_mma(geo, a, as_stream(stream)));
}

int32_t soniq_mp_gemm_path(const soniq_layout* L, int64_t M, int32_t N, uint32_t flags, size_t scratch_bytes) {
    LayoutGeom geo;
    if (make_geom(L, 1, &geo) != SONIQ_OK || M < 1 || M > kMaxRows || N < 1) return -1;
    if ((flags & SONIQ_FLAG_FORCE_GEMV) && (flags & SONIQ_FLAG_FORCE_MMA)) return -1;
    const int p = gemm_path(geo, M, N, flags, scratch_bytes);
    return p < 0 ? -1 : p;
}

int64_t soniq_mp_gemm_scratch_bytes(const soniq_layout* L, int64_t M, int32_t N, uint32_t flags) {
    LayoutGeom geo;
    if (make_geom(L, 1, &geo) != SONIQ_OK || M < 0 || M > kMaxRows || N < 0) return -1;
    if (M == 0 || N == 0) return 0;
    if (geo.variant) return staged_scratch_bytes(geo, M, N);
    if (flags & SONIQ_FLAG_FORCE_FUSED) return 0;
    // the GEMV needs none
    const bool want_gemv =
        (flags & SONIQ_FLAG_FORCE_GEMV) ||
        (M <= SONIQ_GEMV_MAX_M && !(flags & (SONIQ_FLAG_FORCE_MMA | SONIQ_FLAG_FORCE_SKINNY)));
    if (want_gemv) return 0;
    // nor the skinny kernel
    const bool pinned = (flags & (SONIQ_FLAG_FORCE_FUSED | SONIQ_FLAG_FORCE_STAGED)) != 0;
    if ((flags & SONIQ_FLAG_FORCE_SKINNY) || (!pinned && M <= SONIQ_SKINNY_MAX_M && skinny_supported(geo, M, N)))
        return 0;
    return staged_worthwhile(geo, M, N, flags) ? staged_scratch_bytes(geo, M, N) : 0;
}

int64_t soniq_mp_conv2d_scratch_bytes(const soniq_layout* L, const soniq_conv_desc* cd, uint32_t flags) {
    LayoutGeom geo;
    int32_t taps = 0, P = 0, Q = 0;
    int64_t rows = 0;
    if (conv_geometry(cd, &taps, &P, &Q, &rows) != SONIQ_OK || make_geom(L, taps, &geo) != SONIQ_OK) return -1;
    if (flags & SONIQ_FLAG_FORCE_FUSED || !staged_worthwhile(geo, rows, cd->C_out, flags)) return 0;
    return staged_scratch_bytes(geo, rows, cd->C_out);
}

soniq_status soniq_sync_status(soniq_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize(as_stream(stream));
    if (e != cudaSuccess) return SONIQ_ERR_CUDA;
    unsigned* addr = device_error_word();
    if (addr == nullptr) return SONIQ_ERR_CUDA;
    unsigned v = 0;
    if (cudaMemcpy(&v, addr, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return SONIQ_ERR_CUDA;
    if (v == 0) return SONIQ_OK;
    if (v & kErrOneshotBarrier) {
        // The abandoned one-shot barrier kept the arrivals of the CTAs that got
        // there.  Once no kernel of any stream can still be using it, start it afresh.
        unsigned* bar = nullptr;
        float* part = nullptr;
        if (cudaDeviceSynchronize() != cudaSuccess || !oneshot_scratch(&bar, &part) ||
            cudaMemset(bar, 0, 2 * sizeof(unsigned)) != cudaSuccess)
            return SONIQ_ERR_CUDA;
    }
    const unsigned zero = 0;
    if (cudaMemcpy(addr, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess) return SONIQ_ERR_CUDA;
    return SONIQ_ERR_TIMEOUT;
}

void soniq_test_drop_barrier_arrival(int32_t armed) { g_drop_arrival.store(armed != 0 ? 1 : 0); }

}  // extern "C"
