// Device helpers shared by the SONIQ kernels: the quantizers (Sec. 3 steps
// 2 and 3, Eq. (1)), packing of a 32-code block by one warp, and the
// SIMD-in-register expansion of a packed block back to bytes.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

namespace soniq {

// ---- quantizers ------------------------------------------------------------
// Both decide the integer code in fp32 with the operation order of the
// paper's formulas: divide by the group scale (IEEE, round to nearest), then
// multiply by the level count, round half to even, clip.  A zero scale (an
// all-zero group) gives code 0.

// Activation (Sec. 3 step 2): u = clip(round(a / s * (2^n - 1)), 0, 2^n - 1).
__device__ __forceinline__ uint32_t act_code(float a, float s, float levels) {
    if (!(s > 0.0f)) return 0u;
    float t = __fmul_rn(__fdiv_rn(a, s), levels);
    float r = rintf(t);
    r = fminf(fmaxf(r, 0.0f), levels);
    return (uint32_t)r;
}

// Weight (Sec. 3 step 3, Eq. (1)): nearest level j / 2^(n-1) to w / s,
// j in [-2^(n-1), 2^(n-1) - 1]; `half` = 2^(n-1).  The conversion rounds half
// to even and saturates, so +-inf reach the end levels through the clip and a
// NaN quotient gives code 0.
__device__ __forceinline__ int32_t weight_code(float w, float s, float half) {
    if (!(s > 0.0f)) return 0;
    const float t = __fmul_rn(__fdiv_rn(w, s), half);
    const int32_t h = (int32_t)half;
    return min(max(__float2int_rn(t), -h), h - 1);
}

// min(x, s) that keeps a NaN x (the plain fminf would return s).
__device__ __forceinline__ float fmin_keep_nan(float x, float s) {
    float r;
    asm("min.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(x), "f"(s));
    return r;
}

// The code of Sec. 3 step 2, t = (a / s) * (2^n - 1) rounded half to even and
// clipped to [0, 2^n - 1].  The quotient is formed by Markstein's correction
// step: q0 = a * r, q = q0 + (a - q0 * s) * r with r = RN(1 / s), both
// products fused; for |a| <= 65504 and s in [2^-60, 2^60] this is the
// correctly rounded quotient (checked exhaustively over every fp16 a); other
// scales take the IEEE division.  Rounding to an unsigned integer saturates
// negative values (and NaN) at 0, which is the clip at 0.  On the Markstein
// path the top clip is taken on the input instead: a above s becomes s, whose
// quotient is exactly 1, so every a >= s (+inf too, which the residual would
// turn into NaN) gets the top code and no quotient exceeds 1; a NaN input
// stays NaN and gets code 0.
template <bool FAST>
__device__ __forceinline__ uint32_t act_code_q(float a, float s, float r, float levels, uint32_t top) {
    if constexpr (FAST) {
        const float x = fmin_keep_nan(a, s);
        const float q0 = x * r;
        const float q = fmaf(fmaf(-q0, s, x), r, q0);
        return __float2uint_rn(__fmul_rn(q, levels));
    } else {
        return min(__float2uint_rn(__fmul_rn(__fdiv_rn(a, s), levels)), top);
    }
}

// Quantizer constants of one (row or tensor, group): scale, its reciprocal,
// the level count and the largest code.
struct QConst {
    float s, r, levels;
    uint32_t top;
    int mode;   // 0: every code is 0 (no positive scale); 1: Markstein quotient; 2: IEEE division
};

__device__ __forceinline__ QConst make_qconst(float s, int n) {
    QConst q;
    q.s = s;
    q.levels = (float)((1 << n) - 1);
    q.top = (1u << n) - 1u;
    q.mode = (s >= 0x1p-60f && s <= 0x1p60f) ? 1 : (s > 0.0f ? 2 : 0);
    q.r = q.mode == 1 ? __frcp_rn(s) : 0.0f;
    return q;
}

// ---- packed block layout ---------------------------------------------------
// 32 codes of n bits -> n words.  Code bits are cut into slices of width 4,
// 2, 1 (low bits first; n = 8 is one slice).  In a w-bit slice, code i
// (t = i/4, b = i%4) sits in slice word t/(8/w) at bit 8*b + w*(t%(8/w)), so
// shifting slice word q right by w*s and masking the low w bits of each byte
// yields codes 4*(q*(8/w)+s) .. +3 in byte order.

// One warp packs one block: lane i holds code pattern i; the return value of
// lane q (q < n) is word q of the block.
__device__ __forceinline__ uint32_t pack_block_warp(uint32_t code, int n) {
    const int lane = threadIdx.x & 31;
    const int t = lane >> 2, b = lane & 3;
    uint32_t mine = 0u;
    int word = 0, off = 0;
    const int widths[3] = {n == 8 ? 8 : (n & 4), n == 8 ? 0 : (n & 2), n == 8 ? 0 : (n & 1)};
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        const int w = widths[k];
        if (w == 0) continue;
        const int per = 8 / w;
        const uint32_t v = (code >> off) & ((1u << w) - 1u);
        const int my_q = t / per;
        const uint32_t shifted = v << (8 * b + w * (t % per));
        for (int q = 0; q < w; ++q) {
            uint32_t r = __reduce_or_sync(0xffffffffu, my_q == q ? shifted : 0u);
            if (lane == word + q) mine = r;
        }
        word += w;
        off += w;
    }
    return mine;
}

// One thread packs one block: the inverse of block_to_bytes.  Byte b of o[t]
// holds code 4*t + b (< 2^N); w receives the block's N words.
template <int N>
__device__ __forceinline__ void bytes_to_block(const uint32_t* o, uint32_t* w) {
    if constexpr (N == 8) {
#pragma unroll
        for (int t = 0; t < 8; ++t) w[t] = o[t];
    } else {
        int word = 0, off = 0;
        if constexpr ((N & 4) != 0) {
#pragma unroll
            for (int q = 0; q < 4; ++q) w[q] = (o[2 * q] & 0x0F0F0F0Fu) | ((o[2 * q + 1] & 0x0F0F0F0Fu) << 4);
            word += 4;
            off += 4;
        }
        if constexpr ((N & 2) != 0) {
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                uint32_t v = 0u;
#pragma unroll
                for (int j = 0; j < 4; ++j) v |= ((o[4 * q + j] >> off) & 0x03030303u) << (2 * j);
                w[word + q] = v;
            }
            word += 2;
            off += 2;
        }
        if constexpr ((N & 1) != 0) {
            uint32_t v = 0u;
#pragma unroll
            for (int t = 0; t < 8; ++t) v |= ((o[t] >> off) & 0x01010101u) << t;
            w[word] = v;
        }
    }
}

// Expands one packed block (N words at w) to 8 words of bytes: byte b of
// o[t] is the N-bit pattern of code 4*t + b.
template <int N>
__device__ __forceinline__ void block_to_bytes(const uint32_t* w, uint32_t* o) {
    if constexpr (N == 8) {
#pragma unroll
        for (int t = 0; t < 8; ++t) o[t] = w[t];
    } else {
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            uint32_t v = 0u;
            int word = 0, off = 0;
            if constexpr ((N & 4) != 0) {
                v |= (w[word + t / 2] >> (4 * (t % 2))) & 0x0F0F0F0Fu;
                word += 4;
                off += 4;
            }
            if constexpr ((N & 2) != 0) {
                v |= ((w[word + t / 4] >> (2 * (t % 4))) & 0x03030303u) << off;
                word += 2;
                off += 2;
            }
            if constexpr ((N & 1) != 0) {
                v |= ((w[word] >> t) & 0x01010101u) << off;
            }
            o[t] = v;
        }
    }
}

// One thread stores a packed block: 8 words of code bytes -> N words at dst
// (16- or 8-byte stores where dst allows).
template <int N>
__device__ __forceinline__ void store_block32(const uint32_t* o, uint8_t* dst) {
    uint32_t w[N];
    bytes_to_block<N>(o, w);
    if constexpr (N % 4 == 0) {
        if ((reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
#pragma unroll
            for (int q = 0; q < N; q += 4)
                *reinterpret_cast<uint4*>(dst + 4 * q) = make_uint4(w[q], w[q + 1], w[q + 2], w[q + 3]);
            return;
        }
    }
    if constexpr (N % 2 == 0) {
        if ((reinterpret_cast<uintptr_t>(dst) & 7u) == 0) {
#pragma unroll
            for (int q = 0; q < N; q += 2) *reinterpret_cast<uint2*>(dst + 4 * q) = make_uint2(w[q], w[q + 1]);
            return;
        }
    }
#pragma unroll
    for (int q = 0; q < N; ++q) reinterpret_cast<uint32_t*>(dst)[q] = w[q];
}

__device__ __forceinline__ void store_block32_n(int n, const uint32_t* o, uint8_t* dst) {
    switch (n) {
        case 1: store_block32<1>(o, dst); break;
        case 2: store_block32<2>(o, dst); break;
        case 3: store_block32<3>(o, dst); break;
        case 4: store_block32<4>(o, dst); break;
        case 5: store_block32<5>(o, dst); break;
        case 6: store_block32<6>(o, dst); break;
        case 7: store_block32<7>(o, dst); break;
        default: store_block32<8>(o, dst); break;
    }
}

// One packed block from 8 words of code bytes (byte b of o[t] is code
// 4*t + b), for a width n known only at run time: the slice words of every
// width are formed and the n output words selected from them, so the code is
// short and indexes no register array by a run-time value.  dst is 4-byte
// aligned.
__device__ __forceinline__ void store_block32_rt(int n, const uint32_t (&o)[8], uint8_t* dst) {
    uint32_t* d = reinterpret_cast<uint32_t*>(dst);
    if (n == 8) {
#pragma unroll
        for (int t = 0; t < 8; ++t) d[t] = o[t];
        return;
    }
    const int off2 = n & 4;                  // bit offset of the 2-bit slice in each code
    const int off1 = (n & 4) + (n & 2);      // bit offset of the 1-bit slice
    uint32_t s4[4], s2[2], s1 = 0u;
#pragma unroll
    for (int q = 0; q < 4; ++q) s4[q] = (o[2 * q] & 0x0F0F0F0Fu) | ((o[2 * q + 1] & 0x0F0F0F0Fu) << 4);
#pragma unroll
    for (int q = 0; q < 2; ++q) {
        uint32_t v = 0u;
#pragma unroll
        for (int j = 0; j < 4; ++j) v |= ((o[4 * q + j] >> off2) & 0x03030303u) << (2 * j);
        s2[q] = v;
    }
#pragma unroll
    for (int t = 0; t < 8; ++t) s1 |= ((o[t] >> off1) & 0x01010101u) << t;
    const int b2 = (n & 4) ? 4 : 0;          // first word of the 2-bit slice
    const int b1 = b2 + ((n & 2) ? 2 : 0);   // the word of the 1-bit slice
#pragma unroll
    for (int q = 0; q < 7; ++q) {
        const uint32_t w = q < b2 ? s4[q & 3] : (q < b1 ? (((q - b2) & 1) ? s2[1] : s2[0]) : s1);
        if (q < n) d[q] = w;
    }
}

// Byte-wise sign-bit flip: n-bit two's complement j -> offset binary j + 2^(n-1).
__device__ __forceinline__ uint32_t sign_flip_mask(int n) { return 0x01010101u << (n - 1); }

// Runtime-n dispatch of block_to_bytes.
__device__ __forceinline__ void block_to_bytes_n(int n, const uint32_t* w, uint32_t* o) {
    switch (n) {
        case 1: block_to_bytes<1>(w, o); break;
        case 2: block_to_bytes<2>(w, o); break;
        case 3: block_to_bytes<3>(w, o); break;
        case 4: block_to_bytes<4>(w, o); break;
        case 5: block_to_bytes<5>(w, o); break;
        case 6: block_to_bytes<6>(w, o); break;
        case 7: block_to_bytes<7>(w, o); break;
        default: block_to_bytes<8>(w, o); break;
    }
}

// Four bytes -> two fp16x2 words holding 1024 + byte (the exponent field of
// 1024.0 is placed above each byte; Kim et al. 2022 "magic number" conversion).
__device__ __forceinline__ void bytes_to_magic_half2(uint32_t x, uint32_t& lo, uint32_t& hi) {
    lo = __byte_perm(x, 0x64646464u, 0x5150);
    hi = __byte_perm(x, 0x64646464u, 0x5352);
}

__device__ __forceinline__ uint32_t half2_sub(uint32_t a, __half2 b) {
    __half2 h = *reinterpret_cast<__half2*>(&a);
    h = __hsub2(h, b);
    return *reinterpret_cast<uint32_t*>(&h);
}

}  // namespace soniq
