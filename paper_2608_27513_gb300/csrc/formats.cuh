// formats.cuh -- the 4-bit and FP8 low tiers (App. A.1, Tab. quantizer_specs):
//   format 3  UINT4 affine, G = 32, FP16 (s, z), H_32 first
//   format 4  UINT4 affine, G = 32, FP16 (s, z)
//   format 5  FP8 E4M3, G = 32, one FP32 scale, natural domain (Eq. fp8_storage):
//             s = max(max|x|, 1e-10) / 448, q = E4M3(clip(x / s, -448, 448)), x^ = s q
// A UINT4 code row holds 32 codes in 16 bytes, value 2i in the low nibble of byte i.
// The UINT8 helpers (formats 0, 1) live in damp_common.cuh.
#pragma once

#include "damp_common.cuh"

namespace damp {

enum : int { kFmtU8H32 = 0, kFmtU8 = 1, kFmtS8Row = 2, kFmtU4H32 = 3, kFmtU4 = 4, kFmtE4M3 = 5 };

__host__ __device__ constexpr bool fmt_had(int fmt) { return fmt == kFmtU8H32 || fmt == kFmtU4H32; }
__host__ __device__ constexpr bool fmt_u4(int fmt) { return fmt == kFmtU4H32 || fmt == kFmtU4; }

// Two integers saturated to [0, 15] and packed as nibbles: (upper << 8) | (hi << 4) | lo.
__device__ __forceinline__ uint32_t pack_sat_u4(uint32_t hi_nib, uint32_t lo_nib, uint32_t upper) {
    uint32_t d;
    asm("cvt.pack.sat.u4.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(hi_nib), "r"(lo_nib), "r"(upper));
    return d;
}

// UINT4 affine parameters from the scaled extrema (levels 15), as affine_params_scaled.
__device__ __forceinline__ uint32_t affine_params_u4(float mn, float mx, float &inv_out, float &z_out) {
    const float s0 = __half2float(__float2half_rn((mx - mn) * (kUp / 15.0f)));
    const float mn0 = fminf(mn, 0.0f), mx0 = fmaxf(mx, 0.0f);
    float s1 = __half2float(__float2half_rn((mx0 - mn0) * (kUp / 15.0f)));
    s1 = (s1 == 0.0f) ? 1.0f : s1;
    const bool degenerate = s0 == 0.0f;
    const float s = degenerate ? s1 : s0;
    const float m = degenerate ? mn0 : mn;
    const float inv = rcp_approx(s);
    const __half zh = __float2half_rn(rintf(-m * (inv * kUp)));
    z_out = __half2float(zh);
    inv_out = inv;
    return (uint32_t)__half_as_ushort(__float2half_rn(s)) | ((uint32_t)__half_as_ushort(zh) << 16);
}

// UINT4 codes of one group of scaled values: 4 words of 8 nibbles + packed (s, z).
__device__ __forceinline__ uint32_t quantize_group_u4(const float2 (&y)[16], uint32_t (&w)[4]) {
    float mn, mx, inv, z;
    minmax32(y, mn, mx);
    const uint32_t sz = affine_params_u4(mn, mx, inv, z);
    const float2 inv2 = splat2(inv * 0x1p-110f), zc2 = splat2(z * 0x1p-149f);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        // values 8i .. 8i+7 = pairs y[4i .. 4i+3]; the last pair goes in first so that
        // value 8i ends in the low nibble of byte 0
        uint32_t acc = 0u;
#pragma unroll
        for (int k = 3; k >= 0; --k) {
            const float2 a = fma2(y[4 * i + k], inv2, zc2);
            acc = pack_sat_u4(__float_as_uint(a.y), __float_as_uint(a.x), acc);
        }
        w[i] = acc;
    }
    return sz;
}

// x_j = (q_j - z) * (s * scale) from 4 words of nibbles.
__device__ __forceinline__ void dequantize_group_u4(const uint32_t (&w)[4], uint32_t sz, float scale,
                                                    float2 (&x)[16]) {
    const float s = __half2float(__ushort_as_half((unsigned short)(sz & 0xffffu)));
    const float z = __half2float(__ushort_as_half((unsigned short)(sz >> 16)));
    const float2 nzb = splat2(-(8388608.0f + z));
    const float2 sa = splat2(s * scale);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t lo = w[i] & 0x0F0F0F0Fu, hi = (w[i] >> 4) & 0x0F0F0F0Fu;  // even / odd values
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const float2 f = make_float2(__uint_as_float(prmt(lo, 0x4B000000u, 0x7650u + b)),
                                         __uint_as_float(prmt(hi, 0x4B000000u, 0x7650u + b)));
            x[4 * i + b] = mul2(add2(f, nzb), sa);
        }
    }
}

// FP8 E4M3 pair <-> floats (hardware conversions, round to nearest even).
__device__ __forceinline__ uint32_t e4m3x2_of(float hi, float lo) {  // bits: hi in [15:8], lo in [7:0]
    unsigned short d;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(hi), "f"(lo));
    return d;
}
__device__ __forceinline__ float2 f2_of_e4m3x2(uint32_t bits16) {  // (value of [7:0], value of [15:8])
    uint32_t h;
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h) : "h"((unsigned short)bits16));
    return h2_to_f2(h);
}

// FP8 codes of one group of natural values: 8 words + the FP32 scale (IEEE division,
// as the definition writes it).
__device__ __forceinline__ float quantize_group_e4m3(const float2 (&x)[16], uint32_t (&w)[8]) {
    float amax = 0.f;
#pragma unroll
    for (int j = 0; j < 16; ++j) amax = fmaxf(amax, fmaxf(fabsf(x[j].x), fabsf(x[j].y)));
    const float s = __fdiv_rn(fmaxf(amax, 1e-10f), 448.0f);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        float t[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float v = (e & 1) ? x[2 * i + (e >> 1)].y : x[2 * i + (e >> 1)].x;
            t[e] = fminf(fmaxf(__fdiv_rn(v, s), -448.0f), 448.0f);
        }
        w[i] = e4m3x2_of(t[1], t[0]) | (e4m3x2_of(t[3], t[2]) << 16);  // value 4i in byte 0
    }
    return s;
}

// x_j = s * FP32(q_j) * scale (scale = 1 or an exact power of two).
__device__ __forceinline__ void dequantize_group_e4m3(const uint32_t (&w)[8], float s, float scale,
                                                      float2 (&x)[16]) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const float2 a = f2_of_e4m3x2(w[i] & 0xffffu), b = f2_of_e4m3x2(w[i] >> 16);
        x[2 * i] = make_float2(__fmul_rn(__fmul_rn(s, a.x), scale), __fmul_rn(__fmul_rn(s, a.y), scale));
        x[2 * i + 1] = make_float2(__fmul_rn(__fmul_rn(s, b.x), scale), __fmul_rn(__fmul_rn(s, b.y), scale));
    }
}

}  // namespace damp
