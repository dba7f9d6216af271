// damp_common.cuh -- device helpers shared by libdamp's kernels (sm_103a).
//
// Inline PTX for the mbarrier / bulk-copy (TMA engine) pipeline, the packed
// record geometry, the block-32 Hadamard butterflies and the UINT8 affine
// requantizer of Sec. 3.2 (Eq. integer_quantizer).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace damp {

constexpr int kG = 32;                        // quantization group = value block (App. A.1)
constexpr float kInvSqrt32 = 0.17677669529663687f;  // fp32(1/sqrt(32)), H_32 normalization
constexpr unsigned kFull = 0xffffffffu;

enum : uint32_t { kDevWaitTimeout = 1u, kDevBadSlot = 2u, kDevBadHead = 4u };

// ---------------------------------------------------------------------------
// Packed record geometry (one (slot, head, value block) record).
//   hi rows:   ceil(K/2) pairs x 128 B at 0: pair i holds rows 2i and 2i+1 as
//              32 column words (binary16 of row 2i in the low half); an odd K
//              leaves the last high half zero.  A lane reads two FP16 rows of its
//              column with one 32-bit load.
//   codes:     (d_k-K) x 32 B, chunk-major: 16-B chunk m (columns 16m .. 16m+15)
//              of lo row r at 16 * (m * (d_k-K) + r); 4-bit formats: one 16-B chunk
//              (all 32 codes) per row at 16 * r
//   meta:      (d_k-K) x 4 B      (s, z) as two binary16, or an FP32 scale
// With one lane per lo row, a warp's 128-bit access to chunk m of 32 consecutive
// rows covers 512 contiguous bytes: conflict-free in shared memory, whole
// sectors in global memory.
// ---------------------------------------------------------------------------
struct RecGeom {
    int codes_off, meta_off, bytes;
};

// code bits of a low-tier format: 4 for the UINT4 formats (3, 4), 8 for the others
__host__ __device__ constexpr int fmt_code_bits(int fmt) { return fmt == 3 || fmt == 4 ? 4 : 8; }

__host__ __device__ inline RecGeom rec_geom(int d_k, int k_hi, int fmt = 0) {
    RecGeom g;
    g.codes_off = 128 * ((k_hi + 1) / 2);
    g.meta_off = g.codes_off + 4 * fmt_code_bits(fmt) * (d_k - k_hi);
    g.bytes = (g.meta_off + 4 * (d_k - k_hi) + 15) & ~15;
    return g;
}

// byte offset of FP16 row u, column j (0..31) inside a record
__host__ __device__ inline int hi_elem_off(int u, int j) { return 128 * (u >> 1) + 4 * j + 2 * (u & 1); }
__host__ __device__ inline int lo_chunk_off(int r, int m, int lo) { return 16 * (m * lo + r); }

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

// Invalidates a completed mbarrier so that its shared memory can be reused (by another
// barrier or by data).
__device__ __forceinline__ void mbar_inval(uint32_t bar) {
    asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t global_timer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait on an mbarrier phase: gives up after limit_ns (~2 s by default) or
// 2^26 polls and returns false, so a lost copy ends the kernel with an error flag,
// not a hang.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  uint64_t limit_ns = 2000000000ull) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; it < (1u << 26); ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 255u) == 255u && global_timer_ns() - t0 > limit_ns) break;
    }
    return false;
}

// Counts `bytes` of expected transaction bytes of the barrier's current phase as done
// (without a copy): used only to settle a phase that was armed for more bytes than
// its copy delivers.
__device__ __forceinline__ void mbar_complete_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.complete_tx.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

// 1-D bulk copy global -> shared (TMA engine), completion on an mbarrier.
// Addresses 16-B aligned, size a multiple of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// Orders this thread's generic-proxy accesses of shared memory before later
// async-proxy accesses (a bulk copy into the same stage).
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 16-byte asynchronous copy global -> shared through the load/store path (not the
// bulk-copy engine); completion per thread with cp.async.wait_group.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void stg128(void *p, uint4 v) {
    asm volatile("st.global.v4.b32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ void stg32(void *p, uint32_t v) {
    asm volatile("st.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ void sts128(uint32_t a, uint4 v) {
    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ void sts32(uint32_t a, uint32_t v) {
    asm volatile("st.shared.b32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}


__device__ __forceinline__ float fmin3(float a, float b, float c) {
    float d;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// ---------------------------------------------------------------------------
// Block-32 Hadamard (Sylvester order, normalized by fp32(1/sqrt 32)).
// ---------------------------------------------------------------------------

// Across the 32 lanes of a warp: lane j holds x_j, returns (H_32 x)_j.
// Butterfly signs of a lane: round m (partner lane ^ 2^m) adds for bit m clear
// and subtracts for bit m set; fma(x, sign, y) is then y - x or x + y, rounded once.
struct LaneSigns {
    float s[5];
};
__device__ __forceinline__ LaneSigns lane_signs(int lane) {
    LaneSigns g;
#pragma unroll
    for (int i = 0; i < 5; ++i) g.s[i] = (lane >> i) & 1 ? -1.0f : 1.0f;
    return g;
}
__device__ __forceinline__ float hadamard_lanes(float x, const LaneSigns &g) {
#pragma unroll
    for (int i = 0; i < 5; ++i) {
        const float y = __shfl_xor_sync(kFull, x, 1 << i);
        x = __fmaf_rn(x, g.s[i], y);
    }
    return x * kInvSqrt32;
}

// Inside one thread: x[0..31] -> H_32 x.
__device__ __forceinline__ void hadamard_regs(float (&x)[32]) {
#pragma unroll
    for (int m = 1; m < 32; m <<= 1) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            if ((j & m) == 0) {
                const float a = x[j], b = x[j + m];
                x[j] = a + b;
                x[j + m] = a - b;
            }
        }
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) x[j] *= kInvSqrt32;
}

// ---------------------------------------------------------------------------
// UINT8 affine codec of one 32-group held in registers (Sec. 3.2; App. A.1).
// ---------------------------------------------------------------------------

// Byte b of the word placed in the low mantissa of 2^23: exact float 2^23 + byte.
__device__ __forceinline__ float u8_biased(uint32_t word, int b) {
    return __uint_as_float(prmt(word, 0x4B000000u, 0x7650u + b) );
}

// ---------------------------------------------------------------------------
// Packed FP32 pairs (FFMA2 / FADD2 / FMUL2 on sm_100+): two lanes of FP32
// arithmetic per issue slot, each component rounded exactly like the scalar op.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float2 splat2(float a) { return make_float2(a, a); }
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 add2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 mul2(float2 a, float2 b) { return __fmul2_rn(a, b); }

__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// ---------------------------------------------------------------------------
// Scaled working domain.  Low-tier values are kept multiplied by 2^-39 while a
// tile is in registers (exact power-of-two scaling: every FP32 rounding is the
// same as in the unscaled domain for |x| >= 2^-87).  This lets the requantizer
// land each code directly on the binary32 denormal grid (below).
// ---------------------------------------------------------------------------
constexpr float kDown = 0x1p-39f;
constexpr float kUp = 0x1p39f;

// Scale and zero point of a group from its scaled extrema mn', mx':
//   s = fp16((max - min)/255), z = fp16(round_even(-min / s)); a block whose s
//   rounds to 0 widens [min, max] to contain 0, and s = 1, z = 0 if s is still 0.
// Returns the packed (s, z) binary16 pair, inv ~ 1/s (hardware reciprocal,
// within one ulp: a code can only move where x/s + z sits at a rounding tie)
// and z as float.
__device__ __forceinline__ uint32_t affine_params_scaled(float mn, float mx, float &inv_out, float &z_out) {
    // branch-free so that the chains of several rows interleave
    const float s0 = __half2float(__float2half_rn((mx - mn) * (kUp / 255.0f)));
    const float mn0 = fminf(mn, 0.0f), mx0 = fmaxf(mx, 0.0f);
    float s1 = __half2float(__float2half_rn((mx0 - mn0) * (kUp / 255.0f)));
    s1 = (s1 == 0.0f) ? 1.0f : s1;
    const bool degenerate = s0 == 0.0f;
    const float s = degenerate ? s1 : s0;
    const float m = degenerate ? mn0 : mn;
    const float inv = rcp_approx(s);
    const __half zh = __float2half_rn(rintf(-m * (inv * kUp)));
    const __half sh = __float2half_rn(s);  // exact: s is already a binary16 value
    z_out = __half2float(zh);
    inv_out = inv;
    return (uint32_t)__half_as_ushort(sh) | ((uint32_t)__half_as_ushort(zh) << 16);
}

// Codes of 4 scaled values: q = sat_[0,255](round_even(x / s) + z), packed
// little-endian.  fma(x', inv * 2^-110, z * 2^-149) computes x/s + z scaled by
// 2^-149 and rounds it once onto the denormal grid, so its bit pattern is the
// integer round_even(x/s + z) (with the sign bit set when negative);
// cvt.pack.sat saturates two such integers to [0, 255] and packs them.
__device__ __forceinline__ uint32_t pack_sat_u8(uint32_t hi_byte, uint32_t lo_byte, uint32_t upper) {
    uint32_t d;
    asm("cvt.pack.sat.u8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(hi_byte), "r"(lo_byte), "r"(upper));
    return d;
}
__device__ __forceinline__ uint32_t encode4(float2 x01, float2 x23, float2 inv2, float2 zc2) {
    const float2 a = fma2(x01, inv2, zc2);
    const float2 b = fma2(x23, inv2, zc2);
    const uint32_t upper = pack_sat_u8(__float_as_uint(b.y), __float_as_uint(b.x), 0u);
    return pack_sat_u8(__float_as_uint(a.y), __float_as_uint(a.x), upper);
}

// Extrema of 32 values with three-input min/max only: 32 -> 11 -> 4 -> 2 -> 1
// (16 operations each for min and max).
__device__ __forceinline__ void minmax32(const float2 (&y)[16], float &mn, float &mx) {
    float v[32];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        v[2 * j] = y[j].x;
        v[2 * j + 1] = y[j].y;
    }
    float a[11], b[11];
#pragma unroll
    for (int i = 0; i < 10; ++i) {
        a[i] = fmin3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
        b[i] = fmax3(v[3 * i], v[3 * i + 1], v[3 * i + 2]);
    }
    a[10] = fminf(v[30], v[31]);
    b[10] = fmaxf(v[30], v[31]);
    const float a0 = fmin3(a[0], a[1], a[2]), a1 = fmin3(a[3], a[4], a[5]), a2 = fmin3(a[6], a[7], a[8]);
    const float b0 = fmax3(b[0], b[1], b[2]), b1 = fmax3(b[3], b[4], b[5]), b2 = fmax3(b[6], b[7], b[8]);
    mn = fmin3(fmin3(a0, a1, a2), a[9], a[10]);
    mx = fmax3(fmax3(b0, b1, b2), b[9], b[10]);
}

// Scale and zero point from the scale s already known to be nonzero (the common
// case): returns the packed (s, z) pair, inv ~ 1/s and z.
__device__ __forceinline__ uint32_t affine_finish(float s, float mn, float &inv_out, float &z_out) {
    const float inv = rcp_approx(s);
    const __half zh = __float2half_rn(rintf(-mn * (inv * kUp)));
    z_out = __half2float(zh);
    inv_out = inv;
    return (uint32_t)__half_as_ushort(__float2half_rn(s)) | ((uint32_t)__half_as_ushort(zh) << 16);
}

// binary16 scale of a scaled range: fp16((max - min) / 255)
__device__ __forceinline__ float scale_of(float mn, float mx) {
    return __half2float(__float2half_rn((mx - mn) * (kUp / 255.0f)));
}

// Quantize y' (one lo row, one value block, 16 pairs, scaled by 2^-39) into
// 8 code words + packed (s, z).
__device__ __forceinline__ uint32_t quantize_group(const float2 (&y)[16], uint32_t (&w)[8]) {
    float mn, mx, inv, z;
    minmax32(y, mn, mx);
    const uint32_t sz = affine_params_scaled(mn, mx, inv, z);
    const float2 inv2 = splat2(inv * 0x1p-110f), zc2 = splat2(z * 0x1p-149f);
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = encode4(y[2 * i], y[2 * i + 1], inv2, zc2);
    return sz;
}

// Dequantize 8 code words with (s, z): x_j = (q_j - z) * (s * scale); scale folds
// the decay and, on the hot path, the 2^-39 working scale.
// 2^23 + q comes straight from a byte permute; subtracting 2^23 + z is exact.
__device__ __forceinline__ void dequantize_group(const uint32_t (&w)[8], uint32_t sz, float scale, float2 (&x)[16]) {
    const float s = __half2float(__ushort_as_half((unsigned short)(sz & 0xffffu)));
    const float z = __half2float(__ushort_as_half((unsigned short)(sz >> 16)));
    const float2 nzb = splat2(-(8388608.0f + z));  // -(2^23 + z), exact for |z| <= 2^23
    const float2 sa = splat2(s * scale);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        x[2 * i] = mul2(add2(make_float2(u8_biased(w[i], 0), u8_biased(w[i], 1)), nzb), sa);
        x[2 * i + 1] = mul2(add2(make_float2(u8_biased(w[i], 2), u8_biased(w[i], 3)), nzb), sa);
    }
}

// Byte b of the word as the binary32 denormal byte * 2^-133 (the byte in bits 16..23,
// every other bit zero): an exact float that an FMA multiplies without rounding.
__device__ __forceinline__ float u8_denormal(uint32_t word, int b) {
    return __uint_as_float(prmt(word, 0u, 0x4044u | ((uint32_t)b << 8)));
}

// Dequantize 8 code words with one FMA per pair: x_j = q_j (s scale) - z (s scale),
// with scale94 = scale * 2^133 (the row's decay times 2^94 on the decode path, whose
// working scale is 2^-39).  The code enters as q_j 2^-133 (u8_denormal) and is
// multiplied by m = s * scale94 = (s scale) 2^133, so the product q_j (s scale) is
// exact inside the FMA; the constant c = (-z 2^-133) m = -z (s scale) is rounded once
// and so is the sum (within one unit in the last place of max(|x_j|, |z s scale|)).
// Needs m < 2^128: s * scale < 2^-5 (for the decode path, decays below 2^18).
__device__ __forceinline__ void dequantize_group_fma(const uint32_t (&w)[8], uint32_t sz, float scale94,
                                                     float2 (&x)[16]) {
    const float s = __half2float(__ushort_as_half((unsigned short)(sz & 0xffffu)));
    const float z = __half2float(__ushort_as_half((unsigned short)(sz >> 16)));
    const float m = s * scale94;
    const float2 m2 = splat2(m);
    const float2 c2 = splat2((z * -0x1p-133f) * m);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        x[2 * i] = fma2(make_float2(u8_denormal(w[i], 0), u8_denormal(w[i], 1)), m2, c2);
        x[2 * i + 1] = fma2(make_float2(u8_denormal(w[i], 2), u8_denormal(w[i], 3)), m2, c2);
    }
}

// In-thread H_32 on 16 pairs (component j of the group is y[j/2].x or .y).
__device__ __forceinline__ void hadamard_pairs(float2 (&y)[16]) {
    float x[32];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        x[2 * j] = y[j].x;
        x[2 * j + 1] = y[j].y;
    }
    hadamard_regs(x);
#pragma unroll
    for (int j = 0; j < 16; ++j) y[j] = make_float2(x[2 * j], x[2 * j + 1]);
}

__device__ __forceinline__ float2 h2_to_f2(uint32_t w) {
    __half2 h;
    memcpy(&h, &w, 4);
    return __half22float2(h);
}

// two floats -> packed binary16 pair, round to nearest even (low half = a)
__device__ __forceinline__ uint32_t f2_to_h2(float a, float b) {
    const __half2 h = __floats2half2_rn(a, b);
    uint32_t w;
    memcpy(&w, &h, 4);
    return w;
}

// Per-warp partial-sum buffer of column_sum2: 32 lane rows of 32 (r, p) pairs + padding.
constexpr int kPartStride = 68;  // floats per lane row

__device__ __forceinline__ float ldsf(uint32_t a) { return __uint_as_float(lds32(a)); }

// Column sums of two per-lane 32-vectors at once: lane j returns
// (sum_l a_l[j], sum_l b_l[j]) over the 32 lanes l.
__device__ __forceinline__ float2 column_sum2(const float2 (&a)[16], const float2 (&b)[16], uint32_t part, int lane) {
#pragma unroll
    for (int m = 0; m < 16; ++m) {  // row of lane l: (a_j, b_j) pairs in column order
        sts128(part + (lane * kPartStride + 4 * m) * 4,
               make_uint4(__float_as_uint(a[m].x), __float_as_uint(b[m].x), __float_as_uint(a[m].y),
                          __float_as_uint(b[m].y)));
    }
    __syncwarp();
    float2 s0 = make_float2(0.f, 0.f), s1 = s0, s2 = s0, s3 = s0;
#pragma unroll
    for (int l = 0; l < 32; l += 4) {
        const uint32_t base = part + (2 * lane) * 4;
        uint2 v0, v1, v2, v3;
        asm volatile("ld.shared.v2.b32 {%0,%1}, [%2];" : "=r"(v0.x), "=r"(v0.y) : "r"(base + (l + 0) * kPartStride * 4));
        asm volatile("ld.shared.v2.b32 {%0,%1}, [%2];" : "=r"(v1.x), "=r"(v1.y) : "r"(base + (l + 1) * kPartStride * 4));
        asm volatile("ld.shared.v2.b32 {%0,%1}, [%2];" : "=r"(v2.x), "=r"(v2.y) : "r"(base + (l + 2) * kPartStride * 4));
        asm volatile("ld.shared.v2.b32 {%0,%1}, [%2];" : "=r"(v3.x), "=r"(v3.y) : "r"(base + (l + 3) * kPartStride * 4));
        s0 = add2(s0, make_float2(__uint_as_float(v0.x), __uint_as_float(v0.y)));
        s1 = add2(s1, make_float2(__uint_as_float(v1.x), __uint_as_float(v1.y)));
        s2 = add2(s2, make_float2(__uint_as_float(v2.x), __uint_as_float(v2.y)));
        s3 = add2(s3, make_float2(__uint_as_float(v3.x), __uint_as_float(v3.y)));
    }
    __syncwarp();
    return add2(add2(s0, s1), add2(s2, s3));
}

__device__ __forceinline__ float bf16_at(uint32_t base, int i) {
    const uint32_t w = lds32(base + 2 * (i & ~1));
    return __uint_as_float((i & 1) ? (w & 0xffff0000u) : (w << 16));
}

__device__ __forceinline__ float load_in(const void *p, int64_t i, bool bf16) {
    if (bf16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(p)[i]);
    return reinterpret_cast<const float *>(p)[i];
}

}  // namespace damp
