// prefill_tc.cuh -- the GDN prefill chunk on the tensor cores (App. A.5 prefill path),
// in the chunkwise closed form of the delta rule (Sec. 3.1, Eq. delta_update).
//
// Within a piece of C = 64 tokens, with a_t = exp(g_t), the decay from token s to token
// t f_ts = a_{s+1} ... a_t (f_tt = 1), gamma_t = a_0 ... a_t and u_t the update column
// of token t (S_t = a_t S_{t-1} + k_t u_t^T), the per-token recurrence unrolls to
//     u_t + beta_t sum_{s<t} f_ts (k_t . k_s) u_s = beta_t (v_t - gamma_t S_0^T k_t)
//     o_t = gamma_t S_0^T q_t + sum_{s<=t} f_ts (q_t . k_s) u_s
//     S_C = gamma_C S_0 + sum_s f_Cs k_s u_s^T .
// With L = I + (beta_t f_ts k_t.k_s)_{s<t} (unit lower triangular),
// M = (f_ts q_t.k_s)_{s<=t} and Y = diag(beta) (V - diag(gamma) K S_0):
//     U = L^-1 Y,  O = diag(gamma) Q S_0 + M U,  S_C = gamma_C S_0 + K^T diag(f_C.) U.
// One CTA of eight warps owns a (slot, head) for the whole chunk; its state stays in
// tensor memory (FP32, lane = record row) from the reconstruction of the packed record
// to the requantization.  Per piece, four tcgen05.mma products (bf16 operands, FP32
// accumulation in tensor memory, M = 128):
//     [K; Q] S_0         -> W = K S_0 (lanes 0-63), P = Q S_0 (lanes 64-127)
//     [K; Q] K^T         -> K K^T, Q K^T
//     [0; M] U           -> accumulated onto gamma P: O (lanes 64-127)
//     K^T (f_C. U)       -> accumulated onto gamma_C S_0
// k and q are bf16 inputs (exact operands); the FP32 operands (S_0, M, U, f_C. U) enter
// as three bf16 parts x = hi + mid + lo (24 significant bits), and a product of two split
// operands takes the six partial products down to 2^-16 relative, so the products keep
// FP32 accuracy.  U = L^-1 Y is solved by forward substitution on the CUDA cores (one
// thread per value column, in blocks of 16 rows), as are the decay factors
// (running products and shuffle scans: no cancellation of cumulative log sums) and the
// requantization.  With the H_32 formats the whole chunk runs in the transformed domain
// (S~ = S H, v~ = v H, o = o~ H per value block of 32), as the other prefill kernels do.
#pragma once

#include <cuda_bf16.h>

#include "prefill.cuh"

namespace damp {

constexpr int kTcC = 64;          // tokens per piece
constexpr int kTcThreads = 256;   // two threads per tensor-memory lane (warps w and w + 4)
constexpr uint32_t kTcCols = 512; // tensor-memory columns of the CTA (one CTA per SM)
// tensor-memory columns of the accumulators: W | P then O (lanes 64-127), S, K K^T | Q K^T
constexpr uint32_t kColWP = 0, kColS = 128, kColG = 256;
// Shared memory (bytes from the base of the dynamic shared memory).  Each area is live
// from the step that writes it to the step that last reads it; areas that share bytes
// are never live together:
//   staging:        A1 [0, 32K)  B1 [32K, 128K)  records (unit start) [128K, 160K)  V [160K, 177K)
//   after [K;Q]S_0: A3 [16K, 32K)  AO [32K, 80K)  LP [80K, 97K)  YU [97K, 130K)
//   after the solve: BU [80K, 128K)  B4 [128K, 176K)
constexpr int kSmA1 = 0;        // [K; Q] bf16, K-major: 128 rows x 128 channels (K rows stay for A3)
constexpr int kSmB1 = 32768;    // S_0 as three bf16 parts, MN-major (value columns x channels)
constexpr int kSmRec = 131072;  // the four value-block records of the (slot, head)
constexpr int kSmV = 163840;    // v of the piece, bf16, 64 rows of 272 bytes
constexpr int kSmA3 = 16384;    // K^T in record-row order, bf16, MN-major (16 KB)
constexpr int kSmAO = 32768;    // [0; M] three bf16 parts, K-major (128 rows x 64 tokens, 3 x 16 KB)
constexpr int kSmLP = 81920;    // L'^T (L' = L - I strictly lower), 64 rows of 68 FP32
constexpr int kSmYU = 99328;    // Y, then U in place: 64 rows of 132 FP32
constexpr int kSmBU = 81920;    // U as three bf16 parts, K-major (value columns x tokens, 3 x 16 KB)
constexpr int kSmB4 = 131072;   // f_C. U as three bf16 parts, K-major (3 x 16 KB)
constexpr int kSmScal = 181248; // a, beta, gamma, f_C. (64 floats each), pi, g, two mbarriers, tensor-memory address
constexpr int kTcRowL = 68;     // floats per row of L'^T
constexpr int kTcRowY = 132;    // floats per row of Y / U
constexpr int kTcRowV = 272;    // bytes per row of v
constexpr int kTcSmem = kSmScal + 1472;
constexpr int kTcMaxRec = 8192; // largest record (d_k = 128): four fit in [kSmRec, kSmV)
__host__ __device__ constexpr int tc_rec_stride(int rec_bytes) { return (rec_bytes + 127) & ~127; }

// ---- tcgen05 / tensor-memory primitives (inline PTX) ----
__device__ __forceinline__ uint64_t tc_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
    // shared-memory matrix descriptor: start >> 4, leading (K-direction) and stride
    // (M/N-direction) byte offsets >> 4, version 1, no swizzle
    return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46);
}
// instruction descriptor: bf16 x bf16 -> FP32, M = 128, N, A/B MN-major when set
__host__ __device__ constexpr uint32_t tc_idesc(int n, bool a_mn, bool b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (a_mn ? 1u << 15 : 0u) | (b_mn ? 1u << 16 : 0u) |
           ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}
__device__ __forceinline__ void tc_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.u32 p, %4, 0;\n"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d),
                 "l"(a), "l"(b), "r"(idesc), "r"(acc)
                 : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// 32 consecutive columns of this thread's lane (warp w reaches lanes 32 (w % 4) .. + 31)
__device__ __forceinline__ void tc_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
                 "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
                 "tcgen05.wait::ld.sync.aligned;"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
                   "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
                   "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
                   "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
                   "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                 : "r"(taddr)
                 : "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tc_st32(uint32_t taddr, const float (&v)[32]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
                 "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n"
                 "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
                 "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
                 "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
                 "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
                 "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
                 "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
                 "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
                 "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
                 "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
                 "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
                 "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
                 "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
                 : "memory");
}

// x = hi + mid + lo as bf16 parts (each the round-to-nearest of what is left), two
// values per 32-bit word (a in the low half)
__device__ __forceinline__ void split3_pair(float a, float b, uint32_t &h, uint32_t &m, uint32_t &l) {
    const __nv_bfloat162 h2 = __floats2bfloat162_rn(a, b);
    const float2 hf = __bfloat1622float2(h2);
    const float ra = a - hf.x, rb = b - hf.y;  // exact
    const __nv_bfloat162 m2 = __floats2bfloat162_rn(ra, rb);
    const float2 mf = __bfloat1622float2(m2);
    const __nv_bfloat162 l2 = __floats2bfloat162_rn(ra - mf.x, rb - mf.y);
    memcpy(&h, &h2, 4);
    memcpy(&m, &m2, 4);
    memcpy(&l, &l2, 4);
}
// eight consecutive MN-elements of an operand as three 16-byte parts
__device__ __forceinline__ void split3_store8(uint32_t dst, uint32_t part_bytes, const float *x) {
    uint32_t h[4], m[4], l[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) split3_pair(x[2 * i], x[2 * i + 1], h[i], m[i], l[i]);
    sts128(dst, make_uint4(h[0], h[1], h[2], h[3]));
    sts128(dst + part_bytes, make_uint4(m[0], m[1], m[2], m[3]));
    sts128(dst + 2 * part_bytes, make_uint4(l[0], l[1], l[2], l[3]));
}
// byte offset of element (mn, k) in an MN-major bf16 operand whose 8-element groups
// along MN are 128 B apart and whose 8-row groups along K are kstride apart
__device__ __forceinline__ uint32_t tc_mn_off(int mn, int k, uint32_t kstride) {
    return (uint32_t)(mn >> 3) * 128u + (uint32_t)(k >> 3) * kstride + (uint32_t)(k & 7) * 16u + (uint32_t)(mn & 7) * 2u;
}

__device__ __forceinline__ uint32_t lds_u16(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
// all threads of the CTA wait for the phase (bounded) and agree on the outcome
__device__ __forceinline__ bool tc_wait_all(uint32_t bar, uint32_t parity) {
    return __syncthreads_and(mbar_wait_bounded(bar, parity)) != 0;
}
// the 32 values of v as 16 pairs
__device__ __forceinline__ void tc_pairs(const float (&v)[32], float2 (&y)[16]) {
#pragma unroll
    for (int i = 0; i < 16; ++i) y[i] = make_float2(v[2 * i], v[2 * i + 1]);
}

constexpr uint32_t kIdWP = tc_idesc(128, false, true);  // [K; Q] K-major, S_0 MN-major
constexpr uint32_t kIdG = tc_idesc(64, false, false);   // [K; Q] and K, both K-major
constexpr uint32_t kIdO = tc_idesc(128, false, false);  // [0; M] and U, both K-major
constexpr uint32_t kIdS = tc_idesc(128, true, false);   // K^T MN-major, f_C. U K-major
// byte offset of element (row, k) in a K-major bf16 operand of 8-row groups 1024 B apart
// (64 columns of K: eight 16-byte core matrices per group)
__device__ __forceinline__ uint32_t tc_k64_off(int row, int k) {
    return (uint32_t)(row >> 3) * 1024u + (uint32_t)(k >> 3) * 128u + (uint32_t)(row & 7) * 16u + (uint32_t)(k & 7) * 2u;
}

// The record rows of a (slot, head) (four value-block records at `recs`, `rstride` apart
// in shared memory) reconstructed into tensor-memory lane u = record row, the value blocks
// of part `part` of NQ (4 / NQ blocks each): FP32 at the natural scale, FP16 rows taken
// into the H_32 domain with the H_32 formats (where the low tier's codes already are).
template <int FMT, int NQ>
__device__ __forceinline__ void tc_reconstruct(const PrefillParams &p, uint32_t recs, int rstride, int u, int part,
                                               uint32_t tS) {
    constexpr bool HAD = fmt_had(FMT);
    const int K = p.K, lo = 128 - K;
#pragma unroll 1
    for (int c = part * (4 / NQ); c < (part + 1) * (4 / NQ); ++c) {
        const uint32_t rec = recs + (uint32_t)(c * rstride);
        float2 y[16];
        if (u < K) {
            load_hi_row(rec, u, y);
            if (HAD) hadamard_pairs(y);
        } else {
            const int r = u - K;
            const uint4 c0 = lds128(rec + (uint32_t)(p.codes_off + lo_chunk_off(r, 0, lo)));
            const uint32_t sz = lds32(rec + (uint32_t)(p.meta_off + 4 * r));
            if constexpr (fmt_u4(FMT)) {
                const uint32_t w[4] = {c0.x, c0.y, c0.z, c0.w};
                dequantize_group_u4(w, sz, 1.0f, y);
            } else {
                const uint4 c1 = lds128(rec + (uint32_t)(p.codes_off + lo_chunk_off(r, 1, lo)));
                const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                if constexpr (FMT == kFmtE4M3) dequantize_group_e4m3(w, __uint_as_float(sz), 1.0f, y);
                else dequantize_group(w, sz, 1.0f, y);
            }
        }
        float v[32];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            v[2 * i] = y[i].x;
            v[2 * i + 1] = y[i].y;
        }
        tc_st32(tS + 32 * c, v);
    }
}

// U = L^-1 Y by forward substitution for one value column, in place: col addresses row 0 of
// the column (rows kTcRowY floats apart), lt the rows of L'^T (L' = L - I, kTcRowL floats
// apart).  Blocks of 16 rows, 16 / NQ per part of the NQ threads that own the column: the
// rows of a block take the solved rows of the earlier blocks (each loaded once for 16 / NQ
// independent sums), then the parts solve their rows in turn, each first taking the rows
// solved before it out of its own.  Every thread of the CTA calls it (NQ barriers per block).
template <int NQ>
__device__ __forceinline__ void tc_solve(uint32_t col, uint32_t lt, int part) {
    constexpr int RB = 16 / NQ;  // rows per part and block (4 or 8), held as RB / 2 pairs
    constexpr int RP = RB / 2;
    auto ltr = [&](int srow, int t0, float2 (&lv)[RP]) {
        const uint32_t lrow = lt + (uint32_t)(srow * kTcRowL * 4 + 4 * t0);
#pragma unroll
        for (int i = 0; i < RB / 4; ++i) {
            const uint4 l4 = lds128(lrow + 16 * i);
            lv[2 * i] = make_float2(__uint_as_float(l4.x), __uint_as_float(l4.y));
            lv[2 * i + 1] = make_float2(__uint_as_float(l4.z), __uint_as_float(l4.w));
        }
    };
    auto row_at = [&](int r) { return col + (uint32_t)(r * kTcRowY * 4); };
#pragma unroll 1
    for (int t0 = 0; t0 < kTcC; t0 += 16) {
        const int r0 = t0 + RB * part;
        float2 acc[RP];
#pragma unroll
        for (int i = 0; i < RP; ++i) acc[i] = make_float2(ldsf(row_at(r0 + 2 * i)), ldsf(row_at(r0 + 2 * i + 1)));
#pragma unroll 4
        for (int s2 = 0; s2 < t0; ++s2) {
            const float us = ldsf(row_at(s2));
            float2 lv[RP];
            ltr(s2, r0, lv);
#pragma unroll
            for (int i = 0; i < RP; ++i) acc[i] = fma2(lv[i], make_float2(-us, -us), acc[i]);
        }
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            if (part == q) {  // own rows among themselves (the pair holding the solved row takes
                              // zero entries of L'^T, which leave it as it is), then stored
#pragma unroll
                for (int a = 0; a < RB - 1; ++a) {
                    const float ua = (a & 1) ? acc[a >> 1].y : acc[a >> 1].x;
                    float2 lv[RP];
                    ltr(r0 + a, r0, lv);
#pragma unroll
                    for (int i = a >> 1; i < RP; ++i) acc[i] = fma2(lv[i], make_float2(-ua, -ua), acc[i]);
                }
#pragma unroll
                for (int i = 0; i < RP; ++i) {
                    sts32(row_at(r0 + 2 * i), __float_as_uint(acc[i].x));
                    sts32(row_at(r0 + 2 * i + 1), __float_as_uint(acc[i].y));
                }
            }
            __syncthreads();
            if (part > q) {  // the rows part q just solved
#pragma unroll
                for (int a = 0; a < RB; ++a) {
                    const int sr = t0 + RB * q + a;
                    const float us = ldsf(row_at(sr));
                    float2 lv[RP];
                    ltr(sr, r0, lv);
#pragma unroll
                    for (int i = 0; i < RP; ++i) acc[i] = fma2(lv[i], make_float2(-us, -us), acc[i]);
                }
            }
        }
    }
}

// The chunk-final state (tensor-memory lane u = record row u, the value blocks of part
// `part` of NQ) into the records at grec0 in place: FP16 rows back to the natural domain
// and rounded once, low-tier rows requantized (the affine formats at the working scale
// 2^-39, FP8 in the natural domain).  Warps holding FP16 rows store them warp-collectively.
template <int FMT, int NQ>
__device__ __forceinline__ void tc_requantize(const PrefillParams &p, uint8_t *grec0, int u, int part, int lane,
                                              uint32_t tS) {
    constexpr bool HAD = fmt_had(FMT);
    const int K = p.K, lo = 128 - K;
#pragma unroll 1
    for (int c = part * (4 / NQ); c < (part + 1) * (4 / NQ); ++c) {
        float v[32];
        tc_ld32(tS + 32 * c, v);
        uint8_t *const grec = grec0 + (int64_t)c * p.rec_bytes;
        float2 y[16];
        tc_pairs(v, y);
        if ((u & ~31) < K) {  // the warp holds FP16 rows: the row-pair store is warp-collective
            float2 z[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) z[i] = y[i];
            if (HAD) hadamard_pairs(z);
            uint32_t own[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) own[i] = f2_to_h2(z[i].x, z[i].y);
            store_hi_row(grec, u, K, lane, own);
        }
        if (u >= K) {
            const int r = u - K;
            if constexpr (FMT == kFmtE4M3) {  // natural domain, one FP32 scale per group
                uint32_t w[8];
                const float sc = quantize_group_e4m3(y, w);
                stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                stg32(grec + p.meta_off + 4 * r, __float_as_uint(sc));
            } else {
#pragma unroll
                for (int i = 0; i < 16; ++i) y[i] = mul2(y[i], splat2(kDown));  // exact
                if constexpr (fmt_u4(FMT)) {
                    uint32_t w[4];
                    const uint32_t szw = quantize_group_u4(y, w);
                    stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                    stg32(grec + p.meta_off + 4 * r, szw);
                } else {
                    float mn, mx, inv, zq;
                    minmax32(y, mn, mx);
                    const float sc = scale_of(mn, mx);
                    const uint32_t szw =
                        sc == 0.0f ? affine_params_scaled(mn, mx, inv, zq) : affine_finish(sc, mn, inv, zq);
                    const float2 inv2 = splat2(inv * 0x1p-110f), zc2 = splat2(zq * 0x1p-149f);
                    uint32_t w[8];
#pragma unroll
                    for (int m = 0; m < 8; ++m) w[m] = encode4(y[2 * m], y[2 * m + 1], inv2, zc2);
                    stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                    stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                    stg32(grec + p.meta_off + 4 * r, szw);
                }
            }
        }
    }
}

// One CTA of kTcThreads threads per (slot, head) unit at a time (persistent over units);
// d_k = d_v = 128, bf16 q/k/v, low tier FMT (UINT8 or UINT4 affine, with or without H_32;
// the launchers also instantiate no FP8 or row-absmax kernel).  Thread (row, half):
// row = tensor-memory lane (warps w and w + 4 reach the same lanes), half = 0 / 1 splits
// a row's value blocks (0-1 / 2-3) or a phase's tasks between the two.
template <int FMT>
__global__ void __launch_bounds__(kTcThreads, 1) prefill_tc_gdn_kernel(const PrefillParams p) {
    static_assert(FMT != kFmtS8Row, "the row-absmax format shares a row scale over the value blocks");
    constexpr bool HAD = fmt_had(FMT);
    extern __shared__ __align__(128) uint8_t smem[];  // descriptors need 16-byte alignment (no swizzle)
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int row = tid & 127, half = tid >> 7;
    const uint32_t sb = smem_u32(smem);
    const int H = p.H, T = p.T, Hm = p.Hm;
    const int rec_bytes = p.rec_bytes, rstride = tc_rec_stride(rec_bytes);
    const uint32_t scal = sb + (uint32_t)kSmScal;
    const uint32_t s_a = scal, s_beta = scal + 256, s_gam = scal + 512, s_rev = scal + 768, s_perm = scal + 1024;
    const uint32_t s_g = scal + 1152, bar_rec = scal + 1408, bar_mma = scal + 1416, s_taddr = scal + 1424;

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(s_taddr), "r"(kTcCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (tid == 0) {
        mbar_init(bar_rec, 1);
        mbar_init(bar_mma, 1);
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = lds32(s_taddr);
    const uint32_t tl = tmem + ((uint32_t)(32 * (warp & 3)) << 16);  // this warp's lanes
    const uint32_t tWP = tl + kColWP, tS = tl + kColS, tG = tl + kColG;

    uint32_t ph_rec = 0, ph_mma = 0;
    bool bad_slot = false, bad_head = false, timed_out = false;
    bool rec_pending = false, mma_pending = false;  // a copy / a product in flight
    const int64_t units = (int64_t)p.batch * H;
    // a (slot, head) unit that has work: its batch row, held and model head, slot and length
    struct Unit {
        int64_t unit, slot;
        int b, h, mh, hq, Tb;
    };
    // the first unit at or after u (stepping by the grid) with work; unit == units if none
    // (units without work are skipped here, once each, with their status bits)
    auto next_unit = [&](int64_t u) -> Unit {
        Unit n{units, 0, 0, 0, 0, 0, 0};
        for (; u < units; u += gridDim.x) {
            const int b = (int)(u / H), h = (int)(u - (int64_t)b * H);
            const int mh = p.head_map ? p.head_map[h] : h;
            const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
            const int Tb = p.lengths ? min(max(p.lengths[b], 0), T) : T;
            const bool slot_ok = slot >= 0 && slot < p.num_slots, head_ok = mh >= 0 && mh < Hm;
            bad_slot |= !slot_ok;
            bad_head |= !head_ok;
            if (slot_ok && head_ok && Tb > 0) {
                n = Unit{u, slot, b, h, mh, (int)(((int64_t)mh * p.Hqk) / Hm), Tb};
                break;
            }
        }
        return n;
    };
    auto rec_of = [&](const Unit &n) { return p.state + n.slot * p.slot_bytes + (int64_t)(n.h * 4) * rec_bytes; };
    // [K; Q] (bf16, natural channel order, K-major), v, g and beta of unit n's piece at p0
    // (cp.async; a masked token is zero, neither decays nor updates)
    auto load_piece = [&](const Unit &n, int p0) {
        const int nt = min(kTcC, n.Tb - p0);
#pragma unroll 1
        for (int i = tid; i < 2048; i += kTcThreads) {
            const int m = i >> 4, j = i & 15, t = m & 63;
            const uint32_t dst = sb + (uint32_t)(kSmA1 + (m >> 3) * 2048 + j * 128 + (m & 7) * 16);
            if (t < nt) {
                const uint8_t *src = static_cast<const uint8_t *>(m < 64 ? p.k : p.q) +
                                     (((int64_t)n.b * T + p0 + t) * p.Hqk + n.hq) * 256 + 16 * j;
                cp_async16(dst, src);
            } else {
                sts128(dst, make_uint4(0u, 0u, 0u, 0u));
            }
        }
#pragma unroll 1
        for (int i = tid; i < 1024; i += kTcThreads) {
            const int t = i >> 4, j = i & 15;
            const uint32_t dst = sb + (uint32_t)(kSmV + t * kTcRowV + 16 * j);
            if (t < nt)
                cp_async16(dst, static_cast<const uint8_t *>(p.v) + (((int64_t)n.b * T + p0 + t) * Hm + n.mh) * 256 + 16 * j);
            else
                sts128(dst, make_uint4(0u, 0u, 0u, 0u));
        }
        if (tid < kTcC) {  // log-decay and beta (a masked token: g = 0, beta = 0)
            const int t = tid;
            if (t < nt) {
                const int64_t gi = ((int64_t)n.b * T + p0 + t) * Hm + n.mh;
                cp_async4(s_g + 4 * t, p.g + gi);
                cp_async4(s_beta + 4 * t, p.beta + gi);
            } else {
                sts32(s_g + 4 * t, 0u);
                sts32(s_beta + 4 * t, 0u);
            }
        }
        cp_async_commit();
    };
    // unit n's four records (bulk copies), pi and first piece: issued one unit ahead, so
    // that they land while the previous unit finishes (every area they write is free then)
    auto prefetch = [&](const Unit &n) {
        if (tid == 0) {
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(bar_rec, (uint32_t)(4 * rec_bytes));
            uint8_t *const g0 = rec_of(n);
#pragma unroll
            for (int c = 0; c < 4; ++c)
                bulk_g2s(sb + (uint32_t)(kSmRec + c * rstride), g0 + (int64_t)c * rec_bytes, (uint32_t)rec_bytes, bar_rec);
        }
        if (tid < 8) cp_async16(s_perm + 16 * tid, p.perm + (int64_t)n.h * 128 + 16 * tid);
        load_piece(n, 0);  // commits the perm copies with the piece's
        rec_pending = true;
    };

    Unit cur = next_unit(blockIdx.x);
    if (cur.unit < units) prefetch(cur);
    while (cur.unit < units) {
        const int b = cur.b, Tb = cur.Tb, mh = cur.mh;
        uint8_t *const grec0 = rec_of(cur);
        const Unit nxt = next_unit(cur.unit + gridDim.x);  // its loads overlap this unit's work
        if (!tc_wait_all(bar_rec, ph_rec)) {
            timed_out = true;
            break;
        }
        ph_rec ^= 1u;
        rec_pending = false;

        // ---- S_0: record row u = row, reconstructed (FP32, natural scale, transformed domain
        //      with H_32) into tensor-memory lane u; this half's two value blocks ----
        tc_reconstruct<FMT, 2>(p, sb + (uint32_t)kSmRec, rstride, row, half, tS);

#pragma unroll 1
        for (int p0 = 0; p0 < Tb; p0 += kTcC) {
            const int nt = min(kTcC, Tb - p0);  // live tokens of the piece; the rest are masked
            if (p0 > 0) {
                load_piece(cur, p0);
            } else {  // the first piece's copies (and pi) were issued with the records
                cp_async_wait_all();
                __syncthreads();
            }
            // ---- S_0 as three bf16 parts, MN-major (value columns n x channels), at channel pi(u) ----
            {
                const int ch = (int)(lds_u8(s_perm + row) & 127u);
#pragma unroll 1
                for (int c = 2 * half; c < 2 * half + 2; ++c) {
                    float v[32];
                    tc_ld32(tS + 32 * c, v);
#pragma unroll
                    for (int j8 = 0; j8 < 4; ++j8)
                        split3_store8(sb + kSmB1 + tc_mn_off(32 * c + 8 * j8, ch, 2048), 32768, v + 8 * j8);
                }
            }
            cp_async_wait_all();
            fence_proxy_async_smem();  // the operands written through the generic proxy, before the MMAs
            tc_fence_before();
            __syncthreads();
            tc_fence_after();
            if (tid == 0) {
#pragma unroll 1
                for (int q = 0; q < 3; ++q)
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        tc_mma(tmem + kColWP, tc_desc(sb + kSmA1 + 256 * ks, 128, 2048),
                               tc_desc(sb + kSmB1 + 32768 * q + 4096 * ks, 2048, 128), kIdWP, (q | ks) != 0);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    tc_mma(tmem + kColG, tc_desc(sb + kSmA1 + 256 * ks, 128, 2048),
                           tc_desc(sb + kSmA1 + 256 * ks, 128, 2048), kIdG, ks != 0);
                tc_commit(bar_mma);
            }
            // gamma_t = a_0 ... a_t and f_Ct = a_{t+1} ... a_63 (warp 0: lane l holds tokens
            // 2l and 2l + 1; products over the lanes by shuffle scans) while the products run
            if (warp == 0) {
                const float a0 = expf(ldsf(s_g + 8 * lane)), a1 = expf(ldsf(s_g + 8 * lane + 4));
                sts32(s_a + 8 * lane, __float_as_uint(a0));
                sts32(s_a + 8 * lane + 4, __float_as_uint(a1));
                const float tot = a0 * a1;
                float pre = tot, suf = tot;  // inclusive over lanes <= l / >= l
#pragma unroll
                for (int d = 1; d < 32; d <<= 1) {
                    const float up = __shfl_up_sync(kFull, pre, d), dn = __shfl_down_sync(kFull, suf, d);
                    if (lane >= d) pre *= up;
                    if (lane + d < 32) suf *= dn;
                }
                float ex_pre = __shfl_up_sync(kFull, pre, 1), ex_suf = __shfl_down_sync(kFull, suf, 1);
                if (lane == 0) ex_pre = 1.f;
                if (lane == 31) ex_suf = 1.f;
                sts32(s_gam + 8 * lane, __float_as_uint(ex_pre * a0));
                sts32(s_gam + 8 * lane + 4, __float_as_uint(ex_pre * tot));
                sts32(s_rev + 8 * lane, __float_as_uint(a1 * ex_suf));
                sts32(s_rev + 8 * lane + 4, __float_as_uint(ex_suf));
            }
            if (!tc_wait_all(bar_mma, ph_mma)) {
                timed_out = mma_pending = true;
                break;
            }
            ph_mma ^= 1u;
            tc_fence_after();
            // ---- half 0: rows of L' = beta_t f_ts k_t.k_s (s < t; FP32, for the solve) and of
            //      M = f_ts q_t.k_s (s <= t; rows 64 + t of [0; M], three bf16 parts), and
            //      gamma_t P_t in tensor memory;  half 1: K^T in record-row order, the zero
            //      rows of [0; M] and gamma_C S_0 in tensor memory ----
            if (half == 0) {
                const int t = row & 63;
                const bool qside = row >= 64;
                float gr[64];
                {
                    float g0[32], g1[32];
                    tc_ld32(tG, g0);
                    tc_ld32(tG + 32, g1);
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        gr[i] = g0[i];
                        gr[32 + i] = g1[i];
                    }
                }
                const float bt = qside ? 1.f : ldsf(s_beta + 4 * t);
                float f = 1.f;  // f_ts, s running down from t
#pragma unroll
                for (int s2 = 63; s2 >= 0; --s2) {
                    float e = 0.f;
                    if (s2 < t) {
                        f *= ldsf(s_a + 4 * (s2 + 1));
                        e = bt * f * gr[s2];
                    } else if (s2 == t && qside) {
                        e = gr[s2];
                    }
                    gr[s2] = e;
                }
                if (!qside) {  // column t of L'^T (row s holds L'_{., s})
                    const uint32_t colt = sb + (uint32_t)(kSmLP + 4 * t);
#pragma unroll
                    for (int s2 = 0; s2 < 64; ++s2) sts32(colt + (uint32_t)(s2 * kTcRowL * 4), __float_as_uint(gr[s2]));
                } else {
#pragma unroll
                    for (int g = 0; g < 8; ++g) split3_store8(sb + kSmAO + tc_k64_off(64 + t, 8 * g), 16384, gr + 8 * g);
                    // gamma_t P_t: the output product accumulates onto it
                    const float gt = ldsf(s_gam + 4 * t);
#pragma unroll 1
                    for (int c = 0; c < 4; ++c) {
                        float v[32];
                        tc_ld32(tWP + 32 * c, v);
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] *= gt;
                        tc_st32(tWP + 32 * c, v);
                    }
                }
            } else {
                // rows 0 .. 63 of [0; M] are zero
#pragma unroll 1
                for (int i = row; i < 1536; i += 128)
                    sts128(sb + (uint32_t)(kSmAO + (i >> 9) * 16384 + (i & 511) * 16), make_uint4(0u, 0u, 0u, 0u));
                // K^T: element (u, s) = k_s[pi(u)]; this thread takes token s = row & 63 and
                // half the rows (its 64 channel indices first, then independent gathers)
                {
                    const int t = row & 63;
                    const uint32_t krow = sb + (uint32_t)(kSmA1 + (t >> 3) * 2048 + (t & 7) * 16);
                    const int u0 = row >= 64 ? 64 : 0;
                    uint32_t pw[16];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const uint4 w4 = lds128(s_perm + (uint32_t)(u0 + 16 * i));
                        pw[4 * i] = w4.x;
                        pw[4 * i + 1] = w4.y;
                        pw[4 * i + 2] = w4.z;
                        pw[4 * i + 3] = w4.w;
                    }
#pragma unroll
                    for (int uc = 0; uc < 8; ++uc) {
                        uint32_t w[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const uint32_t pp = pw[2 * uc + (e >> 1)] >> (16 * (e & 1));  // channels of rows ua, ua + 1
                            const uint32_t ca = pp & 127u, cb = (pp >> 8) & 127u;
                            const uint32_t va = lds_u16(krow + (ca >> 3) * 128u + (ca & 7u) * 2u);
                            const uint32_t vb = lds_u16(krow + (cb >> 3) * 128u + (cb & 7u) * 2u);
                            w[e] = va | (vb << 16);
                        }
                        sts128(sb + kSmA3 + tc_mn_off(u0 + 8 * uc, t, 2048), make_uint4(w[0], w[1], w[2], w[3]));
                    }
                }
                // gamma_C S_0: the state product accumulates onto it
                const float gC = ldsf(s_gam + 4 * (kTcC - 1));
#pragma unroll 1
                for (int c = 0; c < 4; ++c) {
                    float v[32];
                    tc_ld32(tS + 32 * c, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] *= gC;
                    tc_st32(tS + 32 * c, v);
                }
            }
            // ---- Y = diag(beta) (v~ - diag(gamma) W), FP32 rows (this half's value blocks) ----
            if (row < 64) {
                const int t = row;
                const float bt = ldsf(s_beta + 4 * t), gt = ldsf(s_gam + 4 * t);
                const uint32_t vrow = sb + (uint32_t)(kSmV + t * kTcRowV), yrow = sb + (uint32_t)(kSmYU + t * kTcRowY * 4);
#pragma unroll 1
                for (int c = 2 * half; c < 2 * half + 2; ++c) {
                    float w[32];
                    tc_ld32(tWP + 32 * c, w);
                    float2 y[16];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint4 r = lds128(vrow + 64 * c + 16 * q);
                        const uint32_t rw[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            y[4 * q + e] = make_float2(__uint_as_float(rw[e] << 16), __uint_as_float(rw[e] & 0xffff0000u));
                    }
                    if (HAD) hadamard_pairs(y);
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const float2 ya = y[2 * q], yb = y[2 * q + 1];
                        sts128(yrow + 128 * c + 16 * q,
                               make_uint4(__float_as_uint(bt * (ya.x - gt * w[4 * q])), __float_as_uint(bt * (ya.y - gt * w[4 * q + 1])),
                                          __float_as_uint(bt * (yb.x - gt * w[4 * q + 2])),
                                          __float_as_uint(bt * (yb.y - gt * w[4 * q + 3]))));
                    }
                }
            }
            __syncthreads();
            // ---- U = L^-1 Y by forward substitution (value column n = row, in place) ----
            tc_solve<2>(sb + (uint32_t)(kSmYU + 4 * row), sb + (uint32_t)kSmLP, half);
            // ---- U (half 0) and f_C. U (half 1) as three bf16 parts, K-major (value columns n x
            //      tokens s) ----
            {
                const uint32_t col = sb + (uint32_t)(kSmYU + 4 * row);
                float uc[64];
#pragma unroll
                for (int t = 0; t < 64; ++t) uc[t] = ldsf(col + (uint32_t)(t * kTcRowY * 4));
                __syncthreads();  // every column is read: the parts go over L' and Y / U
                const uint32_t dst = sb + (uint32_t)(half == 0 ? kSmBU : kSmB4);
#pragma unroll
                for (int g = 0; g < 8; ++g) {
                    float x8[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) x8[e] = half == 0 ? uc[8 * g + e] : ldsf(s_rev + 4 * (8 * g + e)) * uc[8 * g + e];
                    split3_store8(dst + tc_k64_off(row, 8 * g), 16384, x8);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncthreads();
            tc_fence_after();
            if (tid == 0) {
                // O = gamma P + [0; M] U and S += K^T (f_C. U); six partial products of two
                // split operands (hh, hm, mh, hl, lh, mm), three of an exact one
                constexpr int pa[6] = {0, 0, 1, 0, 2, 1}, pb[6] = {0, 1, 0, 2, 0, 1};
#pragma unroll
                for (int q = 0; q < 6; ++q)
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        tc_mma(tmem + kColWP, tc_desc(sb + kSmAO + 16384 * pa[q] + 256 * ks, 128, 1024),
                               tc_desc(sb + kSmBU + 16384 * pb[q] + 256 * ks, 128, 1024), kIdO, 1u);
#pragma unroll
                for (int q = 0; q < 3; ++q)
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        tc_mma(tmem + kColS, tc_desc(sb + kSmA3 + 4096 * ks, 2048, 128),
                               tc_desc(sb + kSmB4 + 16384 * q + 256 * ks, 128, 1024), kIdS, 1u);
                tc_commit(bar_mma);
            }
            if (!tc_wait_all(bar_mma, ph_mma)) {
                timed_out = mma_pending = true;
                break;
            }
            ph_mma ^= 1u;
            tc_fence_after();
            if (p0 + kTcC >= Tb && nxt.unit < units) prefetch(nxt);  // the next unit's loads overlap this one's tail
            // ---- o_t = H (gamma_t P_t + (M U)_t) (lanes 64 + t, this half's value blocks) ----
            if (row >= 64) {
                const int t = row - 64;
                float *orow = p.o + (((int64_t)b * T + p0 + min(t, nt - 1)) * Hm + mh) * 128;
#pragma unroll 1
                for (int c = 2 * half; c < 2 * half + 2; ++c) {
                    float ov[32];
                    tc_ld32(tWP + 32 * c, ov);
                    float2 y[16];
                    tc_pairs(ov, y);
                    if (HAD) hadamard_pairs(y);
                    if (t < nt) {
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            stg128(orow + 32 * c + 4 * q,
                                   make_uint4(__float_as_uint(y[2 * q].x), __float_as_uint(y[2 * q].y),
                                              __float_as_uint(y[2 * q + 1].x), __float_as_uint(y[2 * q + 1].y)));
                    }
                }
            }
        }
        if (timed_out) break;
        // ---- the chunk-final state (tensor-memory lane u = record row u, this half's value
        //      blocks) into the record in place ----
        tc_requantize<FMT, 2>(p, grec0, row, half, lane, tS);
        cur = nxt;
    }
    // a copy or a product that did not complete in time gets one more bounded wait before
    // the tensor memory and the shared memory go away
    if (rec_pending) mbar_wait_bounded(bar_rec, ph_rec);
    if (mma_pending) mbar_wait_bounded(bar_mma, ph_mma);
    cp_async_wait_all();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcCols) : "memory");
    }
    if (tid == 0) {
        const uint32_t bits =
            (timed_out ? kDevWaitTimeout : 0u) | (bad_slot ? kDevBadSlot : 0u) | (bad_head ? kDevBadHead : 0u);
        if (bits) atomicOr(p.status, bits);
    }
}

}  // namespace damp
