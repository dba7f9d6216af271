// convert.cu -- kernels that move whole states in and out of the packed cache.
//
//   quantize_state    natural FP32 state -> packed records (App. A.5 "Prefill
//                     path": the FP32 state is written straight into the packed
//                     cache; rows in pi order, FP16 tier for rows < K_hi, H_32 +
//                     UINT8 affine (Sec. 3.2, Eq. integer_quantizer) for the rest)
//   dequantize_state  packed records -> natural FP32 state (the inverse map)
//   pack_tiers / unpack_tiers
//                     logical tier arrays (S_hi, Q_lo, M_lo of Eq.
//                     packed_state_layout) <-> packed records, bit for bit
//
// One warp per (slot, head, value block) record; lane l owns packed rows
// l, l+32, ...; global memory is accessed directly (these kernels are off the
// per-step path).
#include "damp_common.cuh"
#include "damp_internal.h"
#include "formats.cuh"

#include <algorithm>

namespace damp {

static __device__ uint32_t g_status_convert;

struct ConvParams {
    uint8_t *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    const uint8_t *perm;
    float *S;
    uint16_t *hi;
    uint8_t *codes;
    uint16_t *meta;
    int32_t batch, H, dk, dv, V, K;
    int32_t Hm;                // heads of S: held head h is row head_map[h] (or h)
    const int32_t *head_map;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes, total_tiles;
    uint32_t *status;
};

enum ConvOp { kQuantize = 0, kDequantize = 1, kPackTiers = 2, kUnpackTiers = 3 };

template <int R, int FMT, int OP>
__global__ void __launch_bounds__(256) convert_kernel(const ConvParams p) {
    constexpr bool HAD = fmt_had(FMT);
    constexpr bool U4 = fmt_u4(FMT);
    constexpr int CB = U4 ? 16 : 32;  // code bytes per row and value block
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwt = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int K = p.K;
    const int lo = p.dk - K;
    bool bad_slot = false, bad_head = false;
    for (int64_t t = gw; t < p.total_tiles; t += nwt) {
        const int c = (int)(t % p.V);
        const int64_t bh = t / p.V;
        const int h = (int)(bh % p.H);
        const int b = (int)(bh / p.H);
        const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        if (slot < 0 || slot >= p.num_slots) {
            bad_slot = true;
            continue;
        }
        const int mh = p.head_map ? p.head_map[h] : h;  // row of S (conversions only)
        if (mh < 0 || mh >= p.Hm) {
            bad_head = true;
            continue;
        }
        uint8_t *rec = p.state + slot * p.slot_bytes + (int64_t)(h * p.V + c) * p.rec_bytes;
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int u = lane + 32 * i;
            if (u < K) continue;  // FP16 rows: column-mapped loop below
            const int r = u - K;
            uint8_t *crec = rec + p.codes_off + lo_chunk_off(r, 0, lo);  // chunk 0 (the whole row for 4-bit codes)
            uint8_t *crec1 = rec + p.codes_off + lo_chunk_off(r, 1, lo);
            uint32_t *mrec = reinterpret_cast<uint32_t *>(rec + p.meta_off + 4 * r);
            if (OP == kQuantize || OP == kDequantize) {
                const int n = p.perm[(int64_t)h * p.dk + u] & (p.dk - 1);  // d_k is a power of two
                float *row = p.S + ((((int64_t)b * p.Hm + mh) * p.dk + n) * p.dv + c * kG);
                float2 x[16];
                if (OP == kQuantize) {
#pragma unroll
                    for (int m = 0; m < 8; ++m) {
                        const float4 f = reinterpret_cast<const float4 *>(row)[m];
                        x[2 * m] = make_float2(f.x, f.y);
                        x[2 * m + 1] = make_float2(f.z, f.w);
                    }
                    if (HAD) hadamard_pairs(x);
                    if (FMT == kFmtE4M3) {
                        uint32_t w[8];
                        const float sc = quantize_group_e4m3(x, w);
                        *reinterpret_cast<uint4 *>(crec) = make_uint4(w[0], w[1], w[2], w[3]);
                        *reinterpret_cast<uint4 *>(crec1) = make_uint4(w[4], w[5], w[6], w[7]);
                        *mrec = __float_as_uint(sc);
                    } else {
#pragma unroll
                        for (int m = 0; m < 16; ++m) x[m] = mul2(x[m], splat2(kDown));  // working scale
                        if (U4) {
                            uint32_t w[4];
                            *mrec = quantize_group_u4(x, w);
                            *reinterpret_cast<uint4 *>(crec) = make_uint4(w[0], w[1], w[2], w[3]);
                        } else {
                            uint32_t w[8];
                            *mrec = quantize_group(x, w);
                            *reinterpret_cast<uint4 *>(crec) = make_uint4(w[0], w[1], w[2], w[3]);
                            *reinterpret_cast<uint4 *>(crec1) = make_uint4(w[4], w[5], w[6], w[7]);
                        }
                    }
                } else {
                    const uint4 c0 = *reinterpret_cast<const uint4 *>(crec);
                    if (U4) {
                        const uint32_t w[4] = {c0.x, c0.y, c0.z, c0.w};
                        dequantize_group_u4(w, *mrec, 1.0f, x);
                    } else {
                        const uint4 c1 = *reinterpret_cast<const uint4 *>(crec1);
                        const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                        if (FMT == kFmtE4M3) dequantize_group_e4m3(w, __uint_as_float(*mrec), 1.0f, x);
                        else dequantize_group(w, *mrec, 1.0f, x);
                    }
                    if (HAD) hadamard_pairs(x);
#pragma unroll
                    for (int m = 0; m < 8; ++m)
                        reinterpret_cast<float4 *>(row)[m] = make_float4(x[2 * m].x, x[2 * m].y, x[2 * m + 1].x, x[2 * m + 1].y);
                }
            } else {
                // logical tiers <-> record, 32-bit words (FP16 rows: column-mapped loop below)
                const int64_t row_bytes = (int64_t)p.V * CB;
                uint32_t *crow = reinterpret_cast<uint32_t *>(p.codes + ((((int64_t)b * p.H + h) * lo + r) * row_bytes + c * CB));
                uint32_t *mrow = reinterpret_cast<uint32_t *>(p.meta) + (((int64_t)b * p.H + h) * lo + r) * p.V + c;
#pragma unroll
                for (int m = 0; m < CB / 16; ++m) {
                    uint32_t *r4 = reinterpret_cast<uint32_t *>(m ? crec1 : crec);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        if (OP == kPackTiers) r4[e] = crow[4 * m + e];
                        else crow[4 * m + e] = r4[e];
                    }
                }
                if (OP == kPackTiers) *mrec = *mrow;
                else *mrow = *mrec;
            }
        }
        // ---- FP16 rows, lane = column, two rows per 32-bit word ----
        for (int u = 0; u < K; u += 2) {
            const bool two = u + 1 < K;
            uint32_t *word = reinterpret_cast<uint32_t *>(rec + hi_elem_off(u, lane));
            if (OP == kQuantize || OP == kDequantize) {
                float *r0 = p.S + ((((int64_t)b * p.Hm + mh) * p.dk + (p.perm[(int64_t)h * p.dk + u] & (p.dk - 1))) * p.dv + c * kG + lane);
                float *r1 = two ? p.S + ((((int64_t)b * p.Hm + mh) * p.dk + (p.perm[(int64_t)h * p.dk + u + 1] & (p.dk - 1))) * p.dv + c * kG + lane) : nullptr;
                if (OP == kQuantize) {
                    *word = f2_to_h2(*r0, two ? *r1 : 0.f);
                } else {
                    const float2 f = h2_to_f2(*word);
                    *r0 = f.x;
                    if (two) *r1 = f.y;
                }
            } else {
                uint16_t *t0 = p.hi + ((((int64_t)b * p.H + h) * K + u) * p.dv + c * kG + lane);
                uint16_t *t1 = two ? t0 + p.dv : nullptr;
                if (OP == kPackTiers) {
                    *word = (uint32_t)*t0 | ((uint32_t)(two ? *t1 : 0) << 16);
                } else {
                    const uint32_t w = *word;
                    *t0 = (uint16_t)(w & 0xffffu);
                    if (two) *t1 = (uint16_t)(w >> 16);
                }
            }
        }
        // zero the record padding so packed pools compare bit for bit
        if (OP == kQuantize || OP == kPackTiers) {
            const int used = p.meta_off + 4 * lo;
            if (lane < p.rec_bytes - used) rec[used + lane] = 0;
        }
    }
    if (lane == 0 && (bad_slot || bad_head))
        atomicOr(p.status, (bad_slot ? (uint32_t)kDevBadSlot : 0u) | (bad_head ? (uint32_t)kDevBadHead : 0u));
}

template <int OP>
static cudaError_t launch_convert(const ConvArgs &a, cudaStream_t stream) {
    ConvParams p{};
    static std::atomic<uint32_t *> cache[64];
    cudaError_t e = symbol_address_cached(&g_status_convert, cache, &p.status);
    if (e != cudaSuccess) return e;
    const RecGeom rg = rec_geom(a.dk, a.K, a.fmt);
    p.state = static_cast<uint8_t *>(a.state);
    p.num_slots = a.num_slots;
    p.slot_idx = a.slot_idx;
    p.perm = a.perm;
    p.S = a.S;
    p.hi = a.hi;
    p.codes = a.codes;
    p.meta = a.meta;
    p.batch = a.batch;
    p.H = a.H;
    p.Hm = a.head_map ? a.Hm : a.H;  // the tiers of pack / unpack are pool-indexed
    p.head_map = a.head_map;
    p.dk = a.dk;
    p.dv = a.dv;
    p.V = a.dv / kG;
    p.K = a.K;
    p.rec_bytes = rg.bytes;
    p.codes_off = rg.codes_off;
    p.meta_off = rg.meta_off;
    p.slot_bytes = (int64_t)a.H * p.V * rg.bytes;
    p.total_tiles = (int64_t)a.batch * a.H * p.V;
    if (p.total_tiles == 0) return cudaSuccess;
    const int warps = 8;
    const int64_t want = (p.total_tiles + warps - 1) / warps;
    const int grid = (int)std::min<int64_t>(want, (int64_t)sm_count() * 8);
    void (*kern)(ConvParams) = nullptr;
#define DAMP_PICK(R_)                                                                          \
    if (a.dk == 32 * R_) {                                                                     \
        switch (a.fmt) {                                                                       \
            case kFmtU8H32: kern = convert_kernel<R_, kFmtU8H32, OP>; break;                  \
            case kFmtU8: kern = convert_kernel<R_, kFmtU8, OP>; break;                        \
            case kFmtU4H32: kern = convert_kernel<R_, kFmtU4H32, OP>; break;                  \
            case kFmtU4: kern = convert_kernel<R_, kFmtU4, OP>; break;                        \
            case kFmtE4M3: kern = convert_kernel<R_, kFmtE4M3, OP>; break;                    \
            default: break;                                                                    \
        }                                                                                      \
    }
    DAMP_PICK(1)
    DAMP_PICK(2)
    DAMP_PICK(4)
#undef DAMP_PICK
    if (!kern) return cudaErrorInvalidValue;
    kern<<<grid, 32 * warps, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_quantize(const ConvArgs &a, cudaStream_t s) { return launch_convert<kQuantize>(a, s); }
cudaError_t launch_dequantize(const ConvArgs &a, cudaStream_t s) { return launch_convert<kDequantize>(a, s); }
cudaError_t launch_pack_tiers(const ConvArgs &a, cudaStream_t s) { return launch_convert<kPackTiers>(a, s); }
cudaError_t launch_unpack_tiers(const ConvArgs &a, cudaStream_t s) { return launch_convert<kUnpackTiers>(a, s); }

cudaError_t take_status_convert(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_convert, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_convert, &zero, sizeof(uint32_t));
}

}  // namespace damp
