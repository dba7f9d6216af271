// rowabs.cu -- the per-row symmetric absmax INT8 low tier (lo_format 2).
//
// Quantizer: one FP32 scale per packed row over all d_v values,
//   s = max_j |x_j| / 127,  q_j = sat_[-127,127](round_half_even(x_j / s)),  s = 0 -> q = 0,
// with no block transform; the FP16 tier of the K_hi protected channels is the
// same as in the paper's format (Sec. 3.2, App. A.1).  A row's scale depends on
// every value of the row, so the step cannot requantize one 32-column value
// block on its own: one warp owns a whole (slot, head) and sweeps its value
// blocks twice --
//   sweep 1: reconstruct + decay (S_bar = Lambda S), r = S_bar^T k, the delta
//            d = v - r, the output o = S_bar^T q + beta (k^T q) d, and each
//            row's new absmax over the updated values S_bar + beta k d^T;
//   sweep 2: recompute the updated values (same instructions, so the same bits)
//            and encode them with the new row scales, in place.
// The records of a head are re-read from L1/L2 in the second sweep.
//
// Storage reuses the paper format's record geometry: codes are int8 in the
// code area and the row's FP32 scale sits in the 4-byte metadata slot of the
// row in every value-block record of the head (the same value d_v/32 times).
#include "damp_common.cuh"
#include "damp_internal.h"

#include <algorithm>

namespace damp {

static __device__ uint32_t g_status_rowabs;

namespace {

constexpr int kRaWarps = 4;
constexpr int kRaMaxDv = 1024;
constexpr int kRaMaxDk = 128;

struct RowAbsStep {
    uint8_t *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    const uint8_t *perm;
    const void *q, *k, *v;
    const float *g, *beta;
    float *o;
    int32_t batch, H, Hqk, dk, dv, V, K;
    int32_t Hm;                // heads of the operands: held head h is model head head_map[h] (or h)
    const int32_t *head_map;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes;
    uint32_t *status;
};

// Lane l's sum over the warp of component l of v (a transposing butterfly:
// 16 + 8 + 4 + 2 + 1 shuffles).
__device__ __forceinline__ float transpose_sum32(float (&v)[32], int lane) {
#pragma unroll
    for (int st = 0; st < 5; ++st) {
        const int m = 16 >> st;
        const bool upper = (lane & m) != 0;
#pragma unroll
        for (int e = 0; e < m; ++e) {
            const float send = upper ? v[e] : v[e + m];
            const float keep = upper ? v[e + m] : v[e];
            v[e] = keep + __shfl_xor_sync(kFull, send, m);
        }
    }
    return v[0];
}

// Reconstructed and decayed low-tier row r of one record: a * (s * q_j).
__device__ __forceinline__ void lo_row_decayed(const uint8_t *rec, int codes_off, int meta_off, int lo, int r,
                                               float a, float (&x)[32]) {
    const uint4 c0 = *reinterpret_cast<const uint4 *>(rec + codes_off + lo_chunk_off(r, 0, lo));
    const uint4 c1 = *reinterpret_cast<const uint4 *>(rec + codes_off + lo_chunk_off(r, 1, lo));
    const float s = *reinterpret_cast<const float *>(rec + meta_off + 4 * r);
    const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
    for (int e = 0; e < 32; ++e) {
        const int qv = (int)(int8_t)(uint8_t)(w[e >> 2] >> (8 * (e & 3)));
        x[e] = __fmul_rn(a, __fmul_rn(s, (float)qv));
    }
}

__device__ __forceinline__ int8_t encode_s8(float x, float s) {
    float t = s == 0.f ? 0.f : rintf(__fdiv_rn(x, s));
    t = fminf(fmaxf(t, -127.f), 127.f);
    return (int8_t)(int)t;
}

template <bool KDA, bool BF16>
__global__ void __launch_bounds__(32 * kRaWarps) rowabs_step_kernel(const RowAbsStep p) {
    __shared__ float sm_d[kRaWarps][kRaMaxDv];
    __shared__ float sm_k[kRaWarps][kRaMaxDk], sm_q[kRaWarps][kRaMaxDk], sm_a[kRaWarps][kRaMaxDk];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t unit = (int64_t)blockIdx.x * kRaWarps + warp;
    if (unit >= (int64_t)p.batch * p.H) return;
    const int b = (int)(unit / p.H), h = (int)(unit % p.H);
    const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
    if (slot < 0 || slot >= p.num_slots) {
        if (lane == 0) atomicOr(p.status, (uint32_t)kDevBadSlot);
        return;
    }
    const int mh = p.head_map ? p.head_map[h] : h;
    if (mh < 0 || mh >= p.Hm) {
        if (lane == 0) atomicOr(p.status, (uint32_t)kDevBadHead);
        return;
    }
    const int64_t mu = (int64_t)b * p.Hm + mh;  // (batch row, model head) of the operands
    const int dk = p.dk, K = p.K, lo = dk - K, V = p.V;
    const int hq = (int)(((int64_t)mh * p.Hqk) / p.Hm);
    float *dsm = sm_d[warp];
    float *ks = sm_k[warp], *qs = sm_q[warp], *as = sm_a[warp];

    // operands in calibrated row order (row u holds key channel perm[h][u])
    const float beta = p.beta[mu];
    const float alpha = KDA ? 0.f : expf(p.g[mu]);
    float kq = 0.f;
    for (int u = lane; u < dk; u += 32) {
        const int ch = p.perm[(int64_t)h * dk + u] & (dk - 1);  // d_k is a power of two
        const float kv = load_in(p.k, ((int64_t)b * p.Hqk + hq) * dk + ch, BF16);
        const float qv = load_in(p.q, ((int64_t)b * p.Hqk + hq) * dk + ch, BF16);
        ks[u] = kv;
        qs[u] = qv;
        as[u] = KDA ? expf(p.g[mu * dk + ch]) : alpha;
        kq = fmaf(kv, qv, kq);
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) kq += __shfl_xor_sync(kFull, kq, m);
    const float bkq = beta * kq;
    __syncwarp();

    uint8_t *head = p.state + slot * p.slot_bytes + (int64_t)h * V * p.rec_bytes;
    float amax[4] = {0.f, 0.f, 0.f, 0.f};  // lo rows lane, lane+32, ... (d_k <= 128)

    // ---- sweep 1: r, d, o and the new row absmax ----
    for (int c = 0; c < V; ++c) {
        const uint8_t *rec = head + (int64_t)c * p.rec_bytes;
        float acc[32], accp[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) acc[e] = accp[e] = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int r = lane + 32 * i;
            if (r < lo) {
                float x[32];
                lo_row_decayed(rec, p.codes_off, p.meta_off, lo, r, as[K + r], x);
                const float kv = ks[K + r], qv = qs[K + r];
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    acc[e] = fmaf(x[e], kv, acc[e]);
                    accp[e] = fmaf(x[e], qv, accp[e]);
                }
            }
        }
        float rj = transpose_sum32(acc, lane);
        float pj = transpose_sum32(accp, lane);
        // FP16 tier, lane = column
        for (int u = 0; u < K; u += 2) {
            const float2 hv = h2_to_f2(*reinterpret_cast<const uint32_t *>(rec + hi_elem_off(u, lane)));
            const float x0 = __fmul_rn(as[u], hv.x);
            rj = fmaf(x0, ks[u], rj);
            pj = fmaf(x0, qs[u], pj);
            if (u + 1 < K) {
                const float x1 = __fmul_rn(as[u + 1], hv.y);
                rj = fmaf(x1, ks[u + 1], rj);
                pj = fmaf(x1, qs[u + 1], pj);
            }
        }
        const int j = kG * c + lane;
        const float dj = load_in(p.v, mu * p.dv + j, BF16) - rj;
        p.o[mu * p.dv + j] = fmaf(bkq, dj, pj);
        dsm[j] = dj;
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int r = lane + 32 * i;
            if (r < lo) {
                float x[32];
                lo_row_decayed(rec, p.codes_off, p.meta_off, lo, r, as[K + r], x);
                const float bk = __fmul_rn(beta, ks[K + r]);
#pragma unroll
                for (int e = 0; e < 32; ++e)
                    amax[i] = fmaxf(amax[i], fabsf(__fadd_rn(x[e], __fmul_rn(bk, dsm[kG * c + e]))));
            }
        }
    }
    float scale[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) scale[i] = __fdiv_rn(amax[i], 127.f);

    // ---- sweep 2: requantize in place ----
    for (int c = 0; c < V; ++c) {
        uint8_t *rec = head + (int64_t)c * p.rec_bytes;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int r = lane + 32 * i;
            if (r < lo) {
                float x[32];
                lo_row_decayed(rec, p.codes_off, p.meta_off, lo, r, as[K + r], x);
                const float bk = __fmul_rn(beta, ks[K + r]);
                uint32_t w[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const float xn = __fadd_rn(x[e], __fmul_rn(bk, dsm[kG * c + e]));
                    w[e >> 2] |= (uint32_t)(uint8_t)encode_s8(xn, scale[i]) << (8 * (e & 3));
                }
                *reinterpret_cast<uint4 *>(rec + p.codes_off + lo_chunk_off(r, 0, lo)) = make_uint4(w[0], w[1], w[2], w[3]);
                *reinterpret_cast<uint4 *>(rec + p.codes_off + lo_chunk_off(r, 1, lo)) = make_uint4(w[4], w[5], w[6], w[7]);
                *reinterpret_cast<float *>(rec + p.meta_off + 4 * r) = scale[i];
            }
        }
        const float dj = dsm[kG * c + lane];
        for (int u = 0; u < K; u += 2) {
            uint32_t *word = reinterpret_cast<uint32_t *>(rec + hi_elem_off(u, lane));
            const float2 hv = h2_to_f2(*word);
            const float y0 = __fadd_rn(__fmul_rn(as[u], hv.x), __fmul_rn(__fmul_rn(beta, ks[u]), dj));
            const float y1 = u + 1 < K
                                 ? __fadd_rn(__fmul_rn(as[u + 1], hv.y), __fmul_rn(__fmul_rn(beta, ks[u + 1]), dj))
                                 : 0.f;
            *word = f2_to_h2(y0, y1);
        }
    }
}

// ---- whole-state conversions: one warp per (slot, head, packed row) ----
struct RowAbsConv {
    uint8_t *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    const uint8_t *perm;
    float *S;
    uint16_t *hi;
    int8_t *codes;
    float *meta;
    int32_t batch, H, dk, dv, V, K;
    int32_t Hm;                // heads of S: held head h is row head_map[h] (or h)
    const int32_t *head_map;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes;
    uint32_t *status;
};

enum { kRaQuantize = 0, kRaDequantize = 1, kRaPack = 2, kRaUnpack = 3 };

template <int OP>
__global__ void __launch_bounds__(256) rowabs_convert_kernel(const RowAbsConv p) {
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwt = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int dk = p.dk, K = p.K, lo = dk - K, dv = p.dv;
    const int64_t total = (int64_t)p.batch * p.H * dk;
    bool bad_slot = false, bad_head = false;
    for (int64_t w = gw; w < total; w += nwt) {
        const int u = (int)(w % dk);
        const int64_t bh = w / dk;
        const int h = (int)(bh % p.H), b = (int)(bh / p.H);
        const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        if (slot < 0 || slot >= p.num_slots) {
            bad_slot = true;
            continue;
        }
        const int mh = p.head_map ? p.head_map[h] : h;
        if (mh < 0 || mh >= p.Hm) {
            bad_head = true;
            continue;
        }
        uint8_t *head = p.state + slot * p.slot_bytes + (int64_t)h * p.V * p.rec_bytes;
        const int n = p.perm ? (p.perm[(int64_t)h * dk + u] & (dk - 1)) : 0;
        float *srow = (OP == kRaQuantize || OP == kRaDequantize) ? p.S + (((int64_t)b * p.Hm + mh) * dk + n) * dv
                                                                  : nullptr;
        if (u < K) {
            for (int j = lane; j < dv; j += 32) {
                uint8_t *rec = head + (int64_t)(j >> 5) * p.rec_bytes;
                uint16_t *e = reinterpret_cast<uint16_t *>(rec + hi_elem_off(u, j & 31));
                if (OP == kRaQuantize) *e = __half_as_ushort(__float2half_rn(srow[j]));
                if (OP == kRaDequantize) srow[j] = __half2float(__ushort_as_half(*e));
                if (OP == kRaPack) *e = p.hi[(bh * K + u) * dv + j];
                if (OP == kRaUnpack) p.hi[(bh * K + u) * dv + j] = *e;
                // an odd K leaves the high half of the last row pair zero
                if ((OP == kRaQuantize || OP == kRaPack) && u == K - 1 && (K & 1))
                    *reinterpret_cast<uint16_t *>(rec + hi_elem_off(K, j & 31)) = 0;
            }
        } else {
            const int r = u - K;
            auto code_at = [&](int j) -> int8_t * {
                uint8_t *rec = head + (int64_t)(j >> 5) * p.rec_bytes;
                return reinterpret_cast<int8_t *>(rec + p.codes_off + lo_chunk_off(r, (j & 31) >> 4, lo) + (j & 15));
            };
            auto meta_at = [&](int c) {
                return reinterpret_cast<float *>(head + (int64_t)c * p.rec_bytes + p.meta_off + 4 * r);
            };
            if (OP == kRaQuantize) {
                float amax = 0.f;
                for (int j = lane; j < dv; j += 32) amax = fmaxf(amax, fabsf(srow[j]));
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(kFull, amax, m));
                const float s = __fdiv_rn(amax, 127.f);
                for (int j = lane; j < dv; j += 32) *code_at(j) = encode_s8(srow[j], s);
                for (int c = lane; c < p.V; c += 32) *meta_at(c) = s;
            } else if (OP == kRaDequantize) {
                for (int j = lane; j < dv; j += 32) srow[j] = __fmul_rn(*meta_at(j >> 5), (float)*code_at(j));
            } else if (OP == kRaPack) {
                const int8_t *crow = p.codes + (bh * lo + r) * dv;
                for (int j = lane; j < dv; j += 32) *code_at(j) = crow[j];
                for (int c = lane; c < p.V; c += 32) *meta_at(c) = p.meta[bh * lo + r];
            } else {
                int8_t *crow = p.codes + (bh * lo + r) * dv;
                for (int j = lane; j < dv; j += 32) crow[j] = *code_at(j);
                if (lane == 0) p.meta[bh * lo + r] = *meta_at(0);
            }
        }
        // zero the record padding so packed pools compare bit for bit
        if ((OP == kRaQuantize || OP == kRaPack) && u == 0) {
            const int used = p.meta_off + 4 * lo;
            for (int c = 0; c < p.V; ++c)
                if (lane < p.rec_bytes - used) head[(int64_t)c * p.rec_bytes + used + lane] = 0;
        }
    }
    if (lane == 0 && (bad_slot || bad_head))
        atomicOr(p.status, (bad_slot ? (uint32_t)kDevBadSlot : 0u) | (bad_head ? (uint32_t)kDevBadHead : 0u));
}

uint32_t *status_word(cudaError_t *e) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *p = nullptr;
    *e = symbol_address_cached(&g_status_rowabs, cache, &p);
    return p;
}

}  // namespace

cudaError_t launch_rowabs_step(const StepArgs &a, cudaStream_t stream) {
    if (a.dk > kRaMaxDk || a.dv > kRaMaxDv) return cudaErrorInvalidValue;
    RowAbsStep p{};
    cudaError_t e;
    p.status = status_word(&e);
    if (e != cudaSuccess) return e;
    const RecGeom rg = rec_geom(a.dk, a.K);
    p.state = static_cast<uint8_t *>(a.state);
    p.num_slots = a.num_slots;
    p.slot_idx = a.slot_idx;
    p.perm = a.perm;
    p.q = a.q;
    p.k = a.k;
    p.v = a.v;
    p.g = a.g;
    p.beta = a.beta;
    p.o = a.o;
    p.batch = a.batch;
    p.H = a.H;
    p.Hqk = a.Hqk;
    p.Hm = a.Hm;
    p.head_map = a.head_map;
    p.dk = a.dk;
    p.dv = a.dv;
    p.V = a.dv / kG;
    p.K = a.K;
    p.rec_bytes = rg.bytes;
    p.codes_off = rg.codes_off;
    p.meta_off = rg.meta_off;
    p.slot_bytes = (int64_t)a.H * p.V * rg.bytes;
    const int64_t units = (int64_t)a.batch * a.H;
    if (units == 0) return cudaSuccess;
    const int64_t grid = (units + kRaWarps - 1) / kRaWarps;
    if (grid > INT32_MAX) return cudaErrorInvalidValue;
    void (*kern)(RowAbsStep) = a.kda ? (a.in_bf16 ? rowabs_step_kernel<true, true> : rowabs_step_kernel<true, false>)
                                     : (a.in_bf16 ? rowabs_step_kernel<false, true> : rowabs_step_kernel<false, false>);
    kern<<<(unsigned)grid, 32 * kRaWarps, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_rowabs_convert(const ConvArgs &a, int op, cudaStream_t stream) {
    RowAbsConv p{};
    cudaError_t e;
    p.status = status_word(&e);
    if (e != cudaSuccess) return e;
    const RecGeom rg = rec_geom(a.dk, a.K);
    p.state = static_cast<uint8_t *>(a.state);
    p.num_slots = a.num_slots;
    p.slot_idx = a.slot_idx;
    p.perm = a.perm;
    p.S = a.S;
    p.hi = a.hi;
    p.codes = reinterpret_cast<int8_t *>(a.codes);
    p.meta = reinterpret_cast<float *>(a.meta);
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
    const int64_t warps = (int64_t)a.batch * a.H * a.dk;
    if (warps == 0) return cudaSuccess;
    const int grid = (int)std::min<int64_t>((warps + 7) / 8, (int64_t)sm_count() * 16);
    void (*kern)(RowAbsConv) = op == kRaQuantize     ? rowabs_convert_kernel<kRaQuantize>
                               : op == kRaDequantize ? rowabs_convert_kernel<kRaDequantize>
                               : op == kRaPack       ? rowabs_convert_kernel<kRaPack>
                                                     : rowabs_convert_kernel<kRaUnpack>;
    kern<<<grid, 256, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t take_status_rowabs(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_rowabs, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_rowabs, &zero, sizeof(uint32_t));
}

}  // namespace damp
