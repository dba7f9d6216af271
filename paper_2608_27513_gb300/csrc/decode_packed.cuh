// decode_packed.cuh -- fused DAMP decode step on the packed mixed-precision state.
//
// One launch updates every (request slot, value head) state of one layer for one
// decode step (Sec. 3.1, Eq. delta_update) and requantizes it once (Sec. 3.3,
// Eq. quantized_recurrence) in place in the packed cache of Sec. 5.2 / App. A.5.
//
// Work decomposition (own design for sm_103a): value columns are independent in
// the update, and a quantization group is 32 columns of one row, so a tile is
// (slot, head, value block c): all d_k packed rows x 32 columns.  A tile is one
// contiguous record (value-block-major, App. A.5) and is self-contained: no
// cross-tile reduction.  One warp owns one tile at a time; lane l owns packed
// rows l, l+32, ... with all 32 columns in registers, so min/max and the
// requantizer of a group are thread-local.  The two column reductions
// r = S_bar^T k and o = S^T q go through shared memory.
//
// Domains: the low tier stores codes of H_32-transformed rows (App. A.5).  Since
// H_32 acts on the value axis only and is symmetric and orthonormal, the update
// can be carried out in the transformed domain: with S~ = S H,
//     r~ = H r,  S~_t = Lambda S~ + beta k (H v - r~)^T,  o = H (S~^T q).
// Low-tier rows therefore never pass through a butterfly; only the 32-vectors
// v, r_hi, d and o do (a 5-step butterfly across the warp's lanes).  FP16 rows
// stay in the natural domain: their partial sums are reduced separately and
// transformed once per tile.
//
// Pipeline: a persistent grid; every warp walks a contiguous range of tiles.
// Lane 0 keeps NSTAGE-1 tiles in flight with 1-D bulk copies (TMA engine) into a
// per-warp ring of shared-memory stages, each with its own mbarrier; the updated
// record is written back into its stage and returned with a bulk store.
#pragma once

#include "damp_common.cuh"

namespace damp {

struct PackedParams {
    uint8_t *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    const uint8_t *perm;
    const void *q, *k, *v;
    const float *g, *beta;
    float *o;
    int32_t batch, H, Hqk, dk, dv, V, K;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes;
    int32_t nstage, stage_bytes, warp_smem, stage0_off;
    int32_t off_v, off_q, off_k, off_g, off_perm;
    int32_t bytes_v, bytes_qk, bytes_g, bytes_perm;
    int64_t total_tiles;
    uint32_t *status;
};

constexpr int kPartOff = 64;                        // after NSTAGE (<= 8) mbarriers
constexpr int kPartStride = 36;                     // floats per row of the partial-sum buffer
constexpr int kDvecOff = kPartOff + 32 * kPartStride * 4;
constexpr int kScratchBytes = kDvecOff + 64 * 4;    // bytes before the first stage (rounded up by the host)

__device__ __forceinline__ float ldsf(uint32_t a) { return __uint_as_float(lds32(a)); }

// Column sum over the lanes' 32-vectors: lane j returns sum_l v_l[j].
// Uses part[32][36]; the caller brackets it with __syncwarp.
__device__ __forceinline__ float column_sum(const float (&v)[32], uint32_t part, int lane) {
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
        uint4 w;
        w.x = __float_as_uint(v[4 * jj]);
        w.y = __float_as_uint(v[4 * jj + 1]);
        w.z = __float_as_uint(v[4 * jj + 2]);
        w.w = __float_as_uint(v[4 * jj + 3]);
        sts128(part + (lane * kPartStride + 4 * jj) * 4, w);
    }
    __syncwarp();
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
    for (int l = 0; l < 32; l += 4) {
        s0 += ldsf(part + ((l + 0) * kPartStride + lane) * 4);
        s1 += ldsf(part + ((l + 1) * kPartStride + lane) * 4);
        s2 += ldsf(part + ((l + 2) * kPartStride + lane) * 4);
        s3 += ldsf(part + ((l + 3) * kPartStride + lane) * 4);
    }
    __syncwarp();
    return (s0 + s1) + (s2 + s3);
}

// Sum of the first n rows of part[][] at column `lane`.
__device__ __forceinline__ float partial_rows_sum(uint32_t part, int n, int lane) {
    float s = 0.f;
    for (int l = 0; l < n; ++l) s += ldsf(part + (l * kPartStride + lane) * 4);
    return s;
}

__device__ __forceinline__ void store_row_scaled(uint32_t part, int lane, const float (&x)[32], float c) {
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
        uint4 w;
        w.x = __float_as_uint(x[4 * jj] * c);
        w.y = __float_as_uint(x[4 * jj + 1] * c);
        w.z = __float_as_uint(x[4 * jj + 2] * c);
        w.w = __float_as_uint(x[4 * jj + 3] * c);
        sts128(part + (lane * kPartStride + 4 * jj) * 4, w);
    }
}

template <int R, bool KDA, bool HAD, bool BF16>
__global__ void __launch_bounds__(256, 1) packed_step_kernel(const PackedParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const uint32_t ws = smem_u32(smem) + (uint32_t)(warp * p.warp_smem);
    const uint32_t bar0 = ws;
    const uint32_t part = ws + kPartOff;
    const uint32_t dvec = ws + kDvecOff;
    const uint32_t stage0 = ws + p.stage0_off;
    const int esz = BF16 ? 2 : 4;
    const int K = p.K;

    const int64_t gw = (int64_t)blockIdx.x * nw + warp;
    const int64_t nwt = (int64_t)gridDim.x * nw;
    const int64_t t0 = p.total_tiles * gw / nwt;
    const int64_t t1 = p.total_tiles * (gw + 1) / nwt;
    if (t0 >= t1) return;

    if (lane == 0) {
        for (int s = 0; s < p.nstage; ++s) mbar_init(bar0 + 8 * s, 1);
        fence_mbar_init();
    }
    __syncwarp();

    // ---- producer (lane 0): bulk copies of tile t into stage s ----
    auto issue = [&](int64_t t, int s) {
        const int c = (int)(t % p.V);
        const int64_t bh = t / p.V;
        const int h = (int)(bh % p.H);
        const int b = (int)(bh / p.H);
        const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        const bool ok = slot >= 0 && slot < p.num_slots;
        const bool ops = (t == t0) || (c == 0);
        const uint32_t st = stage0 + (uint32_t)(s * p.stage_bytes);
        const uint32_t bar = bar0 + 8 * s;
        uint32_t bytes = (uint32_t)p.bytes_v;
        if (ok) bytes += (uint32_t)p.rec_bytes;
        if (ops) bytes += 2u * p.bytes_qk + p.bytes_g + p.bytes_perm;
        mbar_arrive_expect_tx(bar, bytes);
        if (ok) bulk_g2s(st, p.state + slot * p.slot_bytes + (int64_t)(h * p.V + c) * p.rec_bytes, p.rec_bytes, bar);
        bulk_g2s(st + p.off_v, (const uint8_t *)p.v + (((int64_t)b * p.H + h) * p.dv + c * kG) * esz, p.bytes_v, bar);
        if (ops) {
            const int hq = (h * p.Hqk) / p.H;
            const int64_t qoff = ((int64_t)b * p.Hqk + hq) * p.dk * esz;
            bulk_g2s(st + p.off_q, (const uint8_t *)p.q + qoff, p.bytes_qk, bar);
            bulk_g2s(st + p.off_k, (const uint8_t *)p.k + qoff, p.bytes_qk, bar);
            if (KDA) bulk_g2s(st + p.off_g, p.g + ((int64_t)b * p.H + h) * p.dk, p.bytes_g, bar);
            bulk_g2s(st + p.off_perm, p.perm + (int64_t)h * p.dk, p.bytes_perm, bar);
        }
    };

    if (lane == 0) {
        for (int j = 0; j < p.nstage - 1 && t0 + j < t1; ++j) issue(t0 + j, j);
    }

    float kk[R], qq[R], bk[R], aa[R];
    int s = 0;
    uint32_t parity = 0;
    bool timed_out = false, bad_slot = false;
    int64_t t_fail = t1;

    for (int64_t t = t0; t < t1; ++t) {
        const uint32_t st = stage0 + (uint32_t)(s * p.stage_bytes);
        if (!__all_sync(kFull, mbar_wait_bounded(bar0 + 8 * s, parity))) {
            timed_out = true;
            t_fail = t;
            break;
        }
        const int c = (int)(t % p.V);
        const int64_t bh = t / p.V;
        const int h = (int)(bh % p.H);
        const int b = (int)(bh / p.H);
        const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        const bool ok = slot >= 0 && slot < p.num_slots;
        bad_slot |= !ok;

        // ---- per-(slot, head) operands, gathered into calibrated key order ----
        if (t == t0 || c == 0) {
            const float beta = p.beta[(int64_t)b * p.H + h];
            const float alpha = KDA ? 0.f : expf(p.g[(int64_t)b * p.H + h]);
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int u = lane + 32 * i;
                // d_k is a power of two: masking keeps a malformed permutation in bounds
                const int ch = (int)(lds32(st + p.off_perm + (u & ~3)) >> (8 * (u & 3))) & (p.dk - 1);
                float kv, qv;
                if (BF16) {
                    const uint32_t kw = lds32(st + p.off_k + 2 * (ch & ~1));
                    const uint32_t qw = lds32(st + p.off_q + 2 * (ch & ~1));
                    kv = __uint_as_float((ch & 1) ? (kw & 0xffff0000u) : (kw << 16));
                    qv = __uint_as_float((ch & 1) ? (qw & 0xffff0000u) : (qw << 16));
                } else {
                    kv = ldsf(st + p.off_k + 4 * ch);
                    qv = ldsf(st + p.off_q + 4 * ch);
                }
                kk[i] = kv;
                qq[i] = qv;
                bk[i] = beta * kv;
                aa[i] = KDA ? expf(ldsf(st + p.off_g + 4 * ch)) : alpha;
            }
        }

        // ---- v block -> transformed domain ----
        float vj;
        if (BF16) {
            const uint32_t w = lds32(st + p.off_v + 2 * (lane & ~1));
            vj = __uint_as_float((lane & 1) ? (w & 0xffff0000u) : (w << 16));
        } else {
            vj = ldsf(st + p.off_v + 4 * lane);
        }
        const float vt = HAD ? hadamard_lanes(vj, lane) : vj;

        float x[R][32];
        float acc[32];
        float rhi = 0.f;

        if (ok) {
            // ---- phase 1: reconstruct, decay, partial r = S_bar^T k ----
#pragma unroll
            for (int j = 0; j < 32; ++j) acc[j] = 0.f;
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int u = lane + 32 * i;
                if (u < K) {
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        const uint4 w = lds128(st + hi_chunk_off(u, m));
                        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float2 f = h2_to_f2(ww[e]);
                            x[i][8 * m + 2 * e] = f.x * aa[i];
                            x[i][8 * m + 2 * e + 1] = f.y * aa[i];
                        }
                    }
                    store_row_scaled(part, lane, x[i], kk[i]);
                } else {
                    const int r = u - K;
                    const uint4 c0 = lds128(st + p.codes_off + lo_chunk_off(r, 0));
                    const uint4 c1 = lds128(st + p.codes_off + lo_chunk_off(r, 1));
                    const uint32_t sz = lds32(st + p.meta_off + 4 * r);
                    const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                    dequantize_group(w, sz, aa[i], x[i]);
#pragma unroll
                    for (int j = 0; j < 32; ++j) acc[j] = fmaf(x[i][j], kk[i], acc[j]);
                }
                if (32 * i < K) {  // warp-uniform: this slot holds FP16 rows
                    __syncwarp();
                    rhi += partial_rows_sum(part, min(32, K - 32 * i), lane);
                    __syncwarp();
                }
            }
            const float rlo = column_sum(acc, part, lane);
            const float rt = rlo + ((HAD && K > 0) ? hadamard_lanes(rhi, lane) : rhi);
            const float dt = vt - rt;                                        // d~ = H(v - r)
            const float dn = (HAD && K > 0) ? hadamard_lanes(dt, lane) : dt;  // natural d
            sts32(dvec + 4 * lane, __float_as_uint(dt));
            sts32(dvec + 128 + 4 * lane, __float_as_uint(dn));
        }

        // ---- keep the ring full: next load goes into the stage of tile t-1 ----
        if (lane == 0 && t + p.nstage - 1 < t1) {
            bulk_wait_read_all();
            const int sn = (s + p.nstage - 1) % p.nstage;
            issue(t + p.nstage - 1, sn);
        }

        if (ok) {
            __syncwarp();
            float d[32];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                const uint4 w = lds128(dvec + 16 * jj);
                d[4 * jj] = __uint_as_float(w.x);
                d[4 * jj + 1] = __uint_as_float(w.y);
                d[4 * jj + 2] = __uint_as_float(w.z);
                d[4 * jj + 3] = __uint_as_float(w.w);
            }
            // ---- phase 2: rank-1 correction, partial o, requantize in place ----
            float ohi = 0.f;
#pragma unroll
            for (int j = 0; j < 32; ++j) acc[j] = 0.f;
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int u = lane + 32 * i;
                if (u < K) {
#pragma unroll
                    for (int jj = 0; jj < 8; ++jj) {
                        const uint4 w = lds128(dvec + 128 + 16 * jj);
                        x[i][4 * jj] = fmaf(bk[i], __uint_as_float(w.x), x[i][4 * jj]);
                        x[i][4 * jj + 1] = fmaf(bk[i], __uint_as_float(w.y), x[i][4 * jj + 1]);
                        x[i][4 * jj + 2] = fmaf(bk[i], __uint_as_float(w.z), x[i][4 * jj + 2]);
                        x[i][4 * jj + 3] = fmaf(bk[i], __uint_as_float(w.w), x[i][4 * jj + 3]);
                    }
                    store_row_scaled(part, lane, x[i], qq[i]);
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        uint32_t hw[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            hw[e] = f2_to_h2(x[i][8 * m + 2 * e], x[i][8 * m + 2 * e + 1]);
                        }
                        sts128(st + hi_chunk_off(u, m), make_uint4(hw[0], hw[1], hw[2], hw[3]));
                    }
                } else {
                    const int r = u - K;
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        x[i][j] = fmaf(bk[i], d[j], x[i][j]);
                        acc[j] = fmaf(x[i][j], qq[i], acc[j]);
                    }
                    uint32_t w[8];
                    const uint32_t sz = quantize_group(x[i], w);
                    sts128(st + p.codes_off + lo_chunk_off(r, 0), make_uint4(w[0], w[1], w[2], w[3]));
                    sts128(st + p.codes_off + lo_chunk_off(r, 1), make_uint4(w[4], w[5], w[6], w[7]));
                    sts32(st + p.meta_off + 4 * r, sz);
                }
                if (32 * i < K) {
                    __syncwarp();
                    ohi += partial_rows_sum(part, min(32, K - 32 * i), lane);
                    __syncwarp();
                }
            }
            const float olo = column_sum(acc, part, lane);
            const float oj = ((HAD) ? hadamard_lanes(olo, lane) : olo) + ohi;
            p.o[((int64_t)b * p.H + h) * p.dv + c * kG + lane] = oj;

            // ---- write the updated record back ----
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                bulk_s2g(p.state + slot * p.slot_bytes + (int64_t)(h * p.V + c) * p.rec_bytes, st, p.rec_bytes);
                bulk_commit();
            }
        }
        __syncwarp();
        if (++s == p.nstage) {
            s = 0;
            parity ^= 1u;
        }
    }
    if (timed_out) {
        // let the loads already in flight land (each wait bounded) before the CTA's
        // shared memory goes away
        const int64_t last = min(t1 - 1, t_fail + p.nstage - 2);
        for (int64_t tt = t_fail + 1; tt <= last; ++tt) {
            const int64_t idx = tt - t0;
            mbar_wait_bounded(bar0 + 8 * (int)(idx % p.nstage), (uint32_t)((idx / p.nstage) & 1));
        }
    }
    if (lane == 0) {
        bulk_wait_all();
        const uint32_t bits = (timed_out ? kDevWaitTimeout : 0u) | (bad_slot ? kDevBadSlot : 0u);
        if (bits) atomicOr(p.status, bits);
    }
}

}  // namespace damp
