// prefill.cuh -- one prefill chunk on the packed state (App. A.5, "Prefill path").
//
// The recurrence runs in FP32 over the chunk's tokens (Eq. delta_update per token,
// o_t = S_t^T q_t) and the chunk-final state is quantized once, straight into the
// packed cache that decode steps and later chunks read.
//
// Work unit = tile (slot, head, value block c): all d_k rows x 32 columns, for the
// whole chunk of that slot.  One warp owns a tile from load to store, so its FP32
// state never leaves the SM between tokens:
//   low-tier rows  lane l holds rows l, l+32, ... (32 columns each) in registers,
//                  in the H_32 domain and scaled by 2^-39 as in the decode step
//                  (decay and the rank-1 update are row/column scalings there too);
//   FP16 rows      lane j holds column j of every FP16 row in shared memory as FP32.
// Per token: decay, partial sums of r~ = S~^T k and p~ = S~^T q, column sums, the
// lane butterflies for r, d, p (as in the decode step), o_t, and the update.  The
// next token's operands (q, k, g, v block, beta) stream into a double buffer by
// cp.async while the current token runs.  After the last token the tile is
// requantized like a decode step and stored with plain 128-bit stores.
#pragma once

#include "damp_common.cuh"
#include "formats.cuh"

namespace damp {

struct PrefillParams {
    uint8_t *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    const int32_t *lengths;
    const uint8_t *perm;
    const void *q, *k, *v;
    const float *g, *beta;
    float *o;
    int32_t batch, T, H, Hqk, dk, dv, V, K;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes, total_tiles;
    // per-warp shared memory
    int32_t warp_smem, dvec_off, hops_off, perm_off, hbuf_off, ops_off, ops_bytes;
    int32_t off_q, off_k, off_g, off_v, off_beta;
    uint32_t *status;
};

template <int RL, bool KDA, int FMT, bool BF16>
__global__ void __launch_bounds__(256, 1) prefill_chunk_kernel(const PrefillParams p) {
    constexpr int R = RL > 0 ? RL : 1;
    constexpr bool HAD = fmt_had(FMT);
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const LaneSigns sg = lane_signs(lane);
    const uint32_t ws = smem_u32(smem) + (uint32_t)(warp * p.warp_smem);
    const uint32_t part = ws;  // column_sum2 buffer at the start of the warp's area
    const uint32_t dvec = ws + p.dvec_off;
    const uint32_t hops = ws + p.hops_off;
    const uint32_t perm_s = ws + p.perm_off;
    const uint32_t hbuf = ws + p.hbuf_off;
    const uint32_t ops0 = ws + p.ops_off;
    const int esz = BF16 ? 2 : 4;
    const int K = p.K, dk = p.dk, lo = dk - K, H = p.H, V = p.V, T = p.T;

    const int64_t gw = (int64_t)blockIdx.x * nw + warp;
    const int64_t nwt = (int64_t)gridDim.x * nw;
    bool bad_slot = false;

    // operands of token tok of (b, h) for value block c into buffer dst
    auto load_token = [&](int b, int h, int c, int tok, uint32_t dst) {
        const int hq = (int)(((int64_t)h * p.Hqk) / H);
        const int64_t bt = (int64_t)b * T + tok;
        const uint8_t *qrow = (const uint8_t *)p.q + (bt * p.Hqk + hq) * dk * esz;
        const uint8_t *krow = (const uint8_t *)p.k + (bt * p.Hqk + hq) * dk * esz;
        const uint8_t *grow = (const uint8_t *)(p.g + (bt * H + h) * (KDA ? dk : 1));
        const uint8_t *vblk = (const uint8_t *)p.v + ((bt * H + h) * p.dv + kG * c) * esz;
        const int nq = dk * esz / 16, ng = KDA ? dk * 4 / 16 : 0, nv = kG * esz / 16;
        const int total = 2 * nq + ng + nv;
        for (int ci = lane; ci < total; ci += 32) {
            int j = ci;
            if (j < nq) {
                cp_async16(dst + p.off_q + 16 * j, qrow + 16 * j);
            } else if ((j -= nq) < nq) {
                cp_async16(dst + p.off_k + 16 * j, krow + 16 * j);
            } else if ((j -= nq) < ng) {
                cp_async16(dst + p.off_g + 16 * j, grow + 16 * j);
            } else {
                j -= ng;
                cp_async16(dst + p.off_v + 16 * j, vblk + 16 * j);
            }
        }
        if (lane == 0) {
            cp_async4(dst + p.off_beta, p.beta + bt * H + h);
            if (!KDA) cp_async4(dst + p.off_g, grow);
        }
        cp_async_commit();
    };

    for (int64_t t = p.total_tiles * gw / nwt; t < p.total_tiles * (gw + 1) / nwt; ++t) {
        const int c = (int)(t % V);
        const int64_t bh = t / V;
        const int h = (int)(bh % H), b = (int)(bh / H);
        const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        if (slot < 0 || slot >= p.num_slots) {
            bad_slot = true;
            continue;
        }
        const int Tb = p.lengths ? min(max(p.lengths[b], 0), T) : T;
        if (Tb == 0) continue;
        uint8_t *const grec = p.state + slot * p.slot_bytes + (int64_t)(h * V + c) * p.rec_bytes;

        // π of this head, then token 0's operands
        __syncwarp();  // the previous tile's readers of the shared buffers are done
        for (int ci = lane; ci < dk / 16; ci += 32) cp_async16(perm_s + 16 * ci, p.perm + (int64_t)h * dk + 16 * ci);
        load_token(b, h, c, 0, ops0);

        // ---- reconstruct the tile in FP32 (undecayed; low tier in the H domain at 2^-39) ----
        float2 x[R][16];
#pragma unroll
        for (int i = 0; i < RL; ++i) {
            const int r = min(lane + 32 * i, lo - 1);
            const uint4 c0 = *reinterpret_cast<const uint4 *>(grec + p.codes_off + lo_chunk_off(r, 0, lo));
            const uint32_t sz = *reinterpret_cast<const uint32_t *>(grec + p.meta_off + 4 * r);
            if constexpr (fmt_u4(FMT)) {
                const uint32_t w[4] = {c0.x, c0.y, c0.z, c0.w};
                dequantize_group_u4(w, sz, kDown, x[i]);
            } else {
                const uint4 c1 = *reinterpret_cast<const uint4 *>(grec + p.codes_off + lo_chunk_off(r, 1, lo));
                const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                if constexpr (FMT == kFmtE4M3) dequantize_group_e4m3(w, __uint_as_float(sz), kDown, x[i]);
                else dequantize_group(w, sz, kDown, x[i]);
            }
        }
        for (int u = 0; u < K; u += 2) {
            const float2 f = h2_to_f2(*reinterpret_cast<const uint32_t *>(grec + hi_elem_off(u, lane)));
            sts32(hbuf + 4 * (32 * u + lane), __float_as_uint(f.x));
            if (u + 1 < K) sts32(hbuf + 4 * (32 * (u + 1) + lane), __float_as_uint(f.y));
        }

        for (int tok = 0; tok < Tb; ++tok) {
            const uint32_t ob = ops0 + (uint32_t)((tok & 1) * p.ops_bytes);
            cp_async_wait_all();
            __syncwarp();
            if (tok + 1 < Tb) load_token(b, h, c, tok + 1, ops0 + (uint32_t)(((tok + 1) & 1) * p.ops_bytes));

            // ---- operands in calibrated order ----
            const float beta = ldsf(ob + p.off_beta);
            const float alpha = KDA ? 0.f : expf(ldsf(ob + p.off_g));
            auto chan = [&](int u) { return (int)(lds32(perm_s + (u & ~3)) >> (8 * (u & 3))) & (dk - 1); };
            auto kv_at = [&](int ch) { return BF16 ? bf16_at(ob + p.off_k, ch) : ldsf(ob + p.off_k + 4 * ch); };
            auto qv_at = [&](int ch) { return BF16 ? bf16_at(ob + p.off_q, ch) : ldsf(ob + p.off_q + 4 * ch); };
            auto av_at = [&](int ch) { return KDA ? expf(ldsf(ob + p.off_g + 4 * ch)) : alpha; };
            float2 kk[R], qq[R], bk[R], aa[R];
            float kq = 0.f;
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int r = lane + 32 * i;
                const bool live = r < lo && i < RL;
                const int ch = chan(live ? K + r : 0);
                const float kv = live ? kv_at(ch) : 0.f;
                const float qv = live ? qv_at(ch) : 0.f;
                kk[i] = splat2(kv);
                qq[i] = splat2(qv);
                bk[i] = splat2(beta * kv * kDown);
                aa[i] = splat2(av_at(ch));
                kq = fmaf(kv, qv, kq);
            }
            // FP16 rows: {a_u, k_u, q_u, beta k_u} per row
            for (int u = lane; u < K; u += 32) {
                const int ch = chan(u);
                const float kv = kv_at(ch), qv = qv_at(ch);
                sts128(hops + 16 * u, make_uint4(__float_as_uint(av_at(ch)), __float_as_uint(kv), __float_as_uint(qv),
                                                 __float_as_uint(beta * kv)));
                kq = fmaf(kv, qv, kq);
            }
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) kq += __shfl_xor_sync(kFull, kq, m);
            const float bkq = beta * kq;
            __syncwarp();

            // ---- decay and partial sums ----
            float2 acc[16], accp[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] = accp[j] = make_float2(0.f, 0.f);
#pragma unroll
            for (int i = 0; i < RL; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    x[i][j] = mul2(x[i][j], aa[i]);
                    acc[j] = fma2(x[i][j], kk[i], acc[j]);
                    accp[j] = fma2(x[i][j], qq[i], accp[j]);
                }
            }
            float rhi = 0.f, phi = 0.f;
            for (int u = 0; u < K; ++u) {
                const uint4 op = lds128(hops + 16 * u);
                const float hb = __uint_as_float(op.x) * ldsf(hbuf + 4 * (32 * u + lane));  // decayed FP16 row
                sts32(hbuf + 4 * (32 * u + lane), __float_as_uint(hb));
                rhi = fmaf(hb, __uint_as_float(op.y), rhi);
                phi = fmaf(hb, __uint_as_float(op.z), phi);
            }
            const float2 lo_sums = column_sum2(acc, accp, part, lane);
            const float rlo = lo_sums.x * kUp, plo = lo_sums.y * kUp;

            // ---- d, o_t, H d ----
            const float vj = BF16 ? bf16_at(ob + p.off_v, lane) : ldsf(ob + p.off_v + 4 * lane);
            float dj, dt, pj;
            if (HAD) {
                const float vt = hadamard_lanes(vj, sg);
                const float hr_lo = hadamard_lanes(rlo, sg);
                const float hp_lo = hadamard_lanes(plo, sg);
                const float hr_hi = K > 0 ? hadamard_lanes(rhi, sg) : 0.f;
                dj = vj - (hr_lo + rhi);
                dt = vt - (rlo + hr_hi);
                pj = hp_lo + phi;
            } else {
                dj = vj - (rlo + rhi);
                dt = dj;
                pj = plo + phi;
            }
            p.o[(((int64_t)b * T + tok) * H + h) * p.dv + kG * c + lane] = fmaf(bkq, dj, pj);
            sts32(dvec + 4 * lane, __float_as_uint(dt));
            __syncwarp();

            // ---- rank-1 update ----
            float2 d[16];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                const uint4 w = lds128(dvec + 16 * jj);
                d[2 * jj] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
                d[2 * jj + 1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
            }
#pragma unroll
            for (int i = 0; i < RL; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) x[i][j] = fma2(bk[i], d[j], x[i][j]);
            }
            for (int u = 0; u < K; ++u) {
                const float hb = ldsf(hbuf + 4 * (32 * u + lane));
                sts32(hbuf + 4 * (32 * u + lane), __float_as_uint(fmaf(__uint_as_float(lds128(hops + 16 * u).w), dj, hb)));
            }
            __syncwarp();  // dvec, hops and the token buffer are reused by the next token
        }

        // ---- requantize the chunk-final tile and store it in place ----
#pragma unroll
        for (int i = 0; i < RL; ++i) {
            const int r = lane + 32 * i;
            if constexpr (fmt_u4(FMT)) {
                uint32_t w[4];
                const uint32_t szw = quantize_group_u4(x[i], w);
                if (r < lo) {
                    stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                    stg32(grec + p.meta_off + 4 * r, szw);
                }
            } else if constexpr (FMT == kFmtE4M3) {
                float2 xn[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) xn[j] = mul2(x[i][j], splat2(kUp));  // natural domain (exact)
                uint32_t w[8];
                const float sc = quantize_group_e4m3(xn, w);
                if (r < lo) {
                    stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                    stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                    stg32(grec + p.meta_off + 4 * r, __float_as_uint(sc));
                }
            } else {
                float mn, mx, inv, zq;
                minmax32(x[i], mn, mx);
                const float sc = scale_of(mn, mx);
                const uint32_t szw = sc == 0.0f ? affine_params_scaled(mn, mx, inv, zq) : affine_finish(sc, mn, inv, zq);
                const float2 inv2 = splat2(inv * 0x1p-110f), zc2 = splat2(zq * 0x1p-149f);
                uint32_t w[8];
#pragma unroll
                for (int m = 0; m < 8; ++m) w[m] = encode4(x[i][2 * m], x[i][2 * m + 1], inv2, zc2);
                if (r < lo) {
                    stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                    stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                    stg32(grec + p.meta_off + 4 * r, szw);
                }
            }
        }
        for (int u = 0; u < K; u += 2) {
            const float f0 = ldsf(hbuf + 4 * (32 * u + lane));
            const float f1 = u + 1 < K ? ldsf(hbuf + 4 * (32 * (u + 1) + lane)) : 0.f;  // odd K: padding half 0
            stg32(grec + hi_elem_off(u, lane), f2_to_h2(f0, f1));
        }
    }
    cp_async_wait_all();
    if (bad_slot && lane == 0) atomicOr(p.status, (uint32_t)kDevBadSlot);
}

}  // namespace damp
