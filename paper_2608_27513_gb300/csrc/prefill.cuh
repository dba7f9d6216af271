// prefill.cuh -- one prefill chunk on the packed state (App. A.5, "Prefill path").
//
// The recurrence runs in FP32 over the chunk's tokens (Eq. delta_update per token,
// o_t = S_t^T q_t) and the chunk-final state is quantized once, straight into the
// packed cache that decode steps and later chunks read.
//
// Work unit = tile (slot, head, value block c): all d_k rows x 32 columns, for the
// whole chunk of that slot.  One warp owns a tile from load to store, so its FP32
// state never leaves the SM between tokens.  Lane l holds packed rows l, l+32, ...
// (32 columns each) in registers, FP16 rows and low-tier rows alike, all scaled by
// 2^-39 as in the decode step.  With the H_32 formats every row is kept in the
// transformed domain S~ = S H while the chunk runs: the low-tier rows are stored
// that way, and the FP16 rows are transformed once on load and back once on store
// (H_32 is symmetric and orthonormal, and decay and the rank-1 update are
// row/column scalings that commute with it), so the per-token work is the same for
// every row: decay, partial sums of r~ = S~^T k and p~ = S~^T q, column sums,
// H d = H v - r~ and the update; o_t takes one lane butterfly.  The next token's
// operands (q, k, g, v block, beta) stream into a double buffer by cp.async while
// the current token runs, and the next tile's record comes in by one bulk copy
// (TMA engine) while the current tile runs its tokens.  After the last token the
// low-tier rows are requantized like a decode step and the FP16 rows rounded once;
// both go back with plain stores.
#pragma once

#include "damp_common.cuh"
#include "formats.cuh"

namespace damp {

// Per-warp shared memory of the chunk kernel, fixed by (d_k, decay kind, input type):
// [column-sum buffer][H d][pi][token buffer 0][token buffer 1], each token buffer
// [q][k][g (KDA: d_k floats; GDN: one)][v block][beta].
struct PrefillSmem {
    int dvec_off, perm_off, ops_off, off_q, off_k, off_g, off_v, off_beta, ops_bytes, warp_bytes;
};
__host__ __device__ constexpr int up16(int x) { return (x + 15) & ~15; }
__host__ __device__ constexpr PrefillSmem prefill_smem(int dk, bool kda, bool bf16) {
    const int esz = bf16 ? 2 : 4;
    const int dvec = 32 * kPartStride * 4, perm = dvec + 32 * 4, ops = perm + up16(dk);
    const int oq = 0, ok = up16(dk * esz), og = 2 * up16(dk * esz), ov = og + (kda ? up16(dk * 4) : 16);
    const int ob = ov + up16(kG * esz), bytes = ob + 16;
    return PrefillSmem{dvec, perm, ops, oq, ok, og, ov, ob, bytes, (ops + 2 * bytes + 127) & ~127};
}

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
    int32_t Hm;                // heads of the operands: held head h is model head head_map[h] (or h)
    const int32_t *head_map;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes, total_tiles;
    int32_t warp_stride;  // per-warp shared memory: the fixed buffers, an mbarrier and the record stage
    int32_t amax_off;     // row-absmax format: the groups' row-maximum buffers after the warps' areas
    // per-warp shared memory
    uint32_t *status;
};

__device__ __forceinline__ uint32_t lds_u8(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u8 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
// bf16 at shared address a, widened to FP32 (exact)
__device__ __forceinline__ float lds_bf16(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=r"(v) : "r"(a));
    return __uint_as_float(v << 16);
}

// The same column sums with the pairs stored as they sit in registers (no
// repacking into (a, b) quads).  Lane l writes its row as [a 32 floats][b 32
// floats] at a stride of kPairStride floats (2 mod 32: a half-warp's 64-bit
// stores cover the 32 banks once); lane j < 16 then sums columns (2j, 2j+1) of a
// over the 32 rows and lane 16 + j the same columns of b, and four shuffles hand
// every lane its own column.  Needs 32 * kPairStride floats at part.
constexpr int kPairStride = 66;
static_assert(kPairStride <= kPartStride, "column_sum_pairs uses the column_sum2 buffer");
__device__ __forceinline__ float2 column_sum_pairs(const float2 (&a)[16], const float2 (&b)[16], uint32_t part,
                                                   int lane) {
    const uint32_t row = part + (uint32_t)(lane * kPairStride * 4);
#pragma unroll
    for (int m = 0; m < 16; ++m) {
        asm volatile("st.shared.v2.f32 [%0], {%1,%2};" ::"r"(row + 8 * m), "f"(a[m].x), "f"(a[m].y) : "memory");
        asm volatile("st.shared.v2.f32 [%0], {%1,%2};" ::"r"(row + 128 + 8 * m), "f"(b[m].x), "f"(b[m].y) : "memory");
    }
    __syncwarp();
    const uint32_t base = part + (uint32_t)(((lane >> 4) * 32 + 2 * (lane & 15)) * 4);
    float2 s0 = make_float2(0.f, 0.f), s1 = s0, s2 = s0, s3 = s0;
#pragma unroll
    for (int l = 0; l < 32; l += 4) {
        float2 v0, v1, v2, v3;
        asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v0.x), "=f"(v0.y) : "r"(base + (l + 0) * kPairStride * 4));
        asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v1.x), "=f"(v1.y) : "r"(base + (l + 1) * kPairStride * 4));
        asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v2.x), "=f"(v2.y) : "r"(base + (l + 2) * kPairStride * 4));
        asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v3.x), "=f"(v3.y) : "r"(base + (l + 3) * kPairStride * 4));
        s0 = add2(s0, v0);
        s1 = add2(s1, v1);
        s2 = add2(s2, v2);
        s3 = add2(s3, v3);
    }
    __syncwarp();
    const float2 t = add2(add2(s0, s1), add2(s2, s3));
    const int src = lane >> 1;
    const float ax = __shfl_sync(kFull, t.x, src), ay = __shfl_sync(kFull, t.y, src);
    const float bx = __shfl_sync(kFull, t.x, 16 + src), by = __shfl_sync(kFull, t.y, 16 + src);
    return (lane & 1) ? make_float2(ay, by) : make_float2(ax, bx);
}

// Row-absmax INT8 (format 2): x_j = s q_j * scale from 8 words of int8 codes (the
// codes offset by 128 land on the UINT8 path's 2^23 + byte trick; s q is exact).
__device__ __forceinline__ void dequantize_row_s8(const uint32_t (&w)[8], float s, float scale, float2 (&x)[16]) {
    const float2 nzb = splat2(-(8388608.0f + 128.0f));
    const float2 sa = splat2(s * scale);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const uint32_t u = w[i] ^ 0x80808080u;  // q + 128 in [1, 255]
        x[2 * i] = mul2(add2(make_float2(u8_biased(u, 0), u8_biased(u, 1)), nzb), sa);
        x[2 * i + 1] = mul2(add2(make_float2(u8_biased(u, 2), u8_biased(u, 3)), nzb), sa);
    }
}

// FP16 row u of a record held in shared memory at rec -> 32 FP32 values
// (component j of the group is y[j/2].x or .y).  Row pair u>>1 holds one 32-bit
// word per column, row u in half u & 1.
__device__ __forceinline__ void load_hi_row(uint32_t rec, int u, float2 (&y)[16]) {
    const uint32_t pr = rec + (uint32_t)hi_elem_off(u & ~1, 0);
    const uint32_t sel = (u & 1) ? 0x7632u : 0x5410u;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const uint4 w = lds128(pr + 16 * q);
        y[2 * q] = h2_to_f2(prmt(w.x, w.y, sel));
        y[2 * q + 1] = h2_to_f2(prmt(w.z, w.w, sel));
    }
}

// Store FP16 row u (binary16 pairs own[m] = columns 2m, 2m+1) into its row pair.
// Lanes 2i and 2i+1 (u = lane + 32 i) hold the two rows of a pair: they swap half
// of their words so that the even lane writes columns 0..15 and the odd lane
// columns 16..31, each as 64 contiguous bytes.  Every lane of the warp must call
// this (shuffles); pairs past the FP16 tier store nothing, and the odd half of the
// last pair of an odd K (row K, padding) is written as 0.
__device__ __forceinline__ void store_hi_row(uint8_t *grec, int u, int K, int lane, const uint32_t (&own)[16]) {
    const bool odd = lane & 1;
    uint32_t recv[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) recv[m] = __shfl_xor_sync(kFull, odd ? own[m] : own[8 + m], 1);
    const int ue = u & ~1;  // even row of the pair
    if (ue >= K) return;
    const bool pad = ue + 1 >= K;
    uint32_t w[16];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        const uint32_t ev = odd ? recv[m] : own[m];
        const uint32_t od = pad ? 0u : (odd ? own[8 + m] : recv[m]);
        w[2 * m] = prmt(ev, od, 0x5410u);
        w[2 * m + 1] = prmt(ev, od, 0x7632u);
    }
    uint8_t *pr = grec + hi_elem_off(u & ~1, 0) + (odd ? 64 : 0);
#pragma unroll
    for (int q = 0; q < 4; ++q) stg128(pr + 16 * q, make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]));
}

// the 32-vector H d of the pending update (lane j wrote component j)
__device__ __forceinline__ void load_dvec(uint32_t dvec, float2 (&d)[16]) {
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
        const uint4 w = lds128(dvec + 16 * jj);
        d[2 * jj] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
        d[2 * jj + 1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
    }
}

// R = d_k / 32: packed rows per lane (row u = lane + 32 i), fixed at compile time.
template <int R, bool KDA, int FMT, bool BF16>
__global__ void __launch_bounds__(256, 1) prefill_chunk_kernel(const PrefillParams p) {
    constexpr bool HAD = fmt_had(FMT);
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const LaneSigns sg = lane_signs(lane);
    constexpr PrefillSmem SM = prefill_smem(32 * R, KDA, BF16);
    const uint32_t ws = smem_u32(smem) + (uint32_t)(warp * p.warp_stride);
    const uint32_t bar = ws + SM.warp_bytes;  // completion of the record copy
    const uint32_t st = bar + 128;            // the record of the current tile
    const uint32_t part = ws;  // column-sum buffer at the start of the warp's area
    const uint32_t dvec = ws + SM.dvec_off;
    const uint32_t perm_s = ws + SM.perm_off;
    const uint32_t ops0 = ws + SM.ops_off;
    const int esz = BF16 ? 2 : 4;
    constexpr int dk = 32 * R;
    const int K = p.K, lo = dk - K, H = p.H, V = p.V, T = p.T;

    const int64_t gw = (int64_t)blockIdx.x * nw + warp;
    const int64_t nwt = (int64_t)gridDim.x * nw;
    const int64_t t0 = p.total_tiles * gw / nwt, t1 = p.total_tiles * (gw + 1) / nwt;
    if (t0 >= t1) return;
    bool bad_slot = false, bad_head = false, timed_out = false;

    // The record of the next tile comes in by one bulk copy (TMA engine) while the
    // current tile runs its tokens; tiles that are skipped (slot out of range, no
    // tokens) complete their phase with no bytes.
    auto rec_of = [&](int64_t tt, int &b, int &h, int &c, int &mh, int64_t &slot, int &Tb) -> uint8_t * {
        c = (int)(tt % V);
        const int64_t bh = tt / V;
        h = (int)(bh % H);
        b = (int)(bh / H);
        mh = p.head_map ? p.head_map[h] : h;  // model head of the operands
        slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        Tb = p.lengths ? min(max(p.lengths[b], 0), T) : T;
        return p.state + slot * p.slot_bytes + (int64_t)(h * V + c) * p.rec_bytes;
    };
    auto issue = [&](int64_t tt) {  // lane 0
        int b, h, c, mh, Tb;
        int64_t slot;
        uint8_t *g = rec_of(tt, b, h, c, mh, slot, Tb);
        const bool run = slot >= 0 && slot < p.num_slots && mh >= 0 && mh < p.Hm && Tb > 0;
        mbar_arrive_expect_tx(bar, run ? (uint32_t)p.rec_bytes : 0u);
        if (run) bulk_g2s(st, g, (uint32_t)p.rec_bytes, bar);
    };
    if (lane == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
        issue(t0);
    }
    __syncwarp();
    uint32_t parity = 0;

    for (int64_t t = t0; t < t1; ++t) {
        if (!__all_sync(kFull, mbar_wait_bounded(bar, parity))) {
            timed_out = true;
            break;
        }
        parity ^= 1u;
        int b, h, c, mh, Tb;
        int64_t slot;
        uint8_t *const grec = rec_of(t, b, h, c, mh, slot, Tb);  // written in place
        const bool slot_ok = slot >= 0 && slot < p.num_slots, head_ok = mh >= 0 && mh < p.Hm;
        bad_slot |= !slot_ok;
        bad_head |= !head_ok;
        if (!slot_ok || !head_ok || Tb == 0) {  // nothing landed in the stage: fetch the next record
            if (lane == 0 && t + 1 < t1) issue(t + 1);
            continue;
        }

        // token 0's operands of this tile and their per-token strides (in bytes)
        const int Hm = p.Hm;
        const int hq = (int)(((int64_t)mh * p.Hqk) / Hm);
        const uint8_t *qt = (const uint8_t *)p.q + ((int64_t)b * T * p.Hqk + hq) * dk * esz;
        const uint8_t *kt = (const uint8_t *)p.k + ((int64_t)b * T * p.Hqk + hq) * dk * esz;
        const uint8_t *gt = (const uint8_t *)(p.g + ((int64_t)b * T * Hm + mh) * (KDA ? dk : 1));
        const uint8_t *vt = (const uint8_t *)p.v + (((int64_t)b * T * Hm + mh) * p.dv + kG * c) * esz;
        const uint8_t *bt = (const uint8_t *)(p.beta + (int64_t)b * T * Hm + mh);
        float *ot = p.o + ((int64_t)b * T * Hm + mh) * p.dv + kG * c + lane;
        const int64_t sqk = (int64_t)p.Hqk * dk * esz, sg4 = (int64_t)Hm * (KDA ? dk : 1) * 4,
                      sv = (int64_t)Hm * p.dv * esz, sb = (int64_t)Hm * 4, so = (int64_t)Hm * p.dv;
        // one token's operands into buffer dst: every copy is 16 B (beta and the GDN
        // gate 4 B); the copy counts are compile-time constants
        auto load_token = [&](int tok, uint32_t dst) {
            constexpr int nq = dk * (BF16 ? 2 : 4) / 16, ng = KDA ? dk * 4 / 16 : 0, nv = kG * (BF16 ? 2 : 4) / 16;
            const uint8_t *qs = qt + tok * sqk, *ks = kt + tok * sqk, *gs = gt + tok * sg4, *vs = vt + tok * sv;
#pragma unroll
            for (int j = lane; j < nq; j += 32) cp_async16(dst + SM.off_q + 16 * j, qs + 16 * j);
#pragma unroll
            for (int j = lane; j < nq; j += 32) cp_async16(dst + SM.off_k + 16 * j, ks + 16 * j);
#pragma unroll
            for (int j = lane; j < ng; j += 32) cp_async16(dst + SM.off_g + 16 * j, gs + 16 * j);
#pragma unroll
            for (int j = lane; j < nv; j += 32) cp_async16(dst + SM.off_v + 16 * j, vs + 16 * j);
            if (lane == 0) {
                cp_async4(dst + SM.off_beta, bt + tok * sb);
                if (!KDA) cp_async4(dst + SM.off_g, gs);
            }
            cp_async_commit();
        };

        // π of this head, then token 0's operands
        __syncwarp();  // the previous tile's readers of the shared buffers are done
        for (int ci = lane; ci < dk / 16; ci += 32) cp_async16(perm_s + 16 * ci, p.perm + (int64_t)h * dk + 16 * ci);
        load_token(0, ops0);

        // ---- reconstruct the tile in FP32, undecayed, scaled by 2^-39; with H_32 in
        //      the transformed domain (FP16 rows transformed here) ----
        // low-tier words of every row slot first (rows of the FP16 tier load a valid
        // low row and ignore it), so that all loads are in flight before the branches
        float2 x[R][16];
        uint4 cw0[R], cw1[R];
        uint32_t szw[R];
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int r = lo > 0 ? min(max(lane + 32 * i - K, 0), lo - 1) : 0;
            const uint32_t crow = st + (uint32_t)(lo > 0 ? p.codes_off : 0);  // lo = 0: a valid dummy address
            cw0[i] = lds128(crow + lo_chunk_off(r, 0, lo));
            cw1[i] = fmt_u4(FMT) ? cw0[i] : lds128(crow + lo_chunk_off(r, 1, lo));
            szw[i] = lds32(st + (uint32_t)(lo > 0 ? p.meta_off + 4 * r : 0));
        }
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int u = lane + 32 * i;
            if (u < K) {
                load_hi_row(st, u, x[i]);
                if (HAD) hadamard_pairs(x[i]);
#pragma unroll
                for (int j = 0; j < 16; ++j) x[i][j] = mul2(x[i][j], splat2(kDown));  // exact
                continue;
            }
            if constexpr (fmt_u4(FMT)) {
                const uint32_t w[4] = {cw0[i].x, cw0[i].y, cw0[i].z, cw0[i].w};
                dequantize_group_u4(w, szw[i], kDown, x[i]);
            } else {
                const uint32_t w[8] = {cw0[i].x, cw0[i].y, cw0[i].z, cw0[i].w, cw1[i].x, cw1[i].y, cw1[i].z, cw1[i].w};
                if constexpr (FMT == kFmtE4M3) dequantize_group_e4m3(w, __uint_as_float(szw[i]), kDown, x[i]);
                else dequantize_group(w, szw[i], kDown, x[i]);
            }
        }

        // the stage has been read: the next tile's record comes in during this one
        __syncwarp();
        if (lane == 0 && t + 1 < t1) {
            fence_proxy_async_smem();  // the warp's reads of the stage before the bulk copy's writes
            issue(t + 1);
        }

        // The rank-1 update of token t is applied at the start of token t+1, in the
        // same pass over the registers as that token's decay (and after the loop for
        // the last token): H d of the pending update waits in dvec, beta k in bkp.
        // o_t = H (p~ - beta (k^T q) r~) + beta (k^T q) v (all rows in the transformed
        // domain; H = I without H_32) is finished during token t+1, off the path of
        // the recurrence: o_pend and o_add hold its two parts.
        float2 bkp[R];
#pragma unroll
        for (int i = 0; i < R; ++i) bkp[i] = make_float2(0.f, 0.f);
        sts32(dvec + 4 * lane, 0u);
        float o_pend = 0.f, o_add = 0.f;
        auto finish_o = [&]() { return (HAD ? hadamard_lanes(o_pend, sg) : o_pend) + o_add; };
        for (int tok = 0; tok < Tb; ++tok) {
            const uint32_t ob = ops0 + (uint32_t)((tok & 1) * SM.ops_bytes);
            cp_async_wait_all();
            __syncwarp();
            if (tok + 1 < Tb) load_token(tok + 1, ops0 + (uint32_t)(((tok + 1) & 1) * SM.ops_bytes));

            // ---- operands of this lane's rows, in calibrated order ----
            const float beta = ldsf(ob + SM.off_beta);
            const float alpha = KDA ? 0.f : expf(ldsf(ob + SM.off_g));
            float2 kk[R], qq[R], bk[R], aa[R];
            float kq = 0.f;
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int u = lane + 32 * i;
                const uint32_t ch = lds_u8(perm_s + u) & (dk - 1);
                const float kv = BF16 ? lds_bf16(ob + SM.off_k + 2 * ch) : ldsf(ob + SM.off_k + 4 * ch);
                const float qv = BF16 ? lds_bf16(ob + SM.off_q + 2 * ch) : ldsf(ob + SM.off_q + 4 * ch);
                kk[i] = splat2(kv);
                qq[i] = splat2(qv);
                bk[i] = splat2(beta * kv * kDown);
                aa[i] = splat2(KDA ? expf(ldsf(ob + SM.off_g + 4 * ch)) : alpha);
                kq = fmaf(kv, qv, kq);
            }
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) kq += __shfl_xor_sync(kFull, kq, m);
            const float bkq = beta * kq;
            const float vj = BF16 ? lds_bf16(ob + SM.off_v + 2 * lane) : ldsf(ob + SM.off_v + 4 * lane);
            const float hv = HAD ? hadamard_lanes(vj, sg) : vj;  // H v: independent of the state
            // o of token tok - 1 (meaningless at tok = 0, not stored): computed here without a
            // branch, so that its butterfly and that of H v overlap the pass over the registers
            const float o_prev = finish_o();

            // ---- the previous token's update, decay and partial sums ----
            float2 d[16];
            load_dvec(dvec, d);
            float2 acc[16], accp[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] = accp[j] = make_float2(0.f, 0.f);
#pragma unroll
            for (int i = 0; i < R; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    x[i][j] = mul2(fma2(bkp[i], d[j], x[i][j]), aa[i]);
                    acc[j] = fma2(x[i][j], kk[i], acc[j]);
                    accp[j] = fma2(x[i][j], qq[i], accp[j]);
                }
            }
            const float2 sums = column_sum_pairs(acc, accp, part, lane);
            const float rs = sums.x * kUp, ps = sums.y * kUp;

            // ---- the column vector of the update, H d = H v - r~, and o_t's parts ----
            sts32(dvec + 4 * lane, __float_as_uint(hv - rs));
            if (tok > 0) ot[(tok - 1) * so] = o_prev;
            o_pend = fmaf(-bkq, rs, ps);
            o_add = bkq * vj;
#pragma unroll
            for (int i = 0; i < R; ++i) bkp[i] = bk[i];
        }
        ot[(Tb - 1) * so] = finish_o();
        {  // the last token's update
            __syncwarp();
            float2 d[16];
            load_dvec(dvec, d);
#pragma unroll
            for (int i = 0; i < R; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) x[i][j] = fma2(bkp[i], d[j], x[i][j]);
            }
        }

        // ---- the chunk-final tile: FP16 rows rounded once, low-tier rows requantized ----
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int u = lane + 32 * i;
            if (32 * i < K) {  // warp-uniform: some lanes of this slot hold FP16 rows
                float2 y[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) y[j] = x[i][j];
                if (HAD) hadamard_pairs(y);  // back to the natural domain
                uint32_t own[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) own[j] = f2_to_h2(y[j].x * kUp, y[j].y * kUp);
                store_hi_row(grec, u, K, lane, own);
            }
            if (u < K) continue;
            const int r = u - K;
            if constexpr (fmt_u4(FMT)) {
                uint32_t w[4];
                const uint32_t szw = quantize_group_u4(x[i], w);
                stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                stg32(grec + p.meta_off + 4 * r, szw);
            } else if constexpr (FMT == kFmtE4M3) {
                float2 xn[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) xn[j] = mul2(x[i][j], splat2(kUp));  // natural domain (exact)
                uint32_t w[8];
                const float sc = quantize_group_e4m3(xn, w);
                stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                stg32(grec + p.meta_off + 4 * r, __float_as_uint(sc));
            } else {
                float mn, mx, inv, zq;
                minmax32(x[i], mn, mx);
                const float sc = scale_of(mn, mx);
                const uint32_t szw = sc == 0.0f ? affine_params_scaled(mn, mx, inv, zq) : affine_finish(sc, mn, inv, zq);
                const float2 inv2 = splat2(inv * 0x1p-110f), zc2 = splat2(zq * 0x1p-149f);
                uint32_t w[8];
#pragma unroll
                for (int m = 0; m < 8; ++m) w[m] = encode4(x[i][2 * m], x[i][2 * m + 1], inv2, zc2);
                stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                stg32(grec + p.meta_off + 4 * r, szw);
            }
        }
    }
    if (timed_out) mbar_wait_bounded(bar, parity);  // the copy in flight lands (bounded) before the CTA ends
    cp_async_wait_all();
    if (lane == 0) {
        const uint32_t bits =
            (timed_out ? kDevWaitTimeout : 0u) | (bad_slot ? kDevBadSlot : 0u) | (bad_head ? kDevBadHead : 0u);
        if (bits) atomicOr(p.status, bits);
    }
}

// The row-absmax format (2) in the chunk kernel.  Its row scale spans the V <= 4 value
// blocks of a head, so a group of four warps takes a range of (slot, head) units, warp
// 4g + c the value block c of each, and after the last token the group meets at a named
// barrier to combine each row's maximum; warps with c >= V, and a warp whose record copy
// timed out, keep meeting the group without computing, so no barrier waits on a warp
// that left.  R = d_k / 32 as in prefill_chunk_kernel; no H_32 in this format.
template <int R, bool KDA, bool BF16>
__global__ void __launch_bounds__(256, 1) prefill_row_kernel(const PrefillParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    constexpr PrefillSmem SM = prefill_smem(32 * R, KDA, BF16);
    const uint32_t ws = smem_u32(smem) + (uint32_t)(warp * p.warp_stride);
    const uint32_t bar = ws + SM.warp_bytes;  // completion of the record copy
    const uint32_t st = bar + 128;            // the record of the current tile
    const uint32_t part = ws;  // column-sum buffer at the start of the warp's area
    const uint32_t dvec = ws + SM.dvec_off;
    const uint32_t perm_s = ws + SM.perm_off;
    const uint32_t ops0 = ws + SM.ops_off;
    const int esz = BF16 ? 2 : 4;
    constexpr int dk = 32 * R;
    const int K = p.K, lo = dk - K, H = p.H, V = p.V, T = p.T;

    // the group's range of (slot, head) units; this warp's value block cw
    const int cw = warp & 3;
    const bool idle = cw >= V;
    const int64_t ng = (int64_t)gridDim.x * (nw >> 2), g = (int64_t)blockIdx.x * (nw >> 2) + (warp >> 2);
    const int64_t units = p.total_tiles / V;
    const int64_t u0 = units * g / ng, n = units * (g + 1) / ng - u0;
    // the tile of step k (for an idle warp: block 0 of its unit, whose batch row and head
    // decide, as for the group's other warps, whether the unit runs)
    auto tile_of = [&](int64_t k) -> int64_t { return (u0 + k) * V + (idle ? 0 : cw); };
    if (n <= 0) return;  // the same for the four warps of a group
    const uint32_t amax_s = smem_u32(smem) + (uint32_t)(p.amax_off + (warp >> 2) * 2 * 4 * 128 * 4);
    auto group_sync = [&]() { asm volatile("bar.sync %0, 128;" ::"r"(1 + (warp >> 2)) : "memory"); };
    bool bad_slot = false, bad_head = false, timed_out = false;

    // The record of the next tile comes in by one bulk copy (TMA engine) while the
    // current tile runs its tokens; tiles that are skipped (slot out of range, no
    // tokens) complete their phase with no bytes.
    auto rec_of = [&](int64_t tt, int &b, int &h, int &c, int &mh, int64_t &slot, int &Tb) -> uint8_t * {
        c = (int)(tt % V);
        const int64_t bh = tt / V;
        h = (int)(bh % H);
        b = (int)(bh / H);
        mh = p.head_map ? p.head_map[h] : h;  // model head of the operands
        slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        Tb = p.lengths ? min(max(p.lengths[b], 0), T) : T;
        return p.state + slot * p.slot_bytes + (int64_t)(h * V + c) * p.rec_bytes;
    };
    auto issue = [&](int64_t k) {  // lane 0: the record of step k
        int b, h, c, mh, Tb;
        int64_t slot;
        uint8_t *g = rec_of(tile_of(k), b, h, c, mh, slot, Tb);
        const bool run = !idle && slot >= 0 && slot < p.num_slots && mh >= 0 && mh < p.Hm && Tb > 0;
        mbar_arrive_expect_tx(bar, run ? (uint32_t)p.rec_bytes : 0u);
        if (run) bulk_g2s(st, g, (uint32_t)p.rec_bytes, bar);
    };
    if (lane == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
        issue(0);
    }
    __syncwarp();
    uint32_t parity = 0;

    for (int64_t k = 0; k < n; ++k) {
        // A lost copy ends this warp's work; in a row-absmax group it keeps meeting the
        // other warps (no compute) so that no barrier waits for it.
        if (!timed_out && !__all_sync(kFull, mbar_wait_bounded(bar, parity))) timed_out = true;
        if (!timed_out) parity ^= 1u;
        int b, h, c, mh, Tb;
        int64_t slot;
        uint8_t *const grec = rec_of(tile_of(k), b, h, c, mh, slot, Tb);  // written in place
        const bool slot_ok = slot >= 0 && slot < p.num_slots, head_ok = mh >= 0 && mh < p.Hm;
        bad_slot |= !slot_ok;
        bad_head |= !head_ok;
        if (!slot_ok || !head_ok || Tb == 0) {  // nothing landed in the stage: fetch the next record
            if (lane == 0 && k + 1 < n && !timed_out) issue(k + 1);
            continue;
        }
        if (idle || timed_out) {  // the unit runs: meet the group once, at its row maxima
            if (lane == 0 && k + 1 < n && !timed_out) issue(k + 1);
            group_sync();
            continue;
        }

        // token 0's operands of this tile and their per-token strides (in bytes)
        const int Hm = p.Hm;
        const int hq = (int)(((int64_t)mh * p.Hqk) / Hm);
        const uint8_t *qt = (const uint8_t *)p.q + ((int64_t)b * T * p.Hqk + hq) * dk * esz;
        const uint8_t *kt = (const uint8_t *)p.k + ((int64_t)b * T * p.Hqk + hq) * dk * esz;
        const uint8_t *gt = (const uint8_t *)(p.g + ((int64_t)b * T * Hm + mh) * (KDA ? dk : 1));
        const uint8_t *vt = (const uint8_t *)p.v + (((int64_t)b * T * Hm + mh) * p.dv + kG * c) * esz;
        const uint8_t *bt = (const uint8_t *)(p.beta + (int64_t)b * T * Hm + mh);
        float *ot = p.o + ((int64_t)b * T * Hm + mh) * p.dv + kG * c + lane;
        const int64_t sqk = (int64_t)p.Hqk * dk * esz, sg4 = (int64_t)Hm * (KDA ? dk : 1) * 4,
                      sv = (int64_t)Hm * p.dv * esz, sb = (int64_t)Hm * 4, so = (int64_t)Hm * p.dv;
        // one token's operands into buffer dst: every copy is 16 B (beta and the GDN
        // gate 4 B); the copy counts are compile-time constants
        auto load_token = [&](int tok, uint32_t dst) {
            constexpr int nq = dk * (BF16 ? 2 : 4) / 16, ng = KDA ? dk * 4 / 16 : 0, nv = kG * (BF16 ? 2 : 4) / 16;
            const uint8_t *qs = qt + tok * sqk, *ks = kt + tok * sqk, *gs = gt + tok * sg4, *vs = vt + tok * sv;
#pragma unroll
            for (int j = lane; j < nq; j += 32) cp_async16(dst + SM.off_q + 16 * j, qs + 16 * j);
#pragma unroll
            for (int j = lane; j < nq; j += 32) cp_async16(dst + SM.off_k + 16 * j, ks + 16 * j);
#pragma unroll
            for (int j = lane; j < ng; j += 32) cp_async16(dst + SM.off_g + 16 * j, gs + 16 * j);
#pragma unroll
            for (int j = lane; j < nv; j += 32) cp_async16(dst + SM.off_v + 16 * j, vs + 16 * j);
            if (lane == 0) {
                cp_async4(dst + SM.off_beta, bt + tok * sb);
                if (!KDA) cp_async4(dst + SM.off_g, gs);
            }
            cp_async_commit();
        };

        // π of this head, then token 0's operands
        __syncwarp();  // the previous tile's readers of the shared buffers are done
        for (int ci = lane; ci < dk / 16; ci += 32) cp_async16(perm_s + 16 * ci, p.perm + (int64_t)h * dk + 16 * ci);
        load_token(0, ops0);

        // ---- reconstruct the tile in FP32, undecayed, scaled by 2^-39; with H_32 in
        //      the transformed domain (FP16 rows transformed here) ----
        // low-tier words of every row slot first (rows of the FP16 tier load a valid
        // low row and ignore it), so that all loads are in flight before the branches
        float2 x[R][16];
        uint4 cw0[R], cw1[R];
        uint32_t szw[R];
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int r = lo > 0 ? min(max(lane + 32 * i - K, 0), lo - 1) : 0;
            const uint32_t crow = st + (uint32_t)(lo > 0 ? p.codes_off : 0);  // lo = 0: a valid dummy address
            cw0[i] = lds128(crow + lo_chunk_off(r, 0, lo));
            cw1[i] = lds128(crow + lo_chunk_off(r, 1, lo));
            szw[i] = lds32(st + (uint32_t)(lo > 0 ? p.meta_off + 4 * r : 0));
        }
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int u = lane + 32 * i;
            if (u < K) {
                load_hi_row(st, u, x[i]);
#pragma unroll
                for (int j = 0; j < 16; ++j) x[i][j] = mul2(x[i][j], splat2(kDown));  // exact
                continue;
            }
            const uint32_t w[8] = {cw0[i].x, cw0[i].y, cw0[i].z, cw0[i].w, cw1[i].x, cw1[i].y, cw1[i].z, cw1[i].w};
            dequantize_row_s8(w, __uint_as_float(szw[i]), kDown, x[i]);
        }

        // the stage has been read: the next tile's record comes in during this one
        __syncwarp();
        if (lane == 0 && k + 1 < n) {
            fence_proxy_async_smem();  // the warp's reads of the stage before the bulk copy's writes
            issue(k + 1);
        }

        // The rank-1 update of token t is applied at the start of token t+1, in the
        // same pass over the registers as that token's decay (and after the loop for
        // the last token): H d of the pending update waits in dvec, beta k in bkp.
        // o_t = H (p~ - beta (k^T q) r~) + beta (k^T q) v (all rows in the transformed
        // domain; H = I without H_32) is finished during token t+1, off the path of
        // the recurrence: o_pend and o_add hold its two parts.
        float2 bkp[R];
#pragma unroll
        for (int i = 0; i < R; ++i) bkp[i] = make_float2(0.f, 0.f);
        sts32(dvec + 4 * lane, 0u);
        float o_pend = 0.f, o_add = 0.f;
        auto finish_o = [&](int tok) {
            ot[tok * so] = o_pend + o_add;
        };
        for (int tok = 0; tok < Tb; ++tok) {
            const uint32_t ob = ops0 + (uint32_t)((tok & 1) * SM.ops_bytes);
            cp_async_wait_all();
            __syncwarp();
            if (tok + 1 < Tb) load_token(tok + 1, ops0 + (uint32_t)(((tok + 1) & 1) * SM.ops_bytes));

            // ---- operands of this lane's rows, in calibrated order ----
            const float beta = ldsf(ob + SM.off_beta);
            const float alpha = KDA ? 0.f : expf(ldsf(ob + SM.off_g));
            float2 kk[R], qq[R], bk[R], aa[R];
            float kq = 0.f;
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int u = lane + 32 * i;
                const uint32_t ch = lds_u8(perm_s + u) & (dk - 1);
                const float kv = BF16 ? lds_bf16(ob + SM.off_k + 2 * ch) : ldsf(ob + SM.off_k + 4 * ch);
                const float qv = BF16 ? lds_bf16(ob + SM.off_q + 2 * ch) : ldsf(ob + SM.off_q + 4 * ch);
                kk[i] = splat2(kv);
                qq[i] = splat2(qv);
                bk[i] = splat2(beta * kv * kDown);
                aa[i] = splat2(KDA ? expf(ldsf(ob + SM.off_g + 4 * ch)) : alpha);
                kq = fmaf(kv, qv, kq);
            }
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) kq += __shfl_xor_sync(kFull, kq, m);
            const float bkq = beta * kq;
            const float vj = BF16 ? lds_bf16(ob + SM.off_v + 2 * lane) : ldsf(ob + SM.off_v + 4 * lane);
            const float hv = vj;  // natural domain
            if (tok > 0) finish_o(tok - 1);

            // ---- the previous token's update, decay and partial sums ----
            float2 d[16];
            load_dvec(dvec, d);
            float2 acc[16], accp[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] = accp[j] = make_float2(0.f, 0.f);
#pragma unroll
            for (int i = 0; i < R; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    x[i][j] = mul2(fma2(bkp[i], d[j], x[i][j]), aa[i]);
                    acc[j] = fma2(x[i][j], kk[i], acc[j]);
                    accp[j] = fma2(x[i][j], qq[i], accp[j]);
                }
            }
            const float2 sums = column_sum_pairs(acc, accp, part, lane);
            const float rs = sums.x * kUp, ps = sums.y * kUp;

            // ---- the column vector of the update, H d = H v - r~, and o_t's parts ----
            sts32(dvec + 4 * lane, __float_as_uint(hv - rs));
            o_pend = fmaf(-bkq, rs, ps);
            o_add = bkq * vj;
#pragma unroll
            for (int i = 0; i < R; ++i) bkp[i] = bk[i];
        }
        finish_o(Tb - 1);
        {  // the last token's update
            __syncwarp();
            float2 d[16];
            load_dvec(dvec, d);
#pragma unroll
            for (int i = 0; i < R; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) x[i][j] = fma2(bkp[i], d[j], x[i][j]);
            }
        }

        // ---- the chunk-final tile: FP16 rows rounded once, low-tier rows requantized ----
        {
            // each row's maximum over the V value blocks of the head (buffer k & 1: a warp
            // writes unit k+2's maxima only after the group met at unit k+1)
            const uint32_t ab = amax_s + (uint32_t)((k & 1) * 4 * 128 * 4);
#pragma unroll
            for (int i = 0; i < R; ++i) {
                float mn, mx;
                minmax32(x[i], mn, mx);
                sts32(ab + (uint32_t)((cw * 128 + lane + 32 * i) * 4), __float_as_uint(fmaxf(-mn, mx)));
            }
            group_sync();
        }
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const int u = lane + 32 * i;
            if (32 * i < K) {  // warp-uniform: some lanes of this slot hold FP16 rows
                float2 y[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) y[j] = x[i][j];
                uint32_t own[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) own[j] = f2_to_h2(y[j].x * kUp, y[j].y * kUp);
                store_hi_row(grec, u, K, lane, own);
            }
            if (u < K) continue;
            const int r = u - K;
            {
                // s = max|x| / 127 over the whole row (FP32, IEEE division); codes
                // sat(rne(x / s)) taken as x * (1/s) + 128 on the denormal grid, then
                // moved back to int8 (a code can differ from x / s only at a rounding tie)
                const uint32_t ab = amax_s + (uint32_t)((k & 1) * 4 * 128 * 4);
                float am = 0.f;
                for (int c2 = 0; c2 < V; ++c2) am = fmaxf(am, ldsf(ab + (uint32_t)((c2 * 128 + u) * 4)));
                const float sc = __fdiv_rn(am * kUp, 127.0f);
                const float inv = sc > 0.0f ? __frcp_rn(sc) : 0.0f;
                const float2 inv2 = splat2(inv * 0x1p-110f), zc2 = splat2(128.0f * 0x1p-149f);
                uint32_t w[8];
#pragma unroll
                for (int m = 0; m < 8; ++m) w[m] = encode4(x[i][2 * m], x[i][2 * m + 1], inv2, zc2) ^ 0x80808080u;
                stg128(grec + p.codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                stg128(grec + p.codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                stg32(grec + p.meta_off + 4 * r, __float_as_uint(sc));
            }
        }
    }
    if (timed_out) mbar_wait_bounded(bar, parity);  // the copy in flight lands (bounded) before the CTA ends
    cp_async_wait_all();
    if (lane == 0) {
        const uint32_t bits =
            (timed_out ? kDevWaitTimeout : 0u) | (bad_slot ? kDevBadSlot : 0u) | (bad_head ? kDevBadHead : 0u);
        if (bits) atomicOr(p.status, bits);
    }
}

}  // namespace damp
