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
// cross-tile reduction.  One warp owns one tile at a time:
//   * UINT8 rows: lane l owns low-tier rows l, l+32, ... with all 32 columns in
//     registers, so min/max and requantization of a group are thread-local; the
//     column reductions r = S_bar^T k and o = S^T q go through shared memory.
//     The code is branch-free: lanes past the last row process a clamped row
//     with zero weights and skip its store.
//   * FP16 rows: lane j owns column j of all K_hi rows, so their part of both
//     reductions stays in the lane.
//
// Domains: the low tier stores codes of H_32-transformed rows (App. A.5).  H_32
// acts on the value axis only and is symmetric and orthonormal, so with
// S~ = S H the low-tier rows are updated in the transformed domain:
//     r = H r~_lo + r_hi,  d = v - r,  S~_t = Lambda S~ + beta k (H d)^T,
//     o = H o~_lo + o_hi.
// Low-tier rows never pass through a butterfly; only the 32-vectors r~_lo, d and
// o~_lo do (a 5-step butterfly across the warp's lanes).
//
// Pipeline: a persistent grid; every warp walks a contiguous range of tiles.
// Lane 0 keeps NSTAGE tile records in flight with 1-D bulk copies (TMA engine)
// into a per-warp ring of shared-memory stages, each with its own mbarrier, and
// refills a stage as soon as the warp has read it; the per-(slot, head) operands
// come in by per-lane cp.async one head ahead.  The updated record goes straight
// from registers to HBM with 128-bit stores (chunk-major code rows make them whole
// sectors).  Layouts with d_k = 128 and the K_hi values the launcher lists compile
// with the record geometry and the FP16-row loops fixed (KC, DKC below).
#pragma once

#include "damp_common.cuh"
#include "formats.cuh"

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
    int32_t Hm;                // heads of the operands: held head h is model head head_map[h] (or h)
    const int32_t *head_map;
    int32_t rec_bytes, codes_off, meta_off;
    int64_t slot_bytes;
    int32_t nstage, stage_bytes, warp_smem, stage0_off;
    // per-(slot, head) operand buffer (two per warp): [v row][q][k][g (KDA)][perm]
    int32_t ops_off, ops_bytes;
    int32_t off_v, off_q, off_k, off_g, off_perm;
    int32_t bytes_v, bytes_qk, bytes_g, bytes_perm;
    int64_t total_tiles;
    uint32_t *status;
};

// per-warp scratch before the stage ring
constexpr int kPartOff = 64;                              // after NSTAGE (<= 8) mbarriers
constexpr int kDvecOff = kPartOff + 32 * kPartStride * 4; // 32 floats: H d for the low tier
constexpr int kHopsOff = kDvecOff + 32 * 4;               // FP16-row operands, 32 B per row pair
__host__ __device__ constexpr int scratch_bytes(int k_hi) { return kHopsOff + 16 * ((k_hi + 7) & ~7); }

// (batch row, head, value block) of a tile index, advanced without divisions.
struct Cursor {
    int b, h, c;
};
__device__ __forceinline__ Cursor cursor_at(int64_t t, int H, int V) {
    Cursor k;
    const int64_t bh = t / V;
    k.c = (int)(t - bh * V);
    k.b = (int)(bh / H);
    k.h = (int)(bh - (int64_t)k.b * H);
    return k;
}
__device__ __forceinline__ void advance(Cursor &k, int H, int V) {
    if (++k.c == V) {
        k.c = 0;
        if (++k.h == H) {
            k.h = 0;
            ++k.b;
        }
    }
}

// RL = ceil((d_k - K_hi) / 32): low-tier row slots per lane, fixed at compile time
// so that the row loops unroll into one basic block.
// KC >= 0 fixes K_hi at compile time (KC = 0: no FP16 tier) and DKC > 0 fixes d_k:
// with both fixed, the record geometry and every row offset are constants and the
// FP16 tier runs as straight-line code.  KC = -1, DKC = 0 is the general kernel.
// HMAP: the layout is a head group (held head h reads the operands of model head
// head_map[h]); without it the model heads are the held heads.
// LT: the low tier's code type -- kLtU8 (formats 0, 1), kLtU4 (formats 3, 4: 32 nibbles
// in one 16-byte chunk per row, levels 15) or kLtE4M3 (format 5: FP8 codes in the natural
// domain, one FP32 scale per group).
// WAITTEST: a test instance, outside the decode dispatch, that exercises the bounded
// wait: every stage barrier expects kWaitTestExtra bytes more than its copy delivers,
// so the first wait runs out after kWaitTestNs; the kernel then settles those bytes
// itself, waits for the copies in flight to land, reports DAMP_DEV_WAIT_TIMEOUT and
// returns without touching a record or o.
enum : int { kLtU8 = 0, kLtU4 = 1, kLtE4M3 = 2 };
constexpr uint32_t kWaitTestExtra = 16;
constexpr uint64_t kWaitTestNs = 1000000;  // 1 ms
constexpr int kHiUnroll = 16;             // largest fixed K_hi whose FP16 sums follow the low tier
// The body runs as CTA `blk` of a grid of `nblk` CTAs; it returns true when one of the
// warp's copy waits ran out (its stage barriers are then left as they are).
// UMH (head groups): look the model head up once per (slot, head) unit and keep it in a
// register, instead of once per tile (set where the extra register costs no spills).
template <int RL, int DKC, int KC, bool KDA, bool HAD, bool BF16, bool HMAP, int LT = kLtU8, bool WAITTEST = false,
          bool UMH = false>
__device__ __forceinline__ bool packed_step_body(const PackedParams p, const int blk, const int nblk) {
    constexpr int R = RL > 0 ? RL : 1;
    extern __shared__ __align__(128) uint8_t smem[];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const LaneSigns sg = lane_signs(lane);
    const uint32_t ws = smem_u32(smem) + (uint32_t)(warp * p.warp_smem);
    const uint32_t bar0 = ws;
    const uint32_t part = ws + kPartOff;
    const uint32_t dvec = ws + kDvecOff;
    const uint32_t hops = ws + kHopsOff;
    const uint32_t stage0 = ws + p.stage0_off;
    const int esz = BF16 ? 2 : 4;
    constexpr bool KFIX = KC >= 0, DFIX = DKC > 0;
    const int K = KFIX ? KC : p.K;
    const int dk = DFIX ? DKC : p.dk;
    const int lo = dk - K;  // low-tier rows
    // record geometry (constants for a fixed layout)
    const int codes_off = KFIX ? 128 * ((KC + 1) / 2) : p.codes_off;
    constexpr bool U4 = LT == kLtU4, F8 = LT == kLtE4M3;
    constexpr int kCodeRow = U4 ? 16 : 32;  // code bytes per row and record
    const int meta_off = (KFIX && DFIX) ? 128 * ((KC + 1) / 2) + kCodeRow * (DKC - KC) : p.meta_off;
    const int rec_bytes =
        (KFIX && DFIX) ? (128 * ((KC + 1) / 2) + (kCodeRow + 4) * (DKC - KC) + 15) & ~15 : p.rec_bytes;
    // Compile-time layouts (K_hi and d_k fixed) are launched for d_v = 128 only, with three
    // record stages (the launcher checks both): the stage size, the operand buffer's layout
    // and the value-block count are then constants too.
    constexpr bool FX = KFIX && DFIX;
    constexpr bool kHiFirst = KFIX && KC > kHiUnroll;
    constexpr int FX_ESZ = BF16 ? 2 : 4;
    constexpr int FX_OFF_Q = 128 * FX_ESZ, FX_OFF_K = 256 * FX_ESZ, FX_OFF_G = 384 * FX_ESZ;
    constexpr int FX_OFF_P = FX_OFF_G + (KDA ? 512 : 0), FX_OPS = FX_OFF_P + 128;
    constexpr int FX_REC = FX ? (128 * ((KC + 1) / 2) + (kCodeRow + 4) * (DKC - KC) + 15) & ~15 : 16;
    constexpr int FX_STAGE = (FX_REC + 127) & ~127;
    const int nstage = FX ? 3 : p.nstage;
    const int stage_bytes = FX ? FX_STAGE : p.stage_bytes;
    const int ops_bytes = FX ? FX_OPS : p.ops_bytes;
    const int off_v = FX ? 0 : p.off_v, off_q = FX ? FX_OFF_Q : p.off_q, off_k = FX ? FX_OFF_K : p.off_k;
    const int off_g = FX ? FX_OFF_G : p.off_g, off_perm = FX ? FX_OFF_P : p.off_perm;
    const int dvv = FX ? 128 : p.dv;
    const int H = p.H, V = FX ? 4 : p.V;

    const int64_t gw = (int64_t)blk * nw + warp;
    const int64_t nwt = (int64_t)nblk * nw;
    const int64_t t0 = p.total_tiles * gw / nwt;
    const int64_t t1 = p.total_tiles * (gw + 1) / nwt;
    if (t0 >= t1) return false;

    if (lane == 0) {
        for (int s = 0; s < nstage; ++s) mbar_init(bar0 + 8 * s, 1);
        fence_mbar_init();
    }
    __syncwarp();

    auto slot_of = [&](int b) -> int64_t { return p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b; };
    // model head of the operands of held head h; -1 when the map entry is out of range
    auto model_head = [&](int h) -> int {
        if constexpr (!HMAP) return h;
        const int m = p.head_map[h];
        return (m >= 0 && m < p.Hm) ? m : -1;
    };
    const int Hm = HMAP ? p.Hm : H;  // heads of the operand tensors

    // ---- producer (lane 0): one bulk copy of the record of tile t (cursor k) into stage s ----
    // (a held head whose map entry is out of range still has its records in the slot: they
    // are copied and the consumer skips the tile, so no head-map load sits on this path)
    auto issue = [&](int64_t t, const Cursor &k, int s) {
        const int64_t slot = slot_of(k.b);
        const bool ok = slot >= 0 && slot < p.num_slots;
        const uint32_t st = stage0 + (uint32_t)(s * stage_bytes);
        const uint32_t bar = bar0 + 8 * s;
        mbar_arrive_expect_tx(bar, ok ? (uint32_t)rec_bytes + (WAITTEST ? kWaitTestExtra : 0u) : 0u);
        if (ok) bulk_g2s(st, p.state + slot * p.slot_bytes + (int64_t)(k.h * V + k.c) * rec_bytes, rec_bytes, bar);
    };

    // ---- per-(slot, head) operands: 16-byte copies by all lanes, one head ahead ----
    const uint32_t ops0 = ws + p.ops_off;
    auto load_ops = [&](int ub, int uh, uint32_t dst) {
        const int mh = HMAP ? max(model_head(uh), 0) : uh;  // an invalid head's tiles are skipped
        const int64_t bh = (int64_t)ub * Hm + mh;
        const int hq = (mh * p.Hqk) / Hm;
        const int nv = FX ? 8 * FX_ESZ : p.bytes_v >> 4, nq = FX ? 8 * FX_ESZ : p.bytes_qk >> 4, ng = FX ? (KDA ? 32 : 0) : p.bytes_g >> 4, np = FX ? 8 : p.bytes_perm >> 4;
        const int total = nv + 2 * nq + ng + np;
        const uint8_t *qrow = (const uint8_t *)p.q + ((int64_t)ub * p.Hqk + hq) * dk * esz;
        const uint8_t *krow = (const uint8_t *)p.k + ((int64_t)ub * p.Hqk + hq) * dk * esz;
        for (int ci = lane; ci < total; ci += 32) {
            int j = ci;
            const uint8_t *src;
            if (j < nv) {
                src = (const uint8_t *)p.v + bh * dvv * esz + 16 * j;
            } else if ((j -= nv) < nq) {
                src = qrow + 16 * j;
            } else if ((j -= nq) < nq) {
                src = krow + 16 * j;
            } else if ((j -= nq) < ng) {
                src = (const uint8_t *)(p.g + bh * dk) + 16 * j;
            } else {
                src = p.perm + (int64_t)uh * dk + 16 * (j - ng);
            }
            cp_async16(dst + 16 * ci, src);
        }
        cp_async_commit();
    };

    Cursor cur = cursor_at(t0, H, V);
    load_ops(cur.b, cur.h, ops0);
    Cursor pre = cur;  // next tile to load (lane 0)
    int64_t t_pre = t0;
    if (lane == 0) {
        fence_proxy_async_smem();  // shared memory this warp used before (a previous body) ahead of the copies
        for (int j = 0; j < nstage && t_pre < t1; ++j) {
            issue(t_pre, pre, j);
            ++t_pre;
            advance(pre, H, V);
        }
    }

    // low-tier row operands of this lane (zero weights for lanes past the last row)
    float2 kk[R], qq[R], bk[R];
    float aa[R];
    float unit_beta = 0.f, unit_g = 0.f, bkq = 0.f;
    int unit = 0;
    int unit_mh = 0;     // model head of the current (slot, head) (head groups)
    uint32_t ob = ops0;  // operand buffer of the current (slot, head)
    int s = 0;
    uint32_t parity = 0;
    bool timed_out = false, bad_slot = false, bad_head = false;
    int64_t t_fail = t1;

    for (int64_t t = t0; t < t1; ++t, advance(cur, H, V)) {
        const uint32_t st = stage0 + (uint32_t)(s * stage_bytes);
        if (!__all_sync(kFull, WAITTEST ? mbar_wait_bounded(bar0 + 8 * s, parity, kWaitTestNs)
                                        : mbar_wait_bounded(bar0 + 8 * s, parity))) {
            timed_out = true;
            t_fail = t;
            break;
        }
        const int b = cur.b, h = cur.h, c = cur.c;
        const int64_t slot = slot_of(b);
        if (UMH && (t == t0 || c == 0)) unit_mh = model_head(h);
        const int mh = UMH ? unit_mh : model_head(h);
        const bool slot_ok = slot >= 0 && slot < p.num_slots, ok = slot_ok && (!HMAP || mh >= 0);
        bad_slot |= !slot_ok;
        if (HMAP) bad_head |= mh < 0;
        uint8_t *const grec = p.state + slot * p.slot_bytes + (int64_t)(h * V + c) * rec_bytes;  // written in place

        // ---- per-(slot, head) operands, gathered into calibrated key order ----
        if (t == t0 || c == 0) {
            ob = ops0 + (uint32_t)((unit & 1) * ops_bytes);
            cp_async_wait_all();
            __syncwarp();
            // beta (and the GDN log-decay) of the next 32 (slot, head) units are
            // loaded one per lane, long before they are needed
            if ((unit & 31) == 0) {
                const int64_t ul = (int64_t)b * H + h + lane;  // unit (batch row, held head)
                const bool in = ul < (int64_t)p.batch * H;
                int64_t um = ul;                                // its (batch row, model head)
                if (HMAP && in) {
                    const int64_t ub = ul / H;
                    um = ub * Hm + max(model_head((int)(ul - ub * H)), 0);
                }
                unit_beta = in ? p.beta[um] : 0.f;
                if (!KDA) unit_g = in ? p.g[um] : 0.f;
            }
            const float beta = __shfl_sync(kFull, unit_beta, unit & 31);
            const float alpha = KDA ? 0.f : expf(__shfl_sync(kFull, unit_g, unit & 31));
            ++unit;
            // d_k is a power of two: masking keeps a malformed permutation in bounds
            auto chan = [&](int u) { return (int)(lds32(ob + off_perm + (u & ~3)) >> (8 * (u & 3))) & (dk - 1); };
            auto kv_at = [&](int ch) { return BF16 ? bf16_at(ob + off_k, ch) : ldsf(ob + off_k + 4 * ch); };
            auto qv_at = [&](int ch) { return BF16 ? bf16_at(ob + off_q, ch) : ldsf(ob + off_q + 4 * ch); };
            auto av_at = [&](int ch) { return KDA ? expf(ldsf(ob + off_g + 4 * ch)) : alpha; };
            float kq = 0.f;  // this lane's share of k^T q (all d_k channels)
#pragma unroll
            for (int i = 0; i < R; ++i) {
                const int r = lane + 32 * i;
                const bool live = r < lo;
                const int ch = chan(live ? K + r : (lo > 0 ? K + lo - 1 : 0));  // stays inside perm
                const float kv = live ? kv_at(ch) : 0.f;
                const float qv = live ? qv_at(ch) : 0.f;
                kk[i] = splat2(kv);
                qq[i] = splat2(qv);
                bk[i] = splat2(beta * kv * kDown);  // working scale of the low tier
                // the decay times the working scale 2^-39; UINT8 rows keep it times 2^133
                // for dequantize_group_fma
                aa[i] = av_at(ch) * (LT == kLtU8 ? 0x1p94f : kDown);
                kq = fmaf(kv, qv, kq);
            }
            // FP16 rows in pairs: {a_u, a_u+1, bk_u, bk_u+1} {k_u, k_u+1, q_u, q_u+1};
            // rows K .. K8-1 (padding to whole chunks of 4 pairs) carry zero weights.
            // Lane l writes pair l (and pair l + 32 when K_hi > 64), straight-line.
            const int K8 = (K + 7) & ~7;
            auto hop_pair = [&](int u) {
                const bool one = u < K, two = u + 1 < K;
                const int c0 = chan(one ? u : 0);
                const int c1 = chan(two ? u + 1 : 0);
                const float k0 = one ? kv_at(c0) : 0.f, k1 = two ? kv_at(c1) : 0.f;
                const float q0 = one ? qv_at(c0) : 0.f, q1 = two ? qv_at(c1) : 0.f;
                const float a0 = av_at(c0), a1 = av_at(c1);
                sts128(hops + 16 * u, make_uint4(__float_as_uint(one ? a0 : 0.f), __float_as_uint(two ? a1 : 0.f),
                                                 __float_as_uint(beta * k0), __float_as_uint(beta * k1)));
                sts128(hops + 16 * u + 16, make_uint4(__float_as_uint(k0), __float_as_uint(k1), __float_as_uint(q0),
                                                      __float_as_uint(q1)));
                kq = fmaf(k0, q0, fmaf(k1, q1, kq));
            };
            if (2 * lane < K8) hop_pair(2 * lane);
            if (K8 > 64 && 2 * lane + 64 < K8) hop_pair(2 * lane + 64);
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) kq += __shfl_xor_sync(kFull, kq, m);
            bkq = beta * kq;  // beta k^T q: o = S_bar^T q + beta (k^T q) d
            __syncwarp();
            // operands of the next (slot, head) go into the other buffer
            if (t + (V - c) < t1) {
                const int nb = h + 1 == H ? b + 1 : b, nh = h + 1 == H ? 0 : h + 1;
                load_ops(nb, nh, ops0 + (uint32_t)((unit & 1) * ops_bytes));  // unit was incremented above
            }
        }

        const float vj = BF16 ? bf16_at(ob + off_v + c * kG * 2, lane) : ldsf(ob + off_v + c * kG * 4 + 4 * lane);

        if (ok) {
            const float vt = HAD ? hadamard_lanes(vj, sg) : vj;  // H v
            // ---- phase 1, FP16 tier (lane = column): one 32-bit load per row pair ----
            const uint32_t col = st + 4 * lane;  // this lane's word in FP16 row pair 0
            const int KP = (K + 1) >> 1;         // row pairs in the record
            // pair pi accumulates into rh[pi & 3], ph[pi & 3] (four independent chains)
            float2 rh[4], ph[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) rh[q] = ph[q] = make_float2(0.f, 0.f);
            auto hi_pair1 = [&](int pi, uint32_t wv, const uint4 &oa, const uint4 &ok) {
                const float2 xa = mul2(h2_to_f2(wv), make_float2(__uint_as_float(oa.x), __uint_as_float(oa.y)));
                rh[pi & 3] = fma2(xa, make_float2(__uint_as_float(ok.x), __uint_as_float(ok.y)), rh[pi & 3]);
                ph[pi & 3] = fma2(xa, make_float2(__uint_as_float(ok.z), __uint_as_float(ok.w)), ph[pi & 3]);
            };
            // K_hi above kHiUnroll: the FP16 rows' sums run before the low tier's rows are
            // reconstructed, so their loads do not compete with x for registers
            auto hi_phase1 = [&]() {
                if constexpr (KFIX) {
#pragma unroll
                    for (int pi = 0; pi < (KC + 1) / 2; ++pi)
                        hi_pair1(pi, lds32(col + 128 * pi), lds128(hops + 32 * pi), lds128(hops + 32 * pi + 16));
                } else {
                    // chunks of 4 pairs, loads first; pairs past the last carry zero
                    // weights and read a zero word
                    for (int p0 = 0; p0 < KP; p0 += 4) {
                        uint32_t wv[4];
                        uint4 oa[4], ok[4];
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            wv[q] = p0 + q < KP ? lds32(col + 128 * (p0 + q)) : 0u;
                            oa[q] = lds128(hops + 32 * (p0 + q));
                            ok[q] = lds128(hops + 32 * (p0 + q) + 16);
                        }
#pragma unroll
                        for (int q = 0; q < 4; ++q) hi_pair1(q, wv[q], oa[q], ok[q]);
                    }
                }
            };
            if constexpr (kHiFirst) {
                hi_phase1();
                // K_hi >= 24: a warp barrier keeps the low tier's loads from being scheduled
                // into the FP16 rows' sums (fewer spilled registers)
                if constexpr (KC >= 24) __syncwarp();
            }
            float2 x[R][16];
            float2 acc[16], accp[16];
            // ---- phase 1, low tier: reconstruct and decay (scaled by 2^-39), partial
            //      r~ = S~_bar^T k and p~ = S~_bar^T q ----
#pragma unroll
            for (int i = 0; i < RL; ++i) {
                const int r = min(lane + 32 * i, lo - 1);
                const uint4 c0 = lds128(st + codes_off + lo_chunk_off(r, 0, lo));
                const uint32_t sz = lds32(st + meta_off + 4 * r);
                if constexpr (U4) {
                    const uint32_t w[4] = {c0.x, c0.y, c0.z, c0.w};
                    dequantize_group_u4(w, sz, aa[i], x[i]);
                } else {
                    const uint4 c1 = lds128(st + codes_off + lo_chunk_off(r, 1, lo));
                    const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                    if constexpr (F8) dequantize_group_e4m3(w, __uint_as_float(sz), aa[i], x[i]);
                    else dequantize_group_fma(w, sz, aa[i], x[i]);
                }
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    acc[j] = (i == 0) ? mul2(x[i][j], kk[i]) : fma2(x[i][j], kk[i], acc[j]);
                    accp[j] = (i == 0) ? mul2(x[i][j], qq[i]) : fma2(x[i][j], qq[i], accp[j]);
                }
            }
            if (RL == 0) {
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[j] = accp[j] = make_float2(0.f, 0.f);
            }

            if constexpr (!kHiFirst) hi_phase1();
            rh[0] = add2(add2(rh[0], rh[1]), add2(rh[2], rh[3]));
            ph[0] = add2(add2(ph[0], ph[1]), add2(ph[2], ph[3]));
            const float rhi = rh[0].x + rh[0].y, phi = ph[0].x + ph[0].y;
            // fixed layouts: H r_hi overlaps the column sums, and the butterflies for d and o
            // run during the requantization (the general kernel keeps the plain order:
            // deferring them costs it registers)
            constexpr bool kLateD = KFIX && DFIX;
            const float hr_hi_early = (kLateD && HAD && K > 0) ? hadamard_lanes(rhi, sg) : 0.f;
            const float2 lo_sums = column_sum2(acc, accp, part, lane);
            const float rlo = lo_sums.x * kUp, plo = lo_sums.y * kUp;  // back from the working scale

            // r = H r~_lo + r_hi;  d = v - r (natural, FP16 rows);  H d = H v - r~_lo - H r_hi (low tier);
            // o = S_t^T q = S_bar^T q + beta (k^T q) d, with S_bar^T q = H p~_lo + p_hi.
            // H d goes out first: the low tier's requantization waits on it; the butterflies
            // for d and o run while it proceeds.
            float dj = 0.f, pj = 0.f, dt;
            auto natural_d_and_o = [&]() {
                if (HAD) {
                    dj = vj - (hadamard_lanes(rlo, sg) + rhi);
                    pj = hadamard_lanes(plo, sg) + phi;
                } else {
                    dj = vj - (rlo + rhi);
                    pj = plo + phi;
                }
                p.o[((int64_t)b * Hm + mh) * dvv + c * kG + lane] = fmaf(bkq, dj, pj);
            };
            if constexpr (kLateD) {
                dt = HAD ? vt - (rlo + hr_hi_early) : vj - (rlo + rhi);
            } else {
                const float hr_hi = (HAD && K > 0) ? hadamard_lanes(rhi, sg) : 0.f;
                natural_d_and_o();
                dt = HAD ? vt - (rlo + hr_hi) : dj;
            }
            sts32(dvec + 4 * lane, __float_as_uint(dt));
            __syncwarp();

            // ---- phase 2, low tier: rank-1 correction, requantize in place ----
            float2 d[16];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
                const uint4 w = lds128(dvec + 16 * jj);
                d[2 * jj] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
                d[2 * jj + 1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
            }
            // each stage runs over all row slots before the next starts, so the short
            // dependent chains of the rows (extrema -> scale -> codes) overlap
#pragma unroll
            for (int i = 0; i < RL; ++i) {
#pragma unroll
                for (int j = 0; j < 16; ++j) x[i][j] = fma2(bk[i], d[j], x[i][j]);
            }
            if constexpr (kLateD) natural_d_and_o();
            float mn[R], mx[R], inv[R], zq[R];
            uint32_t szw[R];
#pragma unroll
            for (int i = 0; i < RL; ++i) minmax32(x[i], mn[i], mx[i]);
            // scales: the common path assumes s != 0; a block whose scale rounds to 0
            // (rare) is encoded again below with the general path, over its first stores
            float sc[R];
            bool any_zero = false;
#pragma unroll
            for (int i = 0; i < RL; ++i) {
                if constexpr (U4) {  // levels 15; the widened rule of a degenerate block is built in
                    szw[i] = affine_params_u4(mn[i], mx[i], inv[i], zq[i]);
                } else if constexpr (F8) {
                    // s = max(max|x|, 1e-10) / 448 (IEEE division, natural domain); codes take
                    // x * (1/s), within an ulp of x / s: a code moves only where x / s sits at
                    // a rounding midpoint of E4M3
                    const float s8 = __fdiv_rn(fmaxf(fmaxf(-mn[i], mx[i]) * kUp, 1e-10f), 448.0f);
                    szw[i] = __float_as_uint(s8);
                    inv[i] = __frcp_rn(s8) * kUp;  // exact power-of-two scaling of 1/s
                } else {
                    sc[i] = scale_of(mn[i], mx[i]);
                    any_zero |= sc[i] == 0.0f;
                    szw[i] = affine_finish(sc[i], mn[i], inv[i], zq[i]);
                }
            }
            auto encode_store = [&](int i) {
                const int r = lane + 32 * i;
                const float2 inv2 = splat2(inv[i] * 0x1p-110f), zc2 = splat2(zq[i] * 0x1p-149f);
                if constexpr (F8) {
                    const float2 i2 = splat2(inv[i]);
                    uint32_t w[8];
#pragma unroll
                    for (int m = 0; m < 8; ++m) {  // values 4m .. 4m+3, value 4m in byte 0
                        const float2 a = mul2(x[i][2 * m], i2), b2 = mul2(x[i][2 * m + 1], i2);
                        w[m] = e4m3x2_of(a.y, a.x) | (e4m3x2_of(b2.y, b2.x) << 16);
                    }
                    if (r < lo) {
                        stg128(grec + codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                        stg128(grec + codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                        stg32(grec + meta_off + 4 * r, szw[i]);
                    }
                } else if constexpr (U4) {
                    // values 8m .. 8m+7 = pairs 4m .. 4m+3; value 8m ends in the low nibble
                    uint32_t w[4];
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        uint32_t a = 0u;
#pragma unroll
                        for (int k = 3; k >= 0; --k) {
                            const float2 e = fma2(x[i][4 * m + k], inv2, zc2);
                            a = pack_sat_u4(__float_as_uint(e.y), __float_as_uint(e.x), a);
                        }
                        w[m] = a;
                    }
                    if (r < lo) {
                        stg128(grec + codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                        stg32(grec + meta_off + 4 * r, szw[i]);
                    }
                } else {
                    uint32_t w[8];
#pragma unroll
                    for (int m = 0; m < 8; ++m) w[m] = encode4(x[i][2 * m], x[i][2 * m + 1], inv2, zc2);
                    if (r < lo) {
                        stg128(grec + codes_off + lo_chunk_off(r, 0, lo), make_uint4(w[0], w[1], w[2], w[3]));
                        stg128(grec + codes_off + lo_chunk_off(r, 1, lo), make_uint4(w[4], w[5], w[6], w[7]));
                        stg32(grec + meta_off + 4 * r, szw[i]);
                    }
                }
            };
#pragma unroll
            for (int i = 0; i < RL; ++i) encode_store(i);
            if constexpr (LT == kLtU8) {
                if (__any_sync(kFull, any_zero)) {
#pragma unroll
                    for (int i = 0; i < RL; ++i) {
                        if (sc[i] == 0.0f) {
                            szw[i] = affine_params_scaled(mn[i], mx[i], inv[i], zq[i]);
                            encode_store(i);
                        }
                    }
                }
            }

            // ---- phase 2, FP16 tier: S = S_bar + beta k d, FP16 store (two rows per word) ----
            const float2 dj2 = splat2(dj);
            auto hi_pair2 = [&](int pi, uint32_t wv, const uint4 &oa) {
                const float2 xa = mul2(h2_to_f2(wv), make_float2(__uint_as_float(oa.x), __uint_as_float(oa.y)));
                const float2 y = fma2(make_float2(__uint_as_float(oa.z), __uint_as_float(oa.w)), dj2, xa);
                stg32(grec + 128 * pi + 4 * lane, f2_to_h2(y.x, y.y));  // an odd K's padding half stays 0
            };
            if constexpr (KFIX) {
#pragma unroll
                for (int pi = 0; pi < (KC + 1) / 2; ++pi) hi_pair2(pi, lds32(col + 128 * pi), lds128(hops + 32 * pi));
            } else {
                for (int p0 = 0; p0 < KP; p0 += 4) {
                    uint32_t wv[4];
                    uint4 oa[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        wv[q] = p0 + q < KP ? lds32(col + 128 * (p0 + q)) : 0u;
                        oa[q] = lds128(hops + 32 * (p0 + q));
                    }
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        if (p0 + q < KP) hi_pair2(p0 + q, wv[q], oa[q]);
                }
            }
        }
        // ---- the stage has been read: refill it with tile t + nstage ----
        __syncwarp();
        if (lane == 0 && t_pre < t1) {
            fence_proxy_async_smem();  // the warp's reads of the stage before the bulk copy's writes
            issue(t_pre, pre, s);
            ++t_pre;
            advance(pre, H, V);
        }
        if (++s == nstage) {
            s = 0;
            parity ^= 1u;
        }
    }
    if (timed_out) {
        // let the loads already in flight land (each wait bounded) before the CTA's
        // shared memory goes away
        const int64_t last = min(t1 - 1, t_fail + nstage - 1);
        if constexpr (WAITTEST) {
            // settle the extra bytes of every armed stage, so its phase completes
            // exactly when its copy has landed
            if (lane == 0) {
                for (int64_t tt = t_fail; tt <= last; ++tt) {
                    const Cursor k = cursor_at(tt, H, V);
                    const int64_t slot = slot_of(k.b);
                    if (slot >= 0 && slot < p.num_slots)
                        mbar_complete_tx(bar0 + 8 * (int)((tt - t0) % nstage), kWaitTestExtra);
                }
            }
            __syncwarp();
        }
        for (int64_t tt = t_fail; tt <= last; ++tt) {
            const int64_t idx = tt - t0;
            mbar_wait_bounded(bar0 + 8 * (int)(idx % nstage), (uint32_t)((idx / nstage) & 1));
        }
    }
    cp_async_wait_all();  // operand copies of a (slot, head) that will not run
    if (lane == 0) {
        const uint32_t bits =
            (timed_out ? kDevWaitTimeout : 0u) | (bad_slot ? kDevBadSlot : 0u) | (bad_head ? kDevBadHead : 0u);
        if (bits) atomicOr(p.status, bits);
        // every phase has completed: the barriers' memory may be reused by a following body
        if (!timed_out)
            for (int s2 = 0; s2 < nstage; ++s2) mbar_inval(bar0 + 8 * s2);
    }
    __syncwarp();
    return timed_out;
}

template <int RL, int DKC, int KC, bool KDA, bool HAD, bool BF16, bool HMAP, int LT = kLtU8, bool WAITTEST = false>
__global__ void __launch_bounds__(256, 1) packed_step_kernel(const PackedParams p) {
    packed_step_body<RL, DKC, KC, KDA, HAD, BF16, HMAP, LT, WAITTEST>(p, blockIdx.x, gridDim.x);
}

// Two head groups of one layer in one launch (App. E: per-head budgets as budget-specific
// kernel groups).  Every warp first takes its share of group 1's tiles (K_hi = KC1), then
// its share of group 2's (K_hi = KC2), so each SM carries the same mix of both and no
// split of the grid needs tuning; each group keeps its compile-time record layout, pool,
// permutation table and head map.  Both parameter blocks give the warps the same
// shared-memory stride, so a warp's region is the same in both bodies.  d_k = 128.
template <int KC1, int KC2, bool KDA, bool HAD, bool BF16>
__global__ void __launch_bounds__(256, 1) packed_step2_kernel(const PackedParams p1, const PackedParams p2) {
    // the per-unit model head where both groups keep at most 20 FP16 rows (measured: with a
    // group of 24 or 28 rows the register goes to spills)
    constexpr bool UMH = (KC1 > KC2 ? KC1 : KC2) <= 20;
    if (packed_step_body<(128 - KC1 + 31) / 32, 128, KC1, KDA, HAD, BF16, true, kLtU8, false, UMH>(p1, blockIdx.x,
                                                                                                  gridDim.x))
        return;  // a copy of group 1 was lost (status set): its barriers cannot be reused
    packed_step_body<(128 - KC2 + 31) / 32, 128, KC2, KDA, HAD, BF16, true, kLtU8, false, UMH>(p2, blockIdx.x,
                                                                                              gridDim.x);
}

}  // namespace damp
