// prefill_tc_kda.cuh -- the KDA prefill chunk on the tensor cores: the chunkwise closed form
// of prefill_tc.cuh (App. A.5 prefill path; Sec. 3.1 Eq. delta_update) with a decay per key
// channel.
//
// With a_{t,c} = exp(g_{t,c}) and gamma_t = a_0 (.) ... (.) a_t (a vector over the channels;
// (.) the elementwise product), the per-token recurrence of a piece unrolls to
//     u_t + beta_t sum_{s<t} (k_t (.) gamma_t / gamma_s) . k_s u_s = beta_t (v_t - S_0^T (gamma_t (.) k_t))
//     o_t = S_0^T (gamma_t (.) q_t) + sum_{s<=t} (q_t (.) gamma_t / gamma_s) . k_s u_s
//     S_C = diag(gamma_C) S_0 + sum_s (k_s (.) gamma_C / gamma_s) u_s^T .
// The ratios are taken about a reference token m of the piece: xi_t = gamma_t / gamma_m, as
// running products outward from m (never differences of cumulative log sums), so that
//     gamma_t (.) k_t = gamma_m (.) (xi_t (.) k_t),  gamma_t / gamma_s = xi_t / xi_s,
//     gamma_C / gamma_s = xi_C / xi_s.
// With X = [K (.) Xi; Q (.) Xi], Z = K / Xi and B1 = diag(gamma_m) S_0, one product gives
// W = K~ S_0 and P = Q~ S_0 (X B1) and one the Gram rows X Z^T (the L and M of
// prefill_tc.cuh, decay included); both contract over the channels in two halves of 64
// (the split operands of one half fill the shared memory).  The state's update is
// (K (.) Xi_C / Xi)^T U.  A piece is cut short (64, 32, ..., 1 tokens) where xi or 1 / xi
// would leave FP32 (a channel decaying by more than e^85 on either side of m); tokens
// past a piece or a row's length are masked (xi = 0, beta = 0).  Everything else -- the
// state in tensor memory, split bf16 operands, the solve, the output product, the
// requantization -- is prefill_tc.cuh's.
#pragma once

#include "prefill_tc.cuh"

namespace damp {

// Shared memory (bytes).  Areas that share bytes are never live together:
//   piece inputs:   KQ [0, 34K)  XI [34K, 67K)  V [67K, 84K)   (records at unit start: [84K, 116K))
//   per channel half: X [84K, 132K)  Z [132K, 156K)  B1 [156K, 204K)
//   after the first products: A3 [84K, 132K)  LP [132K, 149K)  AO [149K, 197K)  YU [0, 33K)
//   after the solve: BU [0, 48K)
constexpr int kKdKQ = 0;            // k rows 0..63 then q rows 0..63, bf16, 272 bytes per row
constexpr int kKdRowKQ = 272;
constexpr int kKdXI = 34816;        // g, then xi: 64 rows of 132 FP32 (token t, channel c)
constexpr int kKdRowXI = 132;
constexpr int kKdV = 68608;         // v, bf16, 64 rows of 272 bytes
constexpr int kKdRec = 86016;       // the four value-block records (unit start)
constexpr int kKdX = 86016;         // X half: three bf16 parts, K-major (128 rows x 64 channels)
constexpr int kKdZ = 135168;        // Z half: three bf16 parts, K-major (64 tokens x 64 channels)
constexpr int kKdB1 = 159744;       // B1 half: three bf16 parts, MN-major (128 value columns x 64 channels)
constexpr int kKdA3 = 86016;        // (K (.) Xi_C / Xi)^T: three bf16 parts, K-major (128 record rows x 64 tokens)
constexpr int kKdLP = 135168;       // L'^T, 64 rows of kTcRowL FP32
constexpr int kKdAO = 152576;       // [0; M]: three bf16 parts, K-major (128 rows x 64 tokens)
constexpr int kKdYU = 0;            // Y, then U: 64 rows of kTcRowY FP32
constexpr int kKdBU = 0;            // U: three bf16 parts, K-major (value columns x tokens)
constexpr int kKdScal = 208896;     // beta, pi, gamma_m, xi_C, mbarriers, TMEM address
constexpr int kKdSmem = kKdScal + 2048;
constexpr int kKdMaxRec = 8192;     // four records fit in [kKdRec, kKdZ)
constexpr float kKdMaxLog = 85.0f;  // largest log-range of xi on either side of the reference token
constexpr int kKdThreads = 512;     // four threads per tensor-memory lane (warps w, w + 4, w + 8, w + 12)

// One CTA of kKdThreads threads per (slot, head) unit at a time (persistent over units);
// d_k = d_v = 128, bf16 q/k/v, low tier FMT (UINT8 or UINT4 affine, with or without H_32).
// Thread (row, quarter qq): row = tensor-memory lane (warps w, w + 4, w + 8 and w + 12
// reach the same lanes); the quarters split a row's value blocks (one each) or a phase's tasks.
template <int FMT>
__global__ void __launch_bounds__(kKdThreads, 1) prefill_tc_kda_kernel(const PrefillParams p) {
    static_assert(FMT != kFmtS8Row, "the row-absmax format shares a row scale over the value blocks");
    constexpr bool HAD = fmt_had(FMT);
    extern __shared__ __align__(128) uint8_t smem[];  // descriptors need 16-byte alignment (no swizzle)
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int row = tid & 127, qq = tid >> 7;
    const uint32_t sb = smem_u32(smem);
    const int H = p.H, T = p.T, Hm = p.Hm;
    const int rec_bytes = p.rec_bytes, rstride = tc_rec_stride(rec_bytes);
    const uint32_t scal = sb + (uint32_t)kKdScal;
    const uint32_t s_beta = scal, s_perm = scal + 256, s_gm = scal + 384, s_xiC = scal + 1408;
    const uint32_t bar_rec = scal + 1936, bar_mma = scal + 1944, s_taddr = scal + 1952;
    const uint32_t kq = sb + (uint32_t)kKdKQ, xi = sb + (uint32_t)kKdXI;

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
    struct Unit {
        int64_t unit, slot;
        int b, h, mh, hq, Tb;
    };
    // the first unit at or after u (stepping by the grid) with work; unit == units if none
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
    // k, q, g, v and beta of unit n's tokens p0 .. p0 + 63 (cp.async; rows past the row's
    // length are zero)
    auto load_piece = [&](const Unit &n, int p0) {
        const int nl = min(kTcC, n.Tb - p0);
#pragma unroll 1
        for (int i = tid; i < 2048; i += kKdThreads) {  // k rows 0..63, q rows 64..127: 16 chunks each
            const int m = i >> 4, j = i & 15, t = m & 63;
            const uint32_t dst = kq + (uint32_t)(m * kKdRowKQ + 16 * j);
            if (t < nl)
                cp_async16(dst, static_cast<const uint8_t *>(m < 64 ? p.k : p.q) +
                                    (((int64_t)n.b * T + p0 + t) * p.Hqk + n.hq) * 256 + 16 * j);
            else
                sts128(dst, make_uint4(0u, 0u, 0u, 0u));
        }
#pragma unroll 1
        for (int i = tid; i < 2048; i += kKdThreads) {  // g: 64 rows of 32 chunks
            const int t = i >> 5, j = i & 31;
            const uint32_t dst = xi + (uint32_t)(t * kKdRowXI * 4 + 16 * j);
            if (t < nl)
                cp_async16(dst, reinterpret_cast<const uint8_t *>(p.g + (((int64_t)n.b * T + p0 + t) * Hm + n.mh) * 128) +
                                    16 * j);
            else
                sts128(dst, make_uint4(0u, 0u, 0u, 0u));
        }
#pragma unroll 1
        for (int i = tid; i < 1024; i += kKdThreads) {
            const int t = i >> 4, j = i & 15;
            const uint32_t dst = sb + (uint32_t)(kKdV + t * kTcRowV + 16 * j);
            if (t < nl)
                cp_async16(dst, static_cast<const uint8_t *>(p.v) + (((int64_t)n.b * T + p0 + t) * Hm + n.mh) * 256 + 16 * j);
            else
                sts128(dst, make_uint4(0u, 0u, 0u, 0u));
        }
        if (tid < kTcC) {
            if (tid < nl) cp_async4(s_beta + 4 * tid, p.beta + ((int64_t)n.b * T + p0 + tid) * Hm + n.mh);
            else sts32(s_beta + 4 * tid, 0u);
        }
        cp_async_commit();
    };
    // unit n's records, pi and first piece, one unit ahead
    auto prefetch = [&](const Unit &n) {
        if (tid == 0) {
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(bar_rec, (uint32_t)(4 * rec_bytes));
            uint8_t *const g0 = rec_of(n);
#pragma unroll
            for (int c = 0; c < 4; ++c)
                bulk_g2s(sb + (uint32_t)(kKdRec + c * rstride), g0 + (int64_t)c * rec_bytes, (uint32_t)rec_bytes, bar_rec);
        }
        if (tid < 8) cp_async16(s_perm + 16 * tid, p.perm + (int64_t)n.h * 128 + 16 * tid);
        load_piece(n, 0);
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
        // ---- S_0: record row u = row into tensor-memory lane u (this quarter's value block) ----
        tc_reconstruct<FMT, 4>(p, sb + (uint32_t)kKdRec, rstride, row, qq, tS);
        __syncthreads();  // the records are read: the first piece's operands go over them

        int p0 = 0;
        bool first = true;
#pragma unroll 1
        while (p0 < Tb) {
            if (!first) load_piece(cur, p0);
            first = false;
            cp_async_wait_all();
            __syncthreads();
            // ---- the piece's length: the largest of 64, 32, ..., 1 tokens over which every
            //      channel decays by at most e^kKdMaxLog on either side of the reference
            //      token m = L / 2 - 1 (thread c = row of quarter 0 owns channel c) ----
            float lam[7] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};  // Lambda_t = sum_{i<=t} g_i at t = 0, 1, 3, ..., 63
            if (qq == 0) {
                float acc = 0.f;
#pragma unroll
                for (int t = 0; t < kTcC; ++t) {  // unrolled: the indices of lam are constants
                    acc += ldsf(xi + (uint32_t)(t * kKdRowXI * 4 + 4 * row));
                    if (t == 0) lam[0] = acc;
                    if (t == 1) lam[1] = acc;
                    if (t == 3) lam[2] = acc;
                    if (t == 7) lam[3] = acc;
                    if (t == 15) lam[4] = acc;
                    if (t == 31) lam[5] = acc;
                    if (t == 63) lam[6] = acc;
                }
            }
            int L = 1;
#pragma unroll
            for (int j = 6; j >= 1; --j) {  // L = 2^j, m = 2^(j-1) - 1
                const bool ok_c = qq != 0 || ((lam[0] - lam[j - 1] <= kKdMaxLog) && (lam[j - 1] - lam[j] <= kKdMaxLog));
                if (L == 1 && __syncthreads_and(ok_c)) L = 1 << j;
            }
            const int nt = min(L, Tb - p0);   // tokens of this piece; the rest are masked
            const int m = L > 1 ? L / 2 - 1 : 0;
            // ---- xi_t = gamma_t / gamma_m in place of g (0 for masked tokens), as running
            //      products from m (quarter 0: downward, xi_{t-1} = xi_t e^{-g_t}, and gamma_m;
            //      quarter 1: upward, xi_t = xi_{t-1} e^{g_t}); xi_C at C = nt - 1 ----
            {
                const uint32_t colc = xi + (uint32_t)(4 * row);
                float x = 1.f;
                if (qq == 0) {
                    float gm = 1.f;
#pragma unroll 1
                    for (int t = m; t >= 0; --t) {
                        const uint32_t a = colc + (uint32_t)(t * kKdRowXI * 4);
                        const float g = ldsf(a);
                        sts32(a, __float_as_uint(t < nt ? x : 0.f));
                        if (t == nt - 1) sts32(s_xiC + 4 * row, __float_as_uint(x));
                        gm *= expf(g);
                        x *= expf(-g);
                    }
                    sts32(s_gm + 4 * row, __float_as_uint(gm));
                } else if (qq == 1) {
#pragma unroll 1
                    for (int t = m + 1; t < kTcC; ++t) {
                        const uint32_t a = colc + (uint32_t)(t * kKdRowXI * 4);
                        x *= expf(ldsf(a));
                        sts32(a, __float_as_uint(t < nt ? x : 0.f));
                        if (t == nt - 1) sts32(s_xiC + 4 * row, __float_as_uint(x));
                    }
                }
            }
            if (tid < kTcC && tid >= nt) sts32(s_beta + 4 * tid, 0u);  // tokens past the piece
            __syncthreads();
            // ---- per channel half (64 channels): X = [K (.) Xi; Q (.) Xi], Z = K / Xi and
            //      B1 = diag(gamma_m) S_0 as three bf16 parts; W | P += X B1 and the Gram rows
            //      += X Z^T ----
#pragma unroll 1
            for (int hh = 0; hh < 2; ++hh) {
                const int c0 = 64 * hh;
                {  // X: row m = row, channels c0 + 16 qq .. + 15
                    const uint32_t kqrow = kq + (uint32_t)(row * kKdRowKQ), xrow = xi + (uint32_t)((row & 63) * kKdRowXI * 4);
#pragma unroll
                    for (int jj = 0; jj < 2; ++jj) {
                        const int cl = 16 * qq + 8 * jj;
                        const uint4 kw = lds128(kqrow + (uint32_t)(2 * (c0 + cl)));
                        const uint4 xa = lds128(xrow + (uint32_t)(4 * (c0 + cl))), xb = lds128(xrow + (uint32_t)(4 * (c0 + cl) + 16));
                        const uint32_t kk[4] = {kw.x, kw.y, kw.z, kw.w};
                        const float xv[8] = {__uint_as_float(xa.x), __uint_as_float(xa.y), __uint_as_float(xa.z), __uint_as_float(xa.w),
                                             __uint_as_float(xb.x), __uint_as_float(xb.y), __uint_as_float(xb.z), __uint_as_float(xb.w)};
                        float v[8];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            v[2 * e] = __uint_as_float(kk[e] << 16) * xv[2 * e];
                            v[2 * e + 1] = __uint_as_float(kk[e] & 0xffff0000u) * xv[2 * e + 1];
                        }
                        split3_store8(sb + kKdX + tc_k64_off(row, cl), 16384, v);
                    }
                }
#pragma unroll 1
                for (int i = tid; i < 512; i += kKdThreads) {  // Z: token s, 8 channels per task
                    const int s2 = i >> 3, cl = 8 * (i & 7);
                    const uint4 kw = lds128(kq + (uint32_t)(s2 * kKdRowKQ + 2 * (c0 + cl)));
                    const uint32_t xrow = xi + (uint32_t)(s2 * kKdRowXI * 4 + 4 * (c0 + cl));
                    const uint4 xa = lds128(xrow), xb = lds128(xrow + 16);
                    const uint32_t kk[4] = {kw.x, kw.y, kw.z, kw.w};
                    const float xv[8] = {__uint_as_float(xa.x), __uint_as_float(xa.y), __uint_as_float(xa.z), __uint_as_float(xa.w),
                                         __uint_as_float(xb.x), __uint_as_float(xb.y), __uint_as_float(xb.z), __uint_as_float(xb.w)};
                    float z[8];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float k0 = __uint_as_float(kk[e] << 16), k1 = __uint_as_float(kk[e] & 0xffff0000u);
                        z[2 * e] = xv[2 * e] != 0.f ? __fdiv_rn(k0, xv[2 * e]) : 0.f;  // masked tokens: 0
                        z[2 * e + 1] = xv[2 * e + 1] != 0.f ? __fdiv_rn(k1, xv[2 * e + 1]) : 0.f;
                    }
                    split3_store8(sb + kKdZ + tc_k64_off(s2, cl), 8192, z);
                }
                {  // B1: record row u = row (channel pi(u)) when its channel is in this half
                    const int ch = (int)(lds_u8(s_perm + row) & 127u);
                    const bool mine = (ch >> 6) == hh;
                    const float gmc = ldsf(s_gm + 4 * ch);
                    {
                        const int c = qq;
                        float v[32];
                        tc_ld32(tS + 32 * c, v);  // every lane: warp-collective
                        if (mine) {
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] *= gmc;
#pragma unroll
                            for (int j8 = 0; j8 < 4; ++j8)
                                split3_store8(sb + kKdB1 + tc_mn_off(32 * c + 8 * j8, ch & 63, 2048), 16384, v + 8 * j8);
                        }
                    }
                }
                fence_proxy_async_smem();
                tc_fence_before();
                __syncthreads();
                tc_fence_after();
                if (tid == 0) {
                    constexpr int pa[6] = {0, 0, 1, 0, 2, 1}, pb[6] = {0, 1, 0, 2, 0, 1};
#pragma unroll
                    for (int q = 0; q < 6; ++q)
#pragma unroll
                        for (int ks = 0; ks < 4; ++ks)
                            tc_mma(tmem + kColWP, tc_desc(sb + kKdX + 16384 * pa[q] + 256 * ks, 128, 1024),
                                   tc_desc(sb + kKdB1 + 16384 * pb[q] + 4096 * ks, 2048, 128), kIdWP, (hh | q | ks) != 0);
#pragma unroll
                    for (int q = 0; q < 6; ++q)
#pragma unroll
                        for (int ks = 0; ks < 4; ++ks)
                            tc_mma(tmem + kColG, tc_desc(sb + kKdX + 16384 * pa[q] + 256 * ks, 128, 1024),
                                   tc_desc(sb + kKdZ + 8192 * pb[q] + 256 * ks, 128, 1024), kIdG, (hh | q | ks) != 0);
                    tc_commit(bar_mma);
                }
                if (!tc_wait_all(bar_mma, ph_mma)) {
                    timed_out = mma_pending = true;
                    break;
                }
                ph_mma ^= 1u;
                tc_fence_after();
            }
            if (timed_out) break;
            // ---- quarter 0: rows of L' = beta_t G_ts (s < t) and M = G_ts (s <= t) from the
            //      Gram rows (the decay is in G); quarter 1: the zero rows of [0; M]; all:
            //      (K (.) Xi_C / Xi)^T in record-row order and gamma_C S_0 in tensor memory ----
            if (qq == 0) {
                const int t = row & 63;
                const bool qside = row >= 64;
                const float bt = qside ? 1.f : ldsf(s_beta + 4 * t);
#pragma unroll 1
                for (int h2 = 0; h2 < 2; ++h2) {  // columns s of 32 h2 .. 32 h2 + 31
                    float gr[32];
                    tc_ld32(tG + 32 * h2, gr);
#pragma unroll
                    for (int s2 = 0; s2 < 32; ++s2) {
                        const int sc = 32 * h2 + s2;
                        gr[s2] = sc < t ? bt * gr[s2] : (sc == t && qside ? gr[s2] : 0.f);
                    }
                    if (!qside) {  // column t of L'^T
                        const uint32_t colt = sb + (uint32_t)(kKdLP + 4 * t + 32 * h2 * kTcRowL * 4);
#pragma unroll
                        for (int s2 = 0; s2 < 32; ++s2) sts32(colt + (uint32_t)(s2 * kTcRowL * 4), __float_as_uint(gr[s2]));
                    } else {
#pragma unroll
                        for (int g = 0; g < 4; ++g)
                            split3_store8(sb + kKdAO + tc_k64_off(64 + t, 32 * h2 + 8 * g), 16384, gr + 8 * g);
                    }
                }
            } else if (qq == 1) {
#pragma unroll 1
                for (int i = row; i < 1536; i += 128)
                    sts128(sb + (uint32_t)(kKdAO + (i >> 9) * 16384 + (i & 511) * 16), make_uint4(0u, 0u, 0u, 0u));
            }
            {  // (K (.) Xi_C / Xi)^T, K-major: record row u = row (channel pi(u)), tokens 16 qq .. + 15
                const uint32_t ch = lds_u8(s_perm + row) & 127u;
                const float xic = ldsf(s_xiC + 4u * ch);
#pragma unroll
                for (int g8 = 0; g8 < 2; ++g8) {
                    float v[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int t = 16 * qq + 8 * g8 + e;
                        const float kv = __uint_as_float(lds_u16(kq + (uint32_t)(t * kKdRowKQ) + 2u * ch) << 16);
                        const float xs = ldsf(xi + (uint32_t)(t * kKdRowXI * 4) + 4u * ch);
                        v[e] = xs != 0.f ? kv * (xic * __frcp_rn(xs)) : 0.f;  // masked tokens: 0
                    }
                    split3_store8(sb + kKdA3 + tc_k64_off(row, 16 * qq + 8 * g8), 16384, v);
                }
            }
            {  // gamma_C S_0 = gamma_m xi_C S_0 (per channel; the state product accumulates onto it)
                const uint32_t ch = lds_u8(s_perm + row) & 127u;
                const float gc = ldsf(s_gm + 4u * ch) * ldsf(s_xiC + 4u * ch);
                {
                    const int c = qq;
                    float v[32];
                    tc_ld32(tS + 32 * c, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] *= gc;
                    tc_st32(tS + 32 * c, v);
                }
            }
            __syncthreads();  // K and Xi are read: Y goes over them
            // ---- Y = diag(beta) (v~ - W), FP32 rows (this quarter's value block) ----
            if (row < 64) {
                const int t = row;
                const float bt = ldsf(s_beta + 4 * t);
                const uint32_t vrow = sb + (uint32_t)(kKdV + t * kTcRowV), yrow = sb + (uint32_t)(kKdYU + t * kTcRowY * 4);
                {
                    const int c = qq;
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
                               make_uint4(__float_as_uint(bt * (ya.x - w[4 * q])), __float_as_uint(bt * (ya.y - w[4 * q + 1])),
                                          __float_as_uint(bt * (yb.x - w[4 * q + 2])), __float_as_uint(bt * (yb.y - w[4 * q + 3]))));
                    }
                }
            }
            __syncthreads();
            // ---- U = L^-1 Y (value column n = row, in place) ----
            tc_solve<4>(sb + (uint32_t)(kKdYU + 4 * row), sb + (uint32_t)kKdLP, qq);
            // ---- U as three bf16 parts, K-major (value columns n x tokens s): tokens 16 qq .. + 15 ----
            {
                const uint32_t col = sb + (uint32_t)(kKdYU + 4 * row);
                float uc[16];
#pragma unroll
                for (int t = 0; t < 16; ++t) uc[t] = ldsf(col + (uint32_t)((16 * qq + t) * kTcRowY * 4));
                __syncthreads();  // every column is read: the parts go over Y / U
#pragma unroll
                for (int g = 0; g < 2; ++g) split3_store8(sb + kKdBU + tc_k64_off(row, 16 * qq + 8 * g), 16384, uc + 8 * g);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncthreads();
            tc_fence_after();
            if (tid == 0) {
                // O = P + [0; M] U and S += (K (.) Xi_C / Xi)^T U; six partial products each
                constexpr int pa[6] = {0, 0, 1, 0, 2, 1}, pb[6] = {0, 1, 0, 2, 0, 1};
#pragma unroll
                for (int q = 0; q < 6; ++q)
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        tc_mma(tmem + kColWP, tc_desc(sb + kKdAO + 16384 * pa[q] + 256 * ks, 128, 1024),
                               tc_desc(sb + kKdBU + 16384 * pb[q] + 256 * ks, 128, 1024), kIdO, 1u);
#pragma unroll
                for (int q = 0; q < 6; ++q)
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        tc_mma(tmem + kColS, tc_desc(sb + kKdA3 + 16384 * pa[q] + 256 * ks, 128, 1024),
                               tc_desc(sb + kKdBU + 16384 * pb[q] + 256 * ks, 128, 1024), kIdO, 1u);
                tc_commit(bar_mma);
            }
            if (!tc_wait_all(bar_mma, ph_mma)) {
                timed_out = mma_pending = true;
                break;
            }
            ph_mma ^= 1u;
            tc_fence_after();
            if (p0 + nt >= Tb && nxt.unit < units) prefetch(nxt);  // the next unit's loads overlap this one's tail
            // ---- o_t = H (P_t + (M U)_t) (lanes 64 + t, this quarter's value block) ----
            if (row >= 64) {
                const int t = row - 64;
                float *orow = p.o + (((int64_t)b * T + p0 + min(t, nt - 1)) * Hm + mh) * 128;
                {
                    const int c = qq;
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
            p0 += nt;
        }
        if (timed_out) break;
        // ---- the chunk-final state into the record in place ----
        tc_requantize<FMT, 4>(p, grec0, row, qq, lane, tS);
        cur = nxt;
    }
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
