// launch_packed.cuh -- host-side launcher of the fused packed decode step.
// Included once per decay kind (GDN / KDA) so the two sets of template
// instantiations compile in parallel translation units.
#pragma once

#include <algorithm>
#include <initializer_list>
#include <utility>

#include "damp_internal.h"
#include "decode_packed.cuh"
#include "formats.cuh"

namespace damp {

// Launch shape: one CTA per SM with kPackedWarps warps; every warp owns a
// contiguous range of tiles and keeps kPackedStages tile loads in flight.
constexpr int kPackedWarps = 8;
constexpr int kPackedStages = 3;

// Parameters and launch shape of one packed step (no launch).
struct PackedLaunch {
    PackedParams p;
    int warps, grid, smem;
};

template <bool KDA>
static cudaError_t packed_launch_shape(const StepArgs &a, uint32_t *status, PackedLaunch *out) {
    const int V = a.dv / kG;
    const RecGeom rg = rec_geom(a.dk, a.K, a.fmt);
    const int esz = a.in_bf16 ? 2 : 4;
    PackedParams p{};
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
    p.V = V;
    p.K = a.K;
    p.rec_bytes = rg.bytes;
    p.codes_off = rg.codes_off;
    p.meta_off = rg.meta_off;
    p.slot_bytes = (int64_t)a.H * V * rg.bytes;
    p.bytes_v = a.dv * esz;  // the whole v row of a (slot, head)
    p.bytes_qk = a.dk * esz;
    p.bytes_g = KDA ? a.dk * 4 : 0;
    p.bytes_perm = a.dk;
    // operand buffer: [v][q][k][g][perm], every part a multiple of 16 B
    int off = 0;
    p.off_v = off;
    off += p.bytes_v;
    p.off_q = off;
    off += p.bytes_qk;
    p.off_k = off;
    off += p.bytes_qk;
    p.off_g = off;
    off += p.bytes_g;
    p.off_perm = off;
    off += p.bytes_perm;
    p.ops_bytes = off;
    p.ops_off = (scratch_bytes(a.K) + 15) & ~15;
    p.stage_bytes = (rg.bytes + 127) & ~127;
    p.nstage = kPackedStages;
    p.stage0_off = (p.ops_off + 2 * p.ops_bytes + 127) & ~127;
    p.warp_smem = p.stage0_off + p.nstage * p.stage_bytes;
    p.total_tiles = (int64_t)a.batch * a.H * V;
    p.status = status;

    // shrink the warp count (then the ring) until the per-CTA shared memory fits
    const int smem_cap = max_smem_per_block();
    int warps = kPackedWarps;
    while (warps > 1 && warps * p.warp_smem > smem_cap) --warps;
    if (warps * p.warp_smem > smem_cap) {
        p.nstage = 2;
        p.warp_smem = p.stage0_off + p.nstage * p.stage_bytes;
    }
    if (warps * p.warp_smem > smem_cap) return cudaErrorInvalidConfiguration;
    const int64_t want = (p.total_tiles + warps - 1) / warps;
    out->p = p;
    out->warps = warps;
    out->grid = (int)std::min<int64_t>(std::max<int64_t>(want, 1), (int64_t)sm_count());
    out->smem = p.warp_smem * warps;
    return cudaSuccess;
}

// LT: the low tier's code type (kLtU8: formats 0, 1; kLtU4: formats 3, 4; kLtE4M3: format 5).
// WAITTEST launches the bounded-wait test instance instead of the decode step (layout
// d_k = d_v = 128, K_hi = 10, format 0, BF16 inputs, no head map only).
template <bool KDA, int LT, bool WAITTEST = false>
static cudaError_t launch_packed_impl(const StepArgs &a, cudaStream_t stream, uint32_t *status) {
    PackedLaunch sh;
    cudaError_t e0 = packed_launch_shape<KDA>(a, status, &sh);
    if (e0 != cudaSuccess) return e0;
    const PackedParams &p = sh.p;
    if (p.total_tiles == 0) return cudaSuccess;
    const int warps = sh.warps, grid = sh.grid, smem = sh.smem;

    void (*kern)(PackedParams) = nullptr;
    const bool had = fmt_had(a.fmt);
    // a head group (head map) runs the general instances with model-head indexing
    const bool hmap = a.head_map != nullptr;
    // (each pick is one compound statement; the FP8 tier has no H_32 variant)
#define DAMP_PICK4(RL_, DKC_, KC_)                                                                \
    {                                                                                             \
        if constexpr (LT != kLtE4M3) {                                                            \
            if (had) kern = a.in_bf16 ? packed_step_kernel<RL_, DKC_, KC_, KDA, true, true, false, LT>   \
                                      : packed_step_kernel<RL_, DKC_, KC_, KDA, true, false, false, LT>; \
        }                                                                                         \
        if (!had) kern = a.in_bf16 ? packed_step_kernel<RL_, DKC_, KC_, KDA, false, true, false, LT>     \
                                   : packed_step_kernel<RL_, DKC_, KC_, KDA, false, false, false, LT>;   \
    }
#define DAMP_PICK4_HMAP(RL_)                                                                      \
    {                                                                                             \
        if constexpr (LT != kLtE4M3) {                                                            \
            if (had) kern = a.in_bf16 ? packed_step_kernel<RL_, 0, -1, KDA, true, true, true, LT> \
                                      : packed_step_kernel<RL_, 0, -1, KDA, true, false, true, LT>; \
        }                                                                                         \
        if (!had) kern = a.in_bf16 ? packed_step_kernel<RL_, 0, -1, KDA, false, true, true, LT>   \
                                   : packed_step_kernel<RL_, 0, -1, KDA, false, false, true, LT>; \
    }
    const int rl = (a.dk - a.K + 31) / 32;
    if constexpr (WAITTEST) {
        if (a.dk != 128 || a.dv != 128 || p.nstage != 3 || a.K != 10 || a.fmt != 0 || !a.in_bf16 || hmap)
            return cudaErrorInvalidValue;
        kern = packed_step_kernel<4, 128, 10, KDA, true, true, false, kLtU8, true>;
    }
    if (!kern && hmap) {
        switch (rl) {
            case 0: DAMP_PICK4_HMAP(0) break;
            case 1: DAMP_PICK4_HMAP(1) break;
            case 2: DAMP_PICK4_HMAP(2) break;
            case 3: DAMP_PICK4_HMAP(3) break;
            case 4: DAMP_PICK4_HMAP(4) break;
            default: break;
        }
        if (!kern) return cudaErrorInvalidValue;
    }
    // compile-time layouts: d_k = d_v = 128 with the K_hi values below, three record stages
    // (the kernel takes the stage size and the operand buffer's layout as constants)
    const bool fixed_ok = a.dk == 128 && a.dv == 128 && p.nstage == 3;
#define DAMP_FIXED(KC_)                                                                           \
    if (!kern && fixed_ok && a.K == KC_) {                                                        \
        DAMP_PICK4((128 - KC_ + 31) / 32, 128, KC_)                                               \
    }
    // (the 4-bit and FP8 tiers: uniform and FP16 + low tier at K_hi = 16)
    DAMP_FIXED(0)
    DAMP_FIXED(16)
    if constexpr (LT == kLtU8) {
        DAMP_FIXED(4)
        DAMP_FIXED(8)
        DAMP_FIXED(10)
        DAMP_FIXED(32)
    }
    // general kernels: K_hi = 0 (no FP16 tier) or any K_hi, runtime d_k
#define DAMP_GENERAL(RL_)                                                                         \
    if (!kern && rl == RL_) {                                                                     \
        if constexpr (LT == kLtU8) {                                                              \
            if (a.K == 0) DAMP_PICK4(RL_, 0, 0)                                                   \
        }                                                                                         \
        if (!kern) DAMP_PICK4(RL_, 0, -1)                                                         \
    }
    if (!kern && rl == 0) {
        DAMP_PICK4(0, 0, -1)
    }
    DAMP_GENERAL(1)
    DAMP_GENERAL(2)
    DAMP_GENERAL(3)
    DAMP_GENERAL(4)
#undef DAMP_GENERAL
#undef DAMP_FIXED
#undef DAMP_PICK4
#undef DAMP_PICK4_HMAP
    if (!kern) return cudaErrorInvalidValue;
    cudaError_t e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, 32 * warps, smem, stream>>>(p);
    return cudaGetLastError();
}

// Two head groups of a layer in one launch (packed_step2_kernel): the K_hi pairs of the
// paper's head-budget table (12/20, 8/24, 4/28 of 128 key channels) with BF16 operands and
// the UINT8 tiers.  Returns cudaErrorNotSupported (nothing launched) for other pairs.
template <bool KDA>
static cudaError_t launch_packed2_impl(const StepArgs &a1, const StepArgs &a2, cudaStream_t stream,
                                       uint32_t *status) {
    const StepArgs *g1 = &a1, *g2 = &a2;
    if (g1->K > g2->K) std::swap(g1, g2);
    for (const StepArgs *g : {g1, g2})
        if (g->dk != 128 || !g->in_bf16 || (g->fmt != 0 && g->fmt != 1) || !g->head_map) return cudaErrorNotSupported;
    if (g1->fmt != g2->fmt || g1->dv != 128 || g2->dv != 128) return cudaErrorNotSupported;
    PackedLaunch s1, s2;
    cudaError_t e = packed_launch_shape<KDA>(*g1, status, &s1);
    if (e != cudaSuccess) return e;
    if ((e = packed_launch_shape<KDA>(*g2, status, &s2)) != cudaSuccess) return e;
    if (s1.warps != kPackedWarps || s2.warps != kPackedWarps || s1.p.nstage != 3 || s2.p.nstage != 3)
        return cudaErrorNotSupported;
    const int64_t t1 = s1.p.total_tiles, t2 = s2.p.total_tiles;
    if (t1 == 0 || t2 == 0) return cudaErrorNotSupported;  // one group alone: the one-group launch
    const bool had = fmt_had(g1->fmt);
    void (*kern)(PackedParams, PackedParams) = nullptr;
#define DAMP_PAIR2(A_, B_)                                                                         \
    if (g1->K == A_ && g2->K == B_)                                                                \
        kern = had ? packed_step2_kernel<A_, B_, KDA, true, true> : packed_step2_kernel<A_, B_, KDA, false, true>;
    DAMP_PAIR2(12, 20)
    DAMP_PAIR2(8, 24)
    DAMP_PAIR2(4, 28)
#undef DAMP_PAIR2
    if (!kern) return cudaErrorNotSupported;
    // one warp stride for both bodies (each group's stages and operand buffers fit in it)
    const int ws = std::max(s1.p.warp_smem, s2.p.warp_smem);
    s1.p.warp_smem = s2.p.warp_smem = ws;
    const int smem = ws * kPackedWarps;
    if (smem > max_smem_per_block()) return cudaErrorNotSupported;
    if ((e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem)) != cudaSuccess) return e;
    const int grid = (int)std::min<int64_t>(std::max<int64_t>((std::max(t1, t2) + kPackedWarps - 1) / kPackedWarps, 1),
                                            (int64_t)sm_count());
    kern<<<grid, 32 * kPackedWarps, smem, stream>>>(s1.p, s2.p);
    return cudaGetLastError();
}

}  // namespace damp
