// launch_prefill.cuh -- host-side launcher of the prefill chunk kernel.  Included
// once per decay kind (GDN / KDA) so the instantiations compile in parallel.
#pragma once

#include <algorithm>

#include "damp_internal.h"
#include "formats.cuh"
#include "prefill.cuh"
#include "prefill_cg.cuh"

namespace damp {

constexpr int kPrefillWarps = 8;
// Chunks of at least this many tokens on the UINT8 tiers (d_k 64 or 128, o 16-byte
// aligned) run prefill_cg_kernel, whose per-token work is lower and per-tile work higher;
// shorter chunks and the other tiers run prefill_chunk_kernel.
constexpr int kPrefillCgMinT = 32;
// GDN and KDA chunks of at least this many tokens with d_k = d_v = 128, bf16 inputs, a
// 16-byte aligned o and an affine low tier (UINT8 or UINT4, with or without H_32) run the
// tensor-core kernels (prefill_tc_gdn.cu / prefill_tc_kda.cu: formats 0, 1; the _x units:
// formats 3, 4).  FP8 E4M3 keeps the per-token kernels: its code spacing is relative, so a
// value far below its group's maximum has a spacing finer than the closed form's rounding
// error (absolute, about 2^-24 of the largest terms of its sums).
constexpr int kPrefillTcMinT = 32;
cudaError_t launch_prefill_tc_gdn(const PrefillParams &p, int fmt, cudaStream_t stream);
cudaError_t launch_prefill_tc_gdn_x(const PrefillParams &p, int fmt, cudaStream_t stream);
cudaError_t launch_prefill_tc_kda(const PrefillParams &p, int fmt, cudaStream_t stream);
cudaError_t launch_prefill_tc_kda_x(const PrefillParams &p, int fmt, cudaStream_t stream);

template <bool KDA, bool HAD>
static cudaError_t launch_prefill_cg(const PrefillParams &p0, const StepArgs &a, int rec_bytes, cudaStream_t stream) {
    PrefillParams p = p0;
    const int warp_smem = ((prefill_cg_smem(a.dk, KDA, a.in_bf16).stage_off + rec_bytes + 127) & ~127) + 128 * a.K;
    p.warp_stride = warp_smem;
    int warps = kPrefillWarps;
    while (warps > 1 && warps * warp_smem > max_smem_per_block()) --warps;
    if (warps * warp_smem > max_smem_per_block()) return cudaErrorInvalidValue;
    const int64_t want = (p.total_tiles + warps - 1) / warps;
    const int grid = (int)std::min<int64_t>(want, (int64_t)sm_count());
    const int smem = warp_smem * warps;
    void (*kern)(PrefillParams) = nullptr;
    if (a.dk == 64) kern = a.in_bf16 ? prefill_cg_kernel<64, KDA, HAD, true> : prefill_cg_kernel<64, KDA, HAD, false>;
    if (a.dk == 128) kern = a.in_bf16 ? prefill_cg_kernel<128, KDA, HAD, true> : prefill_cg_kernel<128, KDA, HAD, false>;
    if (!kern) return cudaErrorInvalidValue;
    cudaError_t e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, 32 * warps, smem, stream>>>(p);
    return cudaGetLastError();
}

template <bool KDA, int FMT>
static cudaError_t launch_prefill_impl(const StepArgs &a, cudaStream_t stream, uint32_t *status) {
    const int V = a.dv / kG;
    const RecGeom rg = rec_geom(a.dk, a.K, FMT);
    PrefillParams p{};
    p.state = static_cast<uint8_t *>(a.state);
    p.num_slots = a.num_slots;
    p.slot_idx = a.slot_idx;
    p.lengths = a.lengths;
    p.perm = a.perm;
    p.q = a.q;
    p.k = a.k;
    p.v = a.v;
    p.g = a.g;
    p.beta = a.beta;
    p.o = a.o;
    p.batch = a.batch;
    p.T = a.T;
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
    p.total_tiles = (int64_t)a.batch * a.H * V;
    p.status = status;
    const int warp_smem = prefill_smem(a.dk, KDA, a.in_bf16).warp_bytes + 128 + ((rg.bytes + 127) & ~127);
    p.warp_stride = warp_smem;
    if (p.total_tiles == 0 || a.T == 0) return cudaSuccess;
    if constexpr (FMT != kFmtS8Row && FMT != kFmtE4M3) {
        if (a.T >= kPrefillTcMinT && a.dk == 128 && a.dv == 128 && a.in_bf16 &&
            (reinterpret_cast<uintptr_t>(a.o) & 15) == 0) {
            constexpr bool u8 = FMT == kFmtU8H32 || FMT == kFmtU8;
            const cudaError_t e = KDA ? (u8 ? launch_prefill_tc_kda(p, FMT, stream) : launch_prefill_tc_kda_x(p, FMT, stream))
                                      : (u8 ? launch_prefill_tc_gdn(p, FMT, stream) : launch_prefill_tc_gdn_x(p, FMT, stream));
            if (e != cudaErrorNotSupported) return e;
        }
    }
    if constexpr (FMT == kFmtU8H32 || FMT == kFmtU8) {
        if (a.T >= kPrefillCgMinT && (a.dk == 64 || a.dk == 128) && (reinterpret_cast<uintptr_t>(a.o) & 15) == 0)
            return launch_prefill_cg<KDA, FMT == kFmtU8H32>(p, a, rg.bytes, stream);
    }

    int warps = kPrefillWarps;
    int64_t want;
    int extra = 0;
    if constexpr (FMT == kFmtS8Row) {
        // groups of four warps share each row's maximum over the value blocks of a head
        if (V > 4) return cudaErrorInvalidValue;
        extra = (warps / 4) * 2 * 4 * 128 * 4;  // per group: two buffers of [4 blocks][128 rows]
        if (warps * warp_smem + extra > max_smem_per_block()) return cudaErrorInvalidValue;
        const int64_t units = p.total_tiles / V;
        want = (units + warps / 4 - 1) / (warps / 4);
    } else {
        while (warps > 1 && warps * warp_smem > max_smem_per_block()) --warps;
        if (warps * warp_smem > max_smem_per_block()) return cudaErrorInvalidValue;
        want = (p.total_tiles + warps - 1) / warps;
    }
    p.amax_off = warps * warp_smem;
    const int grid = (int)std::min<int64_t>(want, (int64_t)sm_count());
    const int smem = warp_smem * warps + extra;

    void (*kern)(PrefillParams) = nullptr;
#define DAMP_PICK(R_)                                                                              \
    if constexpr (FMT == kFmtS8Row) {                                                              \
        if (a.dk == 32 * R_) kern = a.in_bf16 ? prefill_row_kernel<R_, KDA, true> : prefill_row_kernel<R_, KDA, false>; \
    } else {                                                                                       \
        if (a.dk == 32 * R_) kern = a.in_bf16 ? prefill_chunk_kernel<R_, KDA, FMT, true> : prefill_chunk_kernel<R_, KDA, FMT, false>; \
    }
    DAMP_PICK(1)
    DAMP_PICK(2)
    DAMP_PICK(4)
#undef DAMP_PICK
    if (!kern) return cudaErrorInvalidValue;
    cudaError_t e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, 32 * warps, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace damp
