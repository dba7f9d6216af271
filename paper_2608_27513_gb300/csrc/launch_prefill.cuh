// launch_prefill.cuh -- host-side launcher of the prefill chunk kernel.  Included
// once per decay kind (GDN / KDA) so the instantiations compile in parallel.
#pragma once

#include <algorithm>

#include "damp_internal.h"
#include "formats.cuh"
#include "prefill.cuh"

namespace damp {

constexpr int kPrefillWarps = 8;

template <bool KDA, int FMT>
static cudaError_t launch_prefill_impl(const StepArgs &a, cudaStream_t stream, uint32_t *status) {
    const int V = a.dv / kG;
    const RecGeom rg = rec_geom(a.dk, a.K, FMT);
    const int esz = a.in_bf16 ? 2 : 4;
    auto up16 = [](int x) { return (x + 15) & ~15; };
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
    // per-warp shared memory: [column-sum buffer][H d][pi][2 token buffers]
    int off = 32 * kPartStride * 4;
    p.dvec_off = off;
    off += 32 * 4;
    p.perm_off = off;
    off += up16(a.dk);
    p.ops_off = off;
    int t = 0;
    p.off_q = t;
    t += up16(a.dk * esz);
    p.off_k = t;
    t += up16(a.dk * esz);
    p.off_g = t;
    t += KDA ? up16(a.dk * 4) : 16;
    p.off_v = t;
    t += up16(kG * esz);
    p.off_beta = t;
    t += 16;
    p.ops_bytes = t;
    off += 2 * t;
    p.warp_smem = (off + 127) & ~127;
    if (p.total_tiles == 0 || a.T == 0) return cudaSuccess;

    int warps = kPrefillWarps;
    while (warps > 1 && warps * p.warp_smem > max_smem_per_block()) --warps;
    if (warps * p.warp_smem > max_smem_per_block()) return cudaErrorInvalidValue;
    const int64_t want = (p.total_tiles + warps - 1) / warps;
    const int grid = (int)std::min<int64_t>(want, (int64_t)sm_count());
    const int smem = p.warp_smem * warps;

    void (*kern)(PrefillParams) = nullptr;
#define DAMP_PICK(R_)                                                                              \
    if (a.dk == 32 * R_) kern = a.in_bf16 ? prefill_chunk_kernel<R_, KDA, FMT, true> : prefill_chunk_kernel<R_, KDA, FMT, false>;
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
