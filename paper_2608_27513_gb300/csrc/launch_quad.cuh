// launch_quad.cuh -- host-side launcher of the full-row quad step (qfr_step_kernel)
// for the row-absmax INT8 low tier at d_k = d_v = 128.  Included once per decay kind
// (GDN / KDA) so the two sets of instantiations compile in parallel.
#pragma once

#include <algorithm>

#include "damp_internal.h"
#include "decode_quad.cuh"

namespace damp {

// Returns cudaErrorNotSupported (nothing launched) for a layout without a compile-time
// instance; the caller then runs the one-token chunk path.
template <bool KDA>
static cudaError_t launch_quad_rowabs_impl(const StepArgs &a, cudaStream_t stream, uint32_t *status) {
    if (a.dk != 128 || a.dv != 128 || !a.in_bf16 || a.fmt != 2) return cudaErrorNotSupported;
    const int64_t units = (int64_t)a.batch * a.H;
    if (units >= (int64_t(1) << 29)) return cudaErrorNotSupported;  // 32-bit unit and tile indices
    void (*kern)(QuadParams) = nullptr;
    int smem = 0, rec = 0;
#define DAMP_QFR(KC_)                                                        \
    if (a.K == KC_) {                                                        \
        kern = qfr_step_kernel<KC_, KDA, false, true, true>;                 \
        smem = QfrGeom<KC_, KDA, true>::SMEM;                                \
        rec = QuadGeom<KC_, KDA, true>::REC;                                 \
    }
    DAMP_QFR(0)
    DAMP_QFR(4)
    DAMP_QFR(8)
    DAMP_QFR(10)
    DAMP_QFR(16)
    DAMP_QFR(32)
#undef DAMP_QFR
    if (!kern) return cudaErrorNotSupported;
    if (smem > max_smem_per_block()) return cudaErrorNotSupported;
    QuadParams p{};
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
    p.slot_bytes = (int64_t)a.H * 4 * rec;
    p.total_tiles = units * 4;
    p.status = status;
    if (units == 0) return cudaSuccess;
    cudaError_t e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    // one CTA (two quads) per SM, fewer when there are fewer units than quads
    const int grid = (int)std::min<int64_t>((units + kQfrWarps / 4 - 1) / (kQfrWarps / 4), (int64_t)sm_count());
    kern<<<grid, 32 * kQfrWarps, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace damp
