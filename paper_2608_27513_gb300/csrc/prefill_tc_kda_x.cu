// prefill_tc_kda_x.cu -- launcher of the KDA prefill chunk on the tensor cores
// (prefill_tc_kda.cuh), d_k = d_v = 128, bf16 q/k/v: the UINT4 tiers with and without H_32
// (formats 3, 4; FP8 E4M3 chunks keep the per-token kernel).
#include <algorithm>

#include "damp_internal.h"
#include "prefill_tc_kda.cuh"

namespace damp {

cudaError_t launch_prefill_tc_kda_x(const PrefillParams &p, int fmt, cudaStream_t stream) {
    void (*kern)(PrefillParams) = nullptr;
    if (fmt == kFmtU4H32) kern = prefill_tc_kda_kernel<kFmtU4H32>;
    if (fmt == kFmtU4) kern = prefill_tc_kda_kernel<kFmtU4>;
    if (!kern) return cudaErrorNotSupported;
    const int smem = kKdSmem;
    if (p.rec_bytes > kKdMaxRec || smem > max_smem_per_block()) return cudaErrorNotSupported;
    // The CTA allocates all 512 tensor-memory columns of its SM, so a second CTA there
    // would wait in its allocation: the shared memory must keep it off the SM.
    const int per_sm = max_smem_per_sm();
    if (per_sm <= 0 || 2 * smem <= per_sm) return cudaErrorNotSupported;
    cudaError_t e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    const int64_t units = (int64_t)p.batch * p.H;
    const int grid = (int)std::min<int64_t>(units, (int64_t)sm_count());
    kern<<<grid, kKdThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace damp
