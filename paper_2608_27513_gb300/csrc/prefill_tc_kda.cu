// prefill_tc_kda.cu -- launcher of the KDA prefill chunk on the tensor cores
// (prefill_tc_kda.cuh), d_k = d_v = 128, bf16 q/k/v: the UINT8 tiers (formats 0 and 1).
#include <algorithm>

#include "damp_internal.h"
#include "prefill_tc_kda.cuh"

namespace damp {

cudaError_t launch_prefill_tc_kda(const PrefillParams &p, int fmt, cudaStream_t stream) {
    void (*kern)(PrefillParams) = nullptr;
    if (fmt == kFmtU8H32) kern = prefill_tc_kda_kernel<kFmtU8H32>;
    if (fmt == kFmtU8) kern = prefill_tc_kda_kernel<kFmtU8>;
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
