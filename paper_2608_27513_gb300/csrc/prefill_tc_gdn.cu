// prefill_tc_gdn.cu -- launcher of the GDN prefill chunk on the tensor cores
// (prefill_tc.cuh): UINT8 tiers (with and without H_32), d_k = d_v = 128, bf16 q/k/v.
#include <algorithm>

#include "damp_internal.h"
#include "prefill_tc.cuh"

namespace damp {

cudaError_t launch_prefill_tc_gdn(const PrefillParams &p, bool had, cudaStream_t stream) {
    const int smem = kTcSmem;
    if (p.rec_bytes > kTcMaxRec || smem > max_smem_per_block()) return cudaErrorNotSupported;
    // The CTA allocates all 512 tensor-memory columns of its SM, so a second CTA there
    // would wait in its allocation: the shared memory must keep it off the SM.
    const int per_sm = max_smem_per_sm();
    if (per_sm <= 0 || 2 * smem <= per_sm) return cudaErrorNotSupported;
    void (*kern)(PrefillParams) = had ? prefill_tc_gdn_kernel<true> : prefill_tc_gdn_kernel<false>;
    cudaError_t e = ensure_smem_limit(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    const int64_t units = (int64_t)p.batch * p.H;
    const int grid = (int)std::min<int64_t>(units, (int64_t)sm_count());
    kern<<<grid, kTcThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace damp
