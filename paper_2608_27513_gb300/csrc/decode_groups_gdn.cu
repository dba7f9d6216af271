// decode_groups_gdn.cu -- instantiations of the two-group packed decode step for
// GDN (scalar decay per head): two head groups of a layer (K_hi pairs 12/20, 8/24, 4/28) in one launch.
#include "launch_packed.cuh"

namespace damp {

static __device__ uint32_t g_status_groups_gdn;

cudaError_t launch_packed2_gdn(const StepArgs &a1, const StepArgs &a2, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_groups_gdn, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_packed2_impl<false>(a1, a2, s, status);
}

cudaError_t take_status_groups_gdn(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_groups_gdn, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_groups_gdn, &zero, sizeof(uint32_t));
}

}  // namespace damp
