// decode_groups_kda.cu -- instantiations of the two-group packed decode step for
// KDA (per-key-channel decay): two head groups of a layer (K_hi pairs 12/20, 8/24, 4/28) in one launch.
#include "launch_packed.cuh"

namespace damp {

static __device__ uint32_t g_status_groups_kda;

cudaError_t launch_packed2_kda(const StepArgs &a1, const StepArgs &a2, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_groups_kda, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_packed2_impl<true>(a1, a2, s, status);
}

cudaError_t take_status_groups_kda(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_groups_kda, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_groups_kda, &zero, sizeof(uint32_t));
}

}  // namespace damp
