// decode_packed_gdn.cu -- instantiations of the fused packed decode step for
// GDN (scalar decay per head, Lambda_t = alpha_t I).
#include "launch_packed.cuh"

namespace damp {

static __device__ uint32_t g_status_packed_gdn;

cudaError_t launch_packed_gdn(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_packed_gdn, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_packed_impl<false, kLtU8>(a, s, status);
}

cudaError_t take_status_packed_gdn(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_packed_gdn, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_packed_gdn, &zero, sizeof(uint32_t));
}

}  // namespace damp
