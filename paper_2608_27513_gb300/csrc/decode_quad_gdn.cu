// decode_quad_gdn.cu -- instantiations of the row-absmax quad decode step for
// GDN (scalar decay per head).
#include "launch_quad.cuh"

namespace damp {

static __device__ uint32_t g_status_quad_gdn;

cudaError_t launch_quad_rowabs_gdn(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_quad_gdn, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_quad_rowabs_impl<false>(a, s, status);
}

cudaError_t take_status_quad_gdn(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_quad_gdn, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_quad_gdn, &zero, sizeof(uint32_t));
}

}  // namespace damp
