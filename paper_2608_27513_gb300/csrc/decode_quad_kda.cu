// decode_quad_kda.cu -- instantiations of the row-absmax quad decode step for
// KDA (per-key-channel decay).
#include "launch_quad.cuh"

namespace damp {

static __device__ uint32_t g_status_quad_kda;

cudaError_t launch_quad_rowabs_kda(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_quad_kda, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_quad_rowabs_impl<true>(a, s, status);
}

cudaError_t take_status_quad_kda(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_quad_kda, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_quad_kda, &zero, sizeof(uint32_t));
}

}  // namespace damp
