// decode_packed_kda_f8.cu -- instantiations of the fused packed decode step for
// KDA (per-key-channel decay, Lambda_t = diag(exp(g_t))) with the FP8 E4M3 low tier (format 5).
#include "launch_packed.cuh"

namespace damp {

static __device__ uint32_t g_status_packed_kda_f8;

cudaError_t launch_packed_kda_f8(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_packed_kda_f8, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_packed_impl<true, kLtE4M3>(a, s, status);
}

cudaError_t take_status_packed_kda_f8(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_packed_kda_f8, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_packed_kda_f8, &zero, sizeof(uint32_t));
}

}  // namespace damp
