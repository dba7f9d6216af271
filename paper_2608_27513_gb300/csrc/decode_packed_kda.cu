// decode_packed_kda.cu -- instantiations of the fused packed decode step for
// KDA (per-key-channel decay, Lambda_t = diag(exp(g_t))).
#include "launch_packed.cuh"

namespace damp {

static __device__ uint32_t g_status_packed_kda;

cudaError_t launch_packed_kda(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_packed_kda, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_packed_impl<true, kLtU8>(a, s, status);
}

// The bounded-wait test instance (see packed_step_kernel's WAITTEST); it reports
// through the same status word as the KDA decode step.
cudaError_t launch_packed_kda_waittest(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_packed_kda, cache, &status);
    if (e != cudaSuccess) return e;
    return launch_packed_impl<true, kLtU8, true>(a, s, status);
}

cudaError_t take_status_packed_kda(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_packed_kda, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_packed_kda, &zero, sizeof(uint32_t));
}

}  // namespace damp
