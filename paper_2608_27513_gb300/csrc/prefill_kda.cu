// prefill_kda.cu -- instantiations of the prefill chunk kernel for
// KDA (per-key-channel decay), UINT8 low tiers (formats 0 and 1); the 4-bit and FP8 tiers are
// instantiated in prefill_kda_x.cu.
#include "launch_prefill.cuh"

namespace damp {

static __device__ uint32_t g_status_prefill_kda;

cudaError_t launch_prefill_kda(const StepArgs &a, cudaStream_t s) {
    if (a.fmt != kFmtU8H32 && a.fmt != kFmtU8) return launch_prefill_kda_x(a, s);
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_prefill_kda, cache, &status);
    if (e != cudaSuccess) return e;
    return a.fmt == kFmtU8H32 ? launch_prefill_impl<true, kFmtU8H32>(a, s, status)
                              : launch_prefill_impl<true, kFmtU8>(a, s, status);
}

cudaError_t take_status_prefill_kda(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_prefill_kda, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_prefill_kda, &zero, sizeof(uint32_t));
}

}  // namespace damp
