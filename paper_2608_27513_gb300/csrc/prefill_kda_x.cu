// prefill_kda_x.cu -- instantiations of the prefill chunk kernel for
// KDA (per-key-channel decay) with the row-absmax INT8, UINT4 (+ H_32) and FP8 E4M3 low tiers (formats 2, 3, 4, 5).
#include "launch_prefill.cuh"

namespace damp {

static __device__ uint32_t g_status_prefill_kda_x;

cudaError_t launch_prefill_kda_x(const StepArgs &a, cudaStream_t s) {
    static std::atomic<uint32_t *> cache[64];
    uint32_t *status = nullptr;
    cudaError_t e = symbol_address_cached(&g_status_prefill_kda_x, cache, &status);
    if (e != cudaSuccess) return e;
    switch (a.fmt) {
        case kFmtU4H32: return launch_prefill_impl<true, kFmtU4H32>(a, s, status);
        case kFmtU4: return launch_prefill_impl<true, kFmtU4>(a, s, status);
        case kFmtE4M3: return launch_prefill_impl<true, kFmtE4M3>(a, s, status);
        case kFmtS8Row: return launch_prefill_impl<true, kFmtS8Row>(a, s, status);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t take_status_prefill_kda_x(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_prefill_kda_x, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_prefill_kda_x, &zero, sizeof(uint32_t));
}

}  // namespace damp
