// damp_internal.h -- host-side parameter blocks and launcher declarations shared
// by libdamp's translation units (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace damp {

struct StepArgs {
    // layout; per-head operands and outputs are indexed by model head
    // m = head_map ? head_map[h] : h over Hm heads
    int32_t H, Hqk, dk, dv, K, fmt;
    int32_t Hm;
    const int32_t *head_map;
    // buffers
    void *state;  // packed pool or FP32 state
    int64_t num_slots;
    const int32_t *slot_idx;
    int32_t batch;
    const uint8_t *perm;
    const void *q, *k, *v;
    const float *g, *beta;
    float *o;
    int32_t in_bf16;  // 1: q/k/v are bf16, 0: fp32
    int32_t kda;      // 1: per-channel decay g[B][H][d_k], 0: scalar g[B][H]
    // prefill chunks only: tokens per chunk (operands gain a [T] axis after the batch
    // axis) and optional per-row lengths
    int32_t T;
    const int32_t *lengths;
};

struct ConvArgs {
    int32_t H, dk, dv, K, fmt;
    int32_t Hm;                // heads of S (rows head_map[h], or h)
    const int32_t *head_map;
    void *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    int32_t batch;
    const uint8_t *perm;
    float *S;  // natural FP32 states [batch][H][d_k][d_v]
    uint16_t *hi;
    uint8_t *codes;
    uint16_t *meta;
};

// Launchers (return the CUDA error of the launch; they perform no host-side argument checks).
cudaError_t launch_packed_gdn(const StepArgs &a, cudaStream_t s);
cudaError_t launch_packed_kda(const StepArgs &a, cudaStream_t s);
cudaError_t launch_packed_kda_waittest(const StepArgs &a, cudaStream_t s);
// two head groups of a layer in one launch (cudaErrorNotSupported, nothing launched, for
// a pair of layouts without a compile-time instance)
cudaError_t launch_packed2_gdn(const StepArgs &a1, const StepArgs &a2, cudaStream_t s);
cudaError_t launch_packed2_kda(const StepArgs &a1, const StepArgs &a2, cudaStream_t s);
// the UINT4 low tiers (formats 3, 4)
cudaError_t launch_packed_gdn_u4(const StepArgs &a, cudaStream_t s);
cudaError_t launch_packed_kda_u4(const StepArgs &a, cudaStream_t s);
// the FP8 E4M3 low tier (format 5)
cudaError_t launch_packed_gdn_f8(const StepArgs &a, cudaStream_t s);
cudaError_t launch_packed_kda_f8(const StepArgs &a, cudaStream_t s);
// the row-absmax format (2) at d_k = d_v = 128 with BF16 operands and a compile-time
// K_hi: the full-row quad step (cudaErrorNotSupported, nothing launched, otherwise)
cudaError_t launch_quad_rowabs_gdn(const StepArgs &a, cudaStream_t s);
cudaError_t launch_quad_rowabs_kda(const StepArgs &a, cudaStream_t s);
cudaError_t launch_fp32_step(const StepArgs &a, cudaStream_t s);
cudaError_t launch_quantize(const ConvArgs &a, cudaStream_t s);
cudaError_t launch_dequantize(const ConvArgs &a, cudaStream_t s);
cudaError_t launch_pack_tiers(const ConvArgs &a, cudaStream_t s);
cudaError_t launch_unpack_tiers(const ConvArgs &a, cudaStream_t s);
// One prefill chunk on the packed state (formats 0 and 1).
cudaError_t launch_prefill_gdn(const StepArgs &a, cudaStream_t s);
cudaError_t launch_prefill_kda(const StepArgs &a, cudaStream_t s);
cudaError_t launch_prefill_gdn_x(const StepArgs &a, cudaStream_t s);  // formats 3, 4, 5
cudaError_t launch_prefill_kda_x(const StepArgs &a, cudaStream_t s);
// Offline key-channel selection (Sec. 5.1, Algorithm 1).
cudaError_t launch_calib_error_energy(const float *S, int32_t batch, int32_t H, int32_t Hm, const int32_t *head_map,
                                      int32_t dk, int32_t dv, int32_t fmt, float *E_acc, cudaStream_t s);
cudaError_t launch_calib_log_decay(const float *g, int32_t batch, int32_t H, int32_t Hm, const int32_t *head_map,
                                   int32_t dk, int32_t kda, float *G_acc, cudaStream_t s);
cudaError_t launch_calib_select(const float *E_acc, int64_t n_samples, const float *G_acc, int64_t n_tokens, float tau,
                                int32_t H, int32_t Hm, const int32_t *head_map, int32_t dk, int32_t k_hi,
                                float *C_out, uint8_t *perm_out, cudaStream_t s);
cudaError_t take_status_calib(uint32_t *bits);
// Row-absmax INT8 low tier (lo_format 2); op: 0 quantize, 1 dequantize, 2 pack, 3 unpack.
cudaError_t launch_rowabs_step(const StepArgs &a, cudaStream_t s);
cudaError_t launch_rowabs_convert(const ConvArgs &a, int op, cudaStream_t s);

// Read-and-clear of each translation unit's device status word.
cudaError_t take_status_packed_gdn(uint32_t *bits);
cudaError_t take_status_packed_kda(uint32_t *bits);
cudaError_t take_status_packed_gdn_u4(uint32_t *bits);
cudaError_t take_status_packed_kda_u4(uint32_t *bits);
cudaError_t take_status_packed_gdn_f8(uint32_t *bits);
cudaError_t take_status_packed_kda_f8(uint32_t *bits);
cudaError_t take_status_groups_gdn(uint32_t *bits);
cudaError_t take_status_groups_kda(uint32_t *bits);
cudaError_t take_status_quad_gdn(uint32_t *bits);
cudaError_t take_status_quad_kda(uint32_t *bits);
cudaError_t take_status_fp32(uint32_t *bits);
cudaError_t take_status_convert(uint32_t *bits);
cudaError_t take_status_rowabs(uint32_t *bits);
cudaError_t take_status_prefill_gdn(uint32_t *bits);
cudaError_t take_status_prefill_kda(uint32_t *bits);
cudaError_t take_status_prefill_gdn_x(uint32_t *bits);
cudaError_t take_status_prefill_kda_x(uint32_t *bits);

// Streaming multiprocessors / opt-in shared memory per block of the current device (cached per device).
int sm_count();
int max_smem_per_block();
int max_smem_per_sm();  // shared memory of one SM (0 if unknown)

// Raises a kernel's dynamic shared-memory limit to at least `bytes` on the current
// device (the attribute call is made once per kernel, device and larger size).
cudaError_t ensure_smem_limit(const void *kernel, int bytes);

// Device address of a __device__ status word, looked up once per device.
// The device address of a status-word symbol, looked up once per device (the cache is
// an array of 64 per-device slots, written atomically: concurrent first calls store the
// same address).
cudaError_t symbol_address_cached(const void *symbol, std::atomic<uint32_t *> *cache_per_device, uint32_t **out);

}  // namespace damp
