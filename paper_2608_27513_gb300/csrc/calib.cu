// calib.cu -- offline key-channel selection on the GPU (Sec. 5.1; App. A.2; Algorithm 1).
//
//   calib_error_energy   E_acc[h][u] += sum_b || Q_lo(S_b,h)_{u:} - S_b,h,u: ||^2
//                        (Eq. empirical_error_energy: the low-tier round trip of every
//                        key-channel row of the sampled states, in the layout's format)
//   calib_log_decay      G_acc[h][u] += sum_b log a_{b,h,u}   (GDN: the head's scalar)
//   calib_select         E = E_acc / n_samples, a_eff = exp(G_acc / n_tokens),
//                        P = 1 / max(1 - a_eff^2, tau), C = E P, H = TopK_{K_hi}(C)
//                        (ties to the lower channel), pi = stable partition (H first,
//                        each part in ascending channel order)
//
// Per-head rows of S, g, E_acc and G_acc are model heads (head_map[h], or h); C_out and
// perm_out rows are the layout's own heads.  A head_map entry outside 0 .. Hm-1 makes the
// head's work a no-op and sets kDevBadHead in the status word.
//
// Every accumulator entry has exactly one writer per call and sums in a fixed order,
// so repeated runs give the same bits; no global scratch is used (partials of the
// error energy meet in shared memory).
#include "damp_common.cuh"
#include "damp_internal.h"
#include "formats.cuh"

#include <algorithm>

namespace damp {

namespace {

// One CTA per (head, 32 key channels); warp w takes batch rows w, w + 16, ...; lane u
// accumulates its row's error over those rows and the value blocks; the sixteen warp
// partials are added in warp order (a fixed order: the result does not depend on
// scheduling).
constexpr int kEeWarps = 16;
constexpr int kEeRow = 36;  // floats per row of a warp's staging tile (32 + 4 of padding)
constexpr int kEeTile = 32 * kEeRow / 4;  // float4 per staging tile
constexpr int kEeStages = 3;
constexpr int kEeSmem = kEeWarps * kEeStages * kEeTile * 16;

__device__ uint32_t g_status_calib;

// model head of held head h, or -1 (flagged) when the map entry is out of range
__device__ __forceinline__ int calib_model_head(const int32_t *head_map, int h, int Hm) {
    const int m = head_map ? head_map[h] : h;
    if (m < 0 || m >= Hm) {
        atomicOr(&g_status_calib, (uint32_t)kDevBadHead);
        return -1;
    }
    return m;
}

template <int FMT>
__global__ void __launch_bounds__(32 * kEeWarps) calib_error_energy_kernel(const float *S, int32_t batch, int32_t H,
                                                                           int32_t Hm, const int32_t *head_map,
                                                                           int32_t dk, int32_t dv, float *E_acc) {
    __shared__ float partial[kEeWarps][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int groups = (dk + 31) / 32;
    const int h = (int)(blockIdx.x / groups);
    const int u = (int)(blockIdx.x % groups) * 32 + lane;  // d_k is a multiple of 32
    const int m = calib_model_head(head_map, h, Hm);  // the same for the whole CTA
    if (m < 0) return;
    float err = 0.f;
    if constexpr (FMT == 2) {
        for (int b = warp; b < batch; b += kEeWarps) {
            const float *row = S + (((int64_t)b * Hm + m) * dk + u) * dv;
            // per-row symmetric absmax INT8: s = max|x| / 127, q = sat(rne(x / s)), x^ = s q
            float amax = 0.f;
            for (int j = 0; j < dv; ++j) amax = fmaxf(amax, fabsf(row[j]));
            const float s = __fdiv_rn(amax, 127.f);
            for (int j = 0; j < dv; ++j) {
                float t = s == 0.f ? 0.f : rintf(__fdiv_rn(row[j], s));
                t = fminf(fmaxf(t, -127.f), 127.f);
                const float dlt = __fmul_rn(s, t) - row[j];
                err = fmaf(dlt, dlt, err);
            }
        }
    } else {
        // items (row b, value block c) of this warp in the order b = warp, warp + 16, ...,
        // c = 0 .. V-1.  An item is the 32 x 32 tile S[b, m, u0 .. u0+31, 32c .. 32c+31]:
        // the warp copies it with 16-byte cp.async (each instruction covers four whole
        // 128-B rows) into one of its kEeStages shared-memory tiles (rows padded to 36
        // floats: the row-wise copies and each lane's reads of its own row are free of bank
        // conflicts); two items are in flight while the current one is quantized.
        extern __shared__ float4 ee_tiles[];
        float4 *tiles = ee_tiles + warp * (kEeStages * kEeTile);
        const int Vb = dv / kG;
        const int nb = warp < batch ? (batch - warp + kEeWarps - 1) / kEeWarps : 0;
        const int n_items = nb * Vb;
        const int u0 = u - lane, lr = lane >> 3, lc = lane & 7;
        auto issue_item = [&](int i) {
            if (i < n_items) {
                const int bi = i / Vb, c = i - bi * Vb;
                const float *base =
                    S + (((int64_t)(warp + kEeWarps * bi) * Hm + m) * dk + u0 + lr) * dv + kG * c + 4 * lc;
                const uint32_t dst = smem_u32(tiles + (i % kEeStages) * kEeTile + lr * (kEeRow / 4) + lc);
#pragma unroll
                for (int q = 0; q < 8; ++q) cp_async16(dst + 16 * q * kEeRow, base + (int64_t)(4 * q) * dv);
            }
            cp_async_commit();  // one group per item index, empty past the end
        };
#pragma unroll
        for (int i = 0; i < kEeStages - 1; ++i) issue_item(i);
        for (int i = 0; i < n_items; ++i) {
            __syncwarp();  // every lane is done reading the tile item i + 2 overwrites
            issue_item(i + kEeStages - 1);
            cp_async_wait<kEeStages - 1>();  // this lane's copies of item i have landed
            __syncwarp();                    // ... and every other lane's
            const float4 *tile = tiles + (i % kEeStages) * kEeTile;
            float2 x[16], y[16];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const float4 t = tile[lane * (kEeRow / 4) + q];
                x[2 * q] = make_float2(t.x, t.y);
                x[2 * q + 1] = make_float2(t.z, t.w);
            }
            // x becomes the group in the quantizer's domain (H_32 x for the Hadamard formats):
            // H_32 / sqrt(32) is orthonormal, so ||H^T y - H^T x||^2 = ||y - x||^2 and the
            // error energy is taken there, without the inverse transform
            if (fmt_had(FMT)) hadamard_pairs(x);
#pragma unroll
            for (int q = 0; q < 16; ++q) y[q] = x[q];
            if (FMT == kFmtE4M3) {  // natural domain, one FP32 scale per group
                uint32_t w[8];
                const float sc = quantize_group_e4m3(y, w);
                dequantize_group_e4m3(w, sc, 1.0f, y);
            } else {
#pragma unroll
                for (int q = 0; q < 16; ++q) y[q] = mul2(y[q], splat2(kDown));  // working scale of the quantizer
                if (fmt_u4(FMT)) {
                    uint32_t w[4];
                    const uint32_t sz = quantize_group_u4(y, w);
                    dequantize_group_u4(w, sz, 1.0f, y);
                } else {
                    uint32_t w[8];
                    const uint32_t sz = quantize_group(y, w);
                    dequantize_group(w, sz, 1.0f, y);
                }
            }
#pragma unroll
            for (int q = 0; q < 16; ++q) {
                const float d0 = y[q].x - x[q].x, d1 = y[q].y - x[q].y;
                err = fmaf(d0, d0, fmaf(d1, d1, err));
            }
        }
    }
    partial[warp][lane] = err;
    __syncthreads();
    if (warp == 0) {
        float sum = 0.f;
#pragma unroll
        for (int i = 0; i < kEeWarps; ++i) sum += partial[i][lane];
        E_acc[(int64_t)m * dk + u] += sum;
    }
}

__global__ void calib_log_decay_kernel(const float *g, int32_t batch, int32_t H, int32_t Hm, const int32_t *head_map,
                                       int32_t dk, int32_t kda, float *G_acc) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)H * dk) return;
    const int h = (int)(i / dk), u = (int)(i % dk);
    const int m = calib_model_head(head_map, h, Hm);
    if (m < 0) return;
    float s = 0.f;
    for (int b = 0; b < batch; ++b) s += kda ? g[((int64_t)b * Hm + m) * dk + u] : g[(int64_t)b * Hm + m];
    G_acc[(int64_t)m * dk + u] += s;
}

// One warp per head: scores, rank of every channel, then the stable partition.
__global__ void __launch_bounds__(32) calib_select_kernel(const float *E_acc, float inv_samples, const float *G_acc,
                                                          float inv_tokens, float tau, int32_t H, int32_t Hm,
                                                          const int32_t *head_map, int32_t dk, int32_t k_hi,
                                                          float *C_out, uint8_t *perm_out) {
    __shared__ float sc[256];
    const int lane = threadIdx.x & 31;
    const int h = blockIdx.x;
    if (h >= H) return;
    int m = head_map ? head_map[h] : h;  // warp-uniform
    if (m < 0 || m >= Hm) {
        if (lane == 0) atomicOr(&g_status_calib, (uint32_t)kDevBadHead);
        return;
    }
    for (int u = lane; u < dk; u += 32) {
        const float E = E_acc[(int64_t)m * dk + u] * inv_samples;
        // 1 - a_eff^2 = 1 - exp(2 mean log a) = -expm1(2 mean log a): no cancellation near a = 1
        const float one_minus_a2 = -expm1f(2.0f * (G_acc[(int64_t)m * dk + u] * inv_tokens));
        const float P = 1.0f / fmaxf(one_minus_a2, tau);
        const float C = E * P;
        sc[u] = C;
        C_out[(int64_t)h * dk + u] = C;
    }
    __syncwarp();
    // protected: fewer than K_hi channels rank above u (larger score, or equal score at a lower index)
    unsigned prot_words[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int u0 = 0; u0 < dk; u0 += 32) {
        const int u = u0 + lane;
        const float cu = sc[u];
        int above = 0;
        for (int v = 0; v < dk; ++v) {
            const float cv = sc[v];
            above += (cv > cu) || (cv == cu && v < u);
        }
        prot_words[u0 / 32] = __ballot_sync(kFull, above < k_hi);
    }
    // stable partition: protected channels in ascending order, then the rest
    int n_prot = 0;
    for (int i = 0; i < dk / 32; ++i) n_prot += __popc(prot_words[i]);
    int before_p = 0, before_r = 0;
    for (int i = 0; i < dk / 32; ++i) {
        const unsigned m = prot_words[i];
        const unsigned below = (1u << lane) - 1u;
        const int u = 32 * i + lane;
        const bool p = (m >> lane) & 1u;
        const int pos = p ? before_p + __popc(m & below) : n_prot + before_r + __popc(~m & below);
        perm_out[(int64_t)h * dk + pos] = (uint8_t)u;
        before_p += __popc(m);
        before_r += 32 - __popc(m);
    }
}

}  // namespace

cudaError_t launch_calib_error_energy(const float *S, int32_t batch, int32_t H, int32_t Hm, const int32_t *head_map,
                                      int32_t dk, int32_t dv, int32_t fmt, float *E_acc, cudaStream_t stream) {
    const int64_t grid = (int64_t)H * ((dk + 31) / 32);
    void (*kern)(const float *, int32_t, int32_t, int32_t, const int32_t *, int32_t, int32_t, float *) = nullptr;
    switch (fmt) {
        case kFmtU8H32: kern = calib_error_energy_kernel<kFmtU8H32>; break;
        case kFmtU8: kern = calib_error_energy_kernel<kFmtU8>; break;
        case kFmtS8Row: kern = calib_error_energy_kernel<kFmtS8Row>; break;
        case kFmtU4H32: kern = calib_error_energy_kernel<kFmtU4H32>; break;
        case kFmtU4: kern = calib_error_energy_kernel<kFmtU4>; break;
        case kFmtE4M3: kern = calib_error_energy_kernel<kFmtE4M3>; break;
        default: return cudaErrorInvalidValue;
    }
    if (fmt != kFmtS8Row) {
        const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kEeSmem);
        if (e != cudaSuccess) return e;
    }
    kern<<<(unsigned)grid, 32 * kEeWarps, fmt == kFmtS8Row ? 0 : kEeSmem, stream>>>(S, batch, H, Hm, head_map, dk, dv, E_acc);
    return cudaGetLastError();
}

cudaError_t launch_calib_log_decay(const float *g, int32_t batch, int32_t H, int32_t Hm, const int32_t *head_map,
                                   int32_t dk, int32_t kda, float *G_acc, cudaStream_t stream) {
    const int64_t n = (int64_t)H * dk;
    calib_log_decay_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(g, batch, H, Hm, head_map, dk, kda,
                                                                              G_acc);
    return cudaGetLastError();
}

cudaError_t launch_calib_select(const float *E_acc, int64_t n_samples, const float *G_acc, int64_t n_tokens, float tau,
                                int32_t H, int32_t Hm, const int32_t *head_map, int32_t dk, int32_t k_hi,
                                float *C_out, uint8_t *perm_out, cudaStream_t stream) {
    calib_select_kernel<<<H, 32, 0, stream>>>(E_acc, 1.0f / (float)n_samples, G_acc, 1.0f / (float)n_tokens, tau, H,
                                               Hm, head_map, dk, k_hi, C_out, perm_out);
    return cudaGetLastError();
}

cudaError_t take_status_calib(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_calib, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_calib, &zero, sizeof(uint32_t));
}

}  // namespace damp
