// decode_fp32.cu -- in-house FP32-state decode step (the deployment baseline of
// Sec. 6.1: FP32 recurrent-state storage), GDN and KDA.
//
// Same tile as the packed kernel -- (slot, head, value block c): d_k rows x 32
// columns -- but with no quantization group the thread mapping is the simple
// one: lane j owns column j of the tile for all d_k rows, so both column
// reductions r = S_bar^T k and o = S^T q are thread-local and every warp-wide
// load or store of a row is one coalesced 128-byte line.  Per-channel operands
// (k, q, decay, beta*k) are staged once per (slot, head) in shared memory and
// read as broadcasts.  A persistent grid: every warp walks a contiguous range of
// tiles, keeping d_k independent loads in flight.
#include "damp_common.cuh"
#include "damp_internal.h"

#include <algorithm>

namespace damp {

static __device__ uint32_t g_status_fp32;

struct Fp32Params {
    float *state;
    int64_t num_slots;
    const int32_t *slot_idx;
    const void *q, *k, *v;
    const float *g, *beta;
    float *o;
    int32_t batch, H, Hqk, dk, dv, V;
    int64_t total_tiles;
    uint32_t *status;
};

constexpr int kFp32Warps = 8;

template <int DK, int DV, bool KDA, bool BF16>
__global__ void __launch_bounds__(256, 1) fp32_step_kernel(const Fp32Params p) {
    __shared__ __align__(16) float ops[kFp32Warps][4][DK];  // k, q, a, beta*k per channel
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    float *sk = ops[warp][0];
    float *sq = ops[warp][1];
    float *sa = ops[warp][2];
    float *sb = ops[warp][3];

    const int64_t gw = (int64_t)blockIdx.x * nw + warp;
    const int64_t nwt = (int64_t)gridDim.x * nw;
    const int64_t t0 = p.total_tiles * gw / nwt;
    const int64_t t1 = p.total_tiles * (gw + 1) / nwt;
    bool bad_slot = false;

    for (int64_t t = t0; t < t1; ++t) {
        const int c = (int)(t % p.V);
        const int64_t bh = t / p.V;
        const int h = (int)(bh % p.H);
        const int b = (int)(bh / p.H);
        if (t == t0 || c == 0) {
            __syncwarp();
            const int hq = (h * p.Hqk) / p.H;
            const int64_t qoff = ((int64_t)b * p.Hqk + hq) * DK;
            const float beta = p.beta[(int64_t)b * p.H + h];
            const float alpha = KDA ? 0.f : expf(p.g[(int64_t)b * p.H + h]);
#pragma unroll
            for (int u = lane; u < DK; u += 32) {
                const float kv = load_in(p.k, qoff + u, BF16);
                sk[u] = kv;
                sq[u] = load_in(p.q, qoff + u, BF16);
                sa[u] = KDA ? expf(p.g[((int64_t)b * p.H + h) * DK + u]) : alpha;
                sb[u] = beta * kv;
            }
            __syncwarp();
        }
        const int64_t slot = p.slot_idx ? (int64_t)p.slot_idx[b] : (int64_t)b;
        if (slot < 0 || slot >= p.num_slots) {
            bad_slot = true;
            continue;
        }
        float *base = p.state + ((slot * p.H + h) * DK) * (int64_t)p.dv + c * kG + lane;
        // a compile-time row stride (DV > 0) turns every row address into an
        // immediate offset from one base register
        const int64_t ld = DV > 0 ? DV : p.dv;
        float x[DK];
#pragma unroll
        for (int u = 0; u < DK; ++u) x[u] = __ldcs(base + u * ld);
        const float vj = load_in(p.v, ((int64_t)b * p.H + h) * p.dv + c * kG + lane, BF16);

        // S_bar = Lambda S ; r = S_bar^T k
        float r0 = 0.f, r1 = 0.f, r2 = 0.f, r3 = 0.f;
#pragma unroll
        for (int u = 0; u < DK; u += 4) {
            const float4 a4 = *reinterpret_cast<const float4 *>(sa + u);
            const float4 k4 = *reinterpret_cast<const float4 *>(sk + u);
            x[u] *= a4.x;
            x[u + 1] *= a4.y;
            x[u + 2] *= a4.z;
            x[u + 3] *= a4.w;
            r0 = fmaf(x[u], k4.x, r0);
            r1 = fmaf(x[u + 1], k4.y, r1);
            r2 = fmaf(x[u + 2], k4.z, r2);
            r3 = fmaf(x[u + 3], k4.w, r3);
        }
        const float d = vj - ((r0 + r1) + (r2 + r3));
        // S = S_bar + beta k d^T ; o = S^T q
        float o0 = 0.f, o1 = 0.f, o2 = 0.f, o3 = 0.f;
#pragma unroll
        for (int u = 0; u < DK; u += 4) {
            const float4 b4 = *reinterpret_cast<const float4 *>(sb + u);
            const float4 q4 = *reinterpret_cast<const float4 *>(sq + u);
            x[u] = fmaf(b4.x, d, x[u]);
            x[u + 1] = fmaf(b4.y, d, x[u + 1]);
            x[u + 2] = fmaf(b4.z, d, x[u + 2]);
            x[u + 3] = fmaf(b4.w, d, x[u + 3]);
            o0 = fmaf(x[u], q4.x, o0);
            o1 = fmaf(x[u + 1], q4.y, o1);
            o2 = fmaf(x[u + 2], q4.z, o2);
            o3 = fmaf(x[u + 3], q4.w, o3);
        }
        // a fresh copy of the row pointer keeps the compiler from holding all
        // d_k load addresses live until the stores
#pragma unroll
        for (int u = 0; u < DK; ++u) __stcs(base + u * ld, x[u]);
        if (p.o) p.o[((int64_t)b * p.H + h) * p.dv + c * kG + lane] = (o0 + o1) + (o2 + o3);  // no o: calibration runs
    }
    if (bad_slot && lane == 0) atomicOr(p.status, (uint32_t)kDevBadSlot);
}

cudaError_t launch_fp32_step(const StepArgs &a, cudaStream_t stream) {
    Fp32Params p{};
    static std::atomic<uint32_t *> cache[64];
    cudaError_t e = symbol_address_cached(&g_status_fp32, cache, &p.status);
    if (e != cudaSuccess) return e;
    p.state = static_cast<float *>(a.state);
    p.num_slots = a.num_slots;
    p.slot_idx = a.slot_idx;
    p.q = a.q;
    p.k = a.k;
    p.v = a.v;
    p.g = a.g;
    p.beta = a.beta;
    p.o = a.o;
    p.batch = a.batch;
    p.H = a.H;
    p.Hqk = a.Hqk;
    p.dk = a.dk;
    p.dv = a.dv;
    p.V = a.dv / kG;
    p.total_tiles = (int64_t)a.batch * a.H * p.V;
    if (p.total_tiles == 0) return cudaSuccess;
    const int64_t want = (p.total_tiles + kFp32Warps - 1) / kFp32Warps;
    const int grid = (int)std::min<int64_t>(want, (int64_t)sm_count());
    void (*kern)(Fp32Params) = nullptr;
#define DAMP_PICK4(DK_, DV_)                                                                   \
    if (a.kda) kern = a.in_bf16 ? fp32_step_kernel<DK_, DV_, true, true> : fp32_step_kernel<DK_, DV_, true, false>; \
    else kern = a.in_bf16 ? fp32_step_kernel<DK_, DV_, false, true> : fp32_step_kernel<DK_, DV_, false, false>;
#define DAMP_PICK(DK_)                                                                         \
    if (a.dk == DK_) {                                                                         \
        if (a.dv == 64) { DAMP_PICK4(DK_, 64) }                                                \
        else if (a.dv == 128) { DAMP_PICK4(DK_, 128) }                                         \
        else { DAMP_PICK4(DK_, 0) }                                                            \
    }
    DAMP_PICK(32)
    DAMP_PICK(64)
    DAMP_PICK(128)
#undef DAMP_PICK
#undef DAMP_PICK4
    if (!kern) return cudaErrorInvalidValue;
    kern<<<grid, 32 * kFp32Warps, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t take_status_fp32(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_status_fp32, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_fp32, &zero, sizeof(uint32_t));
}

}  // namespace damp
