// damp_abi.cu -- the extern "C" entry points of libdamp (include/damp.h):
// host-side argument checks, then one launch on the caller's stream.
#include <atomic>
#include <climits>

#include "damp.h"
#include "damp_common.cuh"
#include "damp_internal.h"

namespace damp {

namespace {

constexpr int kMaxDevices = 64;
std::atomic<int> g_sm_count[kMaxDevices];
std::atomic<int> g_smem_optin[kMaxDevices];
std::atomic<int> g_smem_sm[kMaxDevices];

int device_attr(std::atomic<int> *cache, cudaDeviceAttr attr, int fallback) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return fallback;
    int v = cache[dev].load(std::memory_order_relaxed);
    if (v > 0) return v;
    if (cudaDeviceGetAttribute(&v, attr, dev) != cudaSuccess || v <= 0) return fallback;
    cache[dev].store(v, std::memory_order_relaxed);
    return v;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

struct Range {
    uintptr_t lo, hi;  // [lo, hi)
};
Range range_of(const void *p, int64_t bytes) {
    const uintptr_t lo = reinterpret_cast<uintptr_t>(p);
    return Range{lo, lo + (uintptr_t)(bytes > 0 ? bytes : 0)};
}
bool overlap(Range a, Range b) { return a.lo < b.hi && b.lo < a.hi && a.hi > a.lo && b.hi > b.lo; }

// value heads of the operand tensors (H_m)
int64_t model_heads_of(const damp_layout *L) { return L->model_heads > 0 ? L->model_heads : L->num_heads; }

damp_status check_layout(const damp_layout *L) {
    if (!L) return DAMP_ERR_NULL;
    if (L->num_heads < 1 || L->num_qk_heads < 1 || L->model_heads < 0) return DAMP_ERR_SHAPE;
    const int64_t Hm = model_heads_of(L);
    if (Hm < L->num_heads || Hm % L->num_qk_heads) return DAMP_ERR_SHAPE;
    if (!L->head_map && Hm != L->num_heads) return DAMP_ERR_SHAPE;
    if (L->head_map && !aligned(L->head_map, 4)) return DAMP_ERR_ALIGN;
    if (Hm > (1 << 20)) return DAMP_ERR_SHAPE;
    if (L->d_k != 32 && L->d_k != 64 && L->d_k != 128) return DAMP_ERR_SHAPE;
    if (L->d_v < 32 || L->d_v > 1024 || L->d_v % 32) return DAMP_ERR_SHAPE;
    if (L->k_hi < 0 || L->k_hi > L->d_k) return DAMP_ERR_SHAPE;
    if (L->lo_format < DAMP_LO_U8_AFFINE_G32_H32 || L->lo_format > DAMP_LO_FP8_E4M3_G32) return DAMP_ERR_FORMAT;
    return DAMP_OK;
}

int64_t slot_bytes_of(const damp_layout *L) {
    return (int64_t)L->num_heads * (L->d_v / 32) * rec_geom(L->d_k, L->k_hi, L->lo_format).bytes;
}

// Slots, batch rows and the pool's byte range; shared by every call on a pool.
damp_status check_pool(const void *state, int64_t num_slots, const int32_t *slot_idx, int32_t batch,
                       int64_t slot_bytes, Range *pool) {
    if (batch < 0 || num_slots < 0) return DAMP_ERR_SHAPE;
    if (!state) return DAMP_ERR_NULL;
    if (!aligned(state, 16)) return DAMP_ERR_ALIGN;
    if (slot_idx && !aligned(slot_idx, 4)) return DAMP_ERR_ALIGN;
    if (!slot_idx && num_slots < batch) return DAMP_ERR_SHAPE;
    if (num_slots < 1) return DAMP_ERR_SHAPE;
    if (slot_bytes > 0 && num_slots > INT64_MAX / slot_bytes) return DAMP_ERR_SHAPE;
    *pool = range_of(state, num_slots * slot_bytes);
    return DAMP_OK;
}

cudaError_t launch_step(const StepArgs &a, bool packed, cudaStream_t s, bool waittest = false) {
    if (waittest) return launch_packed_kda_waittest(a, s);
    if (!packed) return launch_fp32_step(a, s);
    if (a.fmt == DAMP_LO_S8_ABSMAX_ROW) {
        if (a.dv > 4 * 32) return launch_rowabs_step(a, s);  // the two-sweep step for d_v > 128
        // d_k = d_v = 128: the full-row quad step (four warps share each row's maximum)
        const cudaError_t eq = a.kda ? launch_quad_rowabs_kda(a, s) : launch_quad_rowabs_gdn(a, s);
        if (eq != cudaErrorNotSupported) return eq;
        StepArgs one = a;  // otherwise a one-token chunk: four warps share each row's maximum
        one.T = 1;
        one.lengths = nullptr;
        return a.kda ? launch_prefill_kda(one, s) : launch_prefill_gdn(one, s);
    }
    if (a.fmt == DAMP_LO_U4_AFFINE_G32_H32 || a.fmt == DAMP_LO_U4_AFFINE_G32)
        return a.kda ? launch_packed_kda_u4(a, s) : launch_packed_gdn_u4(a, s);
    if (a.fmt == DAMP_LO_FP8_E4M3_G32) return a.kda ? launch_packed_kda_f8(a, s) : launch_packed_gdn_f8(a, s);
    return a.kda ? launch_packed_kda(a, s) : launch_packed_gdn(a, s);
}

damp_status step(const damp_layout *L, void *state, int64_t num_slots, const int32_t *slot_idx, int32_t batch,
                 const uint8_t *perm, const void *q, const void *k, const void *v, const float *g,
                 const float *beta, float *o, int32_t in_dtype, void *stream, bool kda, bool packed,
                 bool uniform, bool waittest = false, StepArgs *prepared = nullptr) {
    damp_status st = check_layout(L);
    if (st != DAMP_OK && packed) return st;
    if (!packed) {  // the FP32 state ignores k_hi and lo_format and holds every model head
        if (!L) return DAMP_ERR_NULL;
        damp_layout l2 = *L;
        l2.k_hi = 0;
        l2.lo_format = 0;
        if ((st = check_layout(&l2)) != DAMP_OK) return st;
        if (L->head_map) return DAMP_ERR_SHAPE;
    }
    if (uniform && L->k_hi != 0) return DAMP_ERR_SHAPE;
    if (in_dtype != DAMP_IN_BF16 && in_dtype != DAMP_IN_FP32) return DAMP_ERR_FORMAT;
    if (waittest && (L->d_k != 128 || L->d_v != 128 || L->k_hi != 10 || L->lo_format != DAMP_LO_U8_AFFINE_G32_H32 ||
                     in_dtype != DAMP_IN_BF16 || L->head_map))
        return DAMP_ERR_SHAPE;
    if (batch < 0) return DAMP_ERR_SHAPE;
    if (batch == 0) return DAMP_OK;
    const int64_t sb = packed ? slot_bytes_of(L) : (int64_t)L->num_heads * L->d_k * L->d_v * 4;
    Range pool;
    if ((st = check_pool(state, num_slots, slot_idx, batch, sb, &pool)) != DAMP_OK) return st;
    if ((packed && !perm) || !q || !k || !v || !g || !beta || !o) return DAMP_ERR_NULL;
    if ((packed && !aligned(perm, 16)) || !aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) ||
        !aligned(g, kda ? 16 : 4) || !aligned(beta, 4) || !aligned(o, 4))
        return DAMP_ERR_ALIGN;
    const int64_t B = batch, H = L->num_heads, Hm = model_heads_of(L), Hq = L->num_qk_heads, dk = L->d_k,
                  dv = L->d_v;
    const int64_t esz = in_dtype == DAMP_IN_BF16 ? 2 : 4;
    const Range ro = range_of(o, B * Hm * dv * 4);
    const Range inputs[] = {range_of(q, B * Hq * dk * esz), range_of(k, B * Hq * dk * esz),
                            range_of(v, B * Hm * dv * esz), range_of(g, B * Hm * (kda ? dk : 1) * 4),
                            range_of(beta, B * Hm * 4), range_of(perm, packed ? H * dk : 0),
                            range_of(slot_idx, slot_idx ? B * 4 : 0), range_of(L->head_map, L->head_map ? H * 4 : 0)};
    if (overlap(ro, pool)) return DAMP_ERR_ALIAS;
    for (const Range &r : inputs)
        if (overlap(ro, r) || overlap(pool, r)) return DAMP_ERR_ALIAS;

    StepArgs a{};
    a.H = L->num_heads;
    a.Hqk = L->num_qk_heads;
    a.Hm = (int32_t)Hm;
    a.head_map = L->head_map;
    a.dk = L->d_k;
    a.dv = L->d_v;
    a.K = packed ? L->k_hi : 0;
    a.fmt = packed ? L->lo_format : 0;
    a.state = state;
    a.num_slots = num_slots;
    a.slot_idx = slot_idx;
    a.batch = batch;
    a.perm = perm;
    a.q = q;
    a.k = k;
    a.v = v;
    a.g = g;
    a.beta = beta;
    a.o = o;
    a.in_bf16 = in_dtype == DAMP_IN_BF16;
    a.kda = kda;
    if (prepared) {  // checked, not launched (the head-group step launches)
        *prepared = a;
        return DAMP_OK;
    }
    return launch_step(a, packed, static_cast<cudaStream_t>(stream), waittest) == cudaSuccess ? DAMP_OK
                                                                                           : DAMP_ERR_CUDA;
}

// The head groups of one layer (App. E): each group checked as a one-group step, the
// groups against each other (same operand shapes and format, pools disjoint from each
// other); two groups with a compile-time pair of K_hi run in one launch, other groups
// one launch each.
damp_status step_groups(const damp_layout *layouts, int32_t n_groups, void *const *states, const int64_t *num_slots,
                        const uint8_t *const *perms, const int32_t *slot_idx, int32_t batch, const void *q,
                        const void *k, const void *v, const float *g, const float *beta, float *o, int32_t in_dtype,
                        void *stream, bool kda) {
    constexpr int kMaxGroups = 8;
    if (!layouts || !states || !num_slots || !perms) return DAMP_ERR_NULL;
    if (n_groups < 1 || n_groups > kMaxGroups) return DAMP_ERR_SHAPE;
    if (batch < 0) return DAMP_ERR_SHAPE;
    StepArgs a[kMaxGroups];
    Range pools[kMaxGroups];
    for (int i = 0; i < n_groups; ++i) {
        const damp_layout &L = layouts[i];
        damp_status st = check_layout(&L);
        if (st != DAMP_OK) return st;
        if (!L.head_map) return DAMP_ERR_SHAPE;  // a group is a head subset
        const damp_layout &L0 = layouts[0];
        if (L.model_heads != L0.model_heads || L.num_qk_heads != L0.num_qk_heads || L.d_k != L0.d_k ||
            L.d_v != L0.d_v)
            return DAMP_ERR_SHAPE;
        if (L.lo_format != L0.lo_format) return DAMP_ERR_FORMAT;
        if (batch == 0) continue;
        st = step(&L, states[i], num_slots[i], slot_idx, batch, perms[i], q, k, v, g, beta, o, in_dtype, stream, kda,
                  true, false, false, &a[i]);
        if (st != DAMP_OK) return st;
        pools[i] = range_of(states[i], num_slots[i] * slot_bytes_of(&L));
        for (int j = 0; j < i; ++j)
            if (overlap(pools[i], pools[j])) return DAMP_ERR_ALIAS;
    }
    if (batch == 0) return DAMP_OK;
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (n_groups == 2) {
        const cudaError_t e = kda ? launch_packed2_kda(a[0], a[1], s) : launch_packed2_gdn(a[0], a[1], s);
        if (e != cudaErrorNotSupported) return e == cudaSuccess ? DAMP_OK : DAMP_ERR_CUDA;
    }
    for (int i = 0; i < n_groups; ++i)
        if (launch_step(a[i], true, s) != cudaSuccess) return DAMP_ERR_CUDA;
    return DAMP_OK;
}

damp_status prefill(const damp_layout *L, void *state, int64_t num_slots, const int32_t *slot_idx, int32_t batch,
                    int32_t chunk_len, const int32_t *lengths, const uint8_t *perm, const void *q, const void *k,
                    const void *v, const float *g, const float *beta, float *o, int32_t in_dtype, void *stream,
                    bool kda) {
    damp_status st = check_layout(L);
    if (st != DAMP_OK) return st;
    if (L->lo_format == DAMP_LO_S8_ABSMAX_ROW && L->d_v > 128) return DAMP_ERR_SHAPE;
    if (in_dtype != DAMP_IN_BF16 && in_dtype != DAMP_IN_FP32) return DAMP_ERR_FORMAT;
    if (batch < 0 || chunk_len < 0) return DAMP_ERR_SHAPE;
    if (batch == 0 || chunk_len == 0) return DAMP_OK;
    Range pool;
    if ((st = check_pool(state, num_slots, slot_idx, batch, slot_bytes_of(L), &pool)) != DAMP_OK) return st;
    if (!perm || !q || !k || !v || !g || !beta || !o) return DAMP_ERR_NULL;
    if (!aligned(perm, 16) || !aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(g, kda ? 16 : 4) ||
        !aligned(beta, 4) || !aligned(o, 4) || (lengths && !aligned(lengths, 4)))
        return DAMP_ERR_ALIGN;
    const int64_t B = batch, T = chunk_len, H = L->num_heads, Hm = model_heads_of(L), Hq = L->num_qk_heads,
                  dk = L->d_k, dv = L->d_v;
    const int64_t esz = in_dtype == DAMP_IN_BF16 ? 2 : 4;
    const Range ro = range_of(o, B * T * Hm * dv * 4);
    const Range inputs[] = {range_of(q, B * T * Hq * dk * esz), range_of(k, B * T * Hq * dk * esz),
                            range_of(v, B * T * Hm * dv * esz), range_of(g, B * T * Hm * (kda ? dk : 1) * 4),
                            range_of(beta, B * T * Hm * 4), range_of(perm, H * dk),
                            range_of(slot_idx, slot_idx ? B * 4 : 0), range_of(lengths, lengths ? B * 4 : 0),
                            range_of(L->head_map, L->head_map ? H * 4 : 0)};
    if (overlap(ro, pool)) return DAMP_ERR_ALIAS;
    for (const Range &r : inputs)
        if (overlap(ro, r) || overlap(pool, r)) return DAMP_ERR_ALIAS;

    StepArgs a{};
    a.H = L->num_heads;
    a.Hqk = L->num_qk_heads;
    a.Hm = (int32_t)Hm;
    a.head_map = L->head_map;
    a.dk = L->d_k;
    a.dv = L->d_v;
    a.K = L->k_hi;
    a.fmt = L->lo_format;
    a.state = state;
    a.num_slots = num_slots;
    a.slot_idx = slot_idx;
    a.batch = batch;
    a.perm = perm;
    a.q = q;
    a.k = k;
    a.v = v;
    a.g = g;
    a.beta = beta;
    a.o = o;
    a.in_bf16 = in_dtype == DAMP_IN_BF16;
    a.kda = kda;
    a.T = chunk_len;
    a.lengths = lengths;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    return (kda ? launch_prefill_kda(a, s) : launch_prefill_gdn(a, s)) == cudaSuccess ? DAMP_OK : DAMP_ERR_CUDA;
}

enum ConvKind { kQ, kDQ, kPack, kUnpack };

damp_status convert(const damp_layout *L, void *state, int64_t num_slots, const int32_t *slot_idx, int32_t batch,
                    const uint8_t *perm, float *S, uint16_t *hi, uint8_t *codes, uint16_t *meta, void *stream,
                    ConvKind kind) {
    damp_status st = check_layout(L);
    if (st != DAMP_OK) return st;
    if (batch < 0) return DAMP_ERR_SHAPE;
    if (batch == 0) return DAMP_OK;
    Range pool;
    if ((st = check_pool(state, num_slots, slot_idx, batch, slot_bytes_of(L), &pool)) != DAMP_OK) return st;
    const int64_t B = batch, H = L->num_heads, Hm = model_heads_of(L), dk = L->d_k, dv = L->d_v, K = L->k_hi;
    if (kind == kQ || kind == kDQ) {
        if (!perm || !S) return DAMP_ERR_NULL;
        if (!aligned(perm, 16) || !aligned(S, 16)) return DAMP_ERR_ALIGN;
        const Range rs = range_of(S, B * Hm * dk * dv * 4);
        if (overlap(rs, pool) || overlap(rs, range_of(perm, H * dk)) ||
            overlap(rs, range_of(slot_idx, slot_idx ? B * 4 : 0)) || overlap(pool, range_of(perm, H * dk)))
            return DAMP_ERR_ALIAS;
    } else {
        const int64_t nh = B * H * K * dv * 2, nc = B * H * (dk - K) * dv * fmt_code_bits(L->lo_format) / 8;
        const int64_t nm = B * H * (dk - K) * (L->lo_format == DAMP_LO_S8_ABSMAX_ROW ? 1 : dv / 32) * 4;
        if ((nh && !hi) || (nc && !codes) || (nm && !meta)) return DAMP_ERR_NULL;
        if ((hi && !aligned(hi, 4)) || (codes && !aligned(codes, 4)) || (meta && !aligned(meta, 4)))
            return DAMP_ERR_ALIGN;
        const Range t[] = {range_of(hi, nh), range_of(codes, nc), range_of(meta, nm)};
        for (const Range &r : t) {
            if (overlap(r, pool) || overlap(r, range_of(slot_idx, slot_idx ? B * 4 : 0))) return DAMP_ERR_ALIAS;
        }
        if (overlap(t[0], t[1]) || overlap(t[0], t[2]) || overlap(t[1], t[2])) return DAMP_ERR_ALIAS;
    }
    ConvArgs a{};
    a.H = L->num_heads;
    a.Hm = (int32_t)Hm;
    a.head_map = kind == kQ || kind == kDQ ? L->head_map : nullptr;  // tiers are pool-indexed
    a.dk = L->d_k;
    a.dv = L->d_v;
    a.K = L->k_hi;
    a.fmt = L->lo_format;
    a.state = state;
    a.num_slots = num_slots;
    a.slot_idx = slot_idx;
    a.batch = batch;
    a.perm = perm;
    a.S = S;
    a.hi = hi;
    a.codes = codes;
    a.meta = meta;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (a.fmt == DAMP_LO_S8_ABSMAX_ROW)
        return launch_rowabs_convert(a, (int)kind, s) == cudaSuccess ? DAMP_OK : DAMP_ERR_CUDA;
    cudaError_t e = kind == kQ ? launch_quantize(a, s)
                    : kind == kDQ ? launch_dequantize(a, s)
                    : kind == kPack ? launch_pack_tiers(a, s)
                                    : launch_unpack_tiers(a, s);
    return e == cudaSuccess ? DAMP_OK : DAMP_ERR_CUDA;
}

}  // namespace

int sm_count() { return device_attr(g_sm_count, cudaDevAttrMultiProcessorCount, 1); }

namespace {
struct SmemEntry {
    std::atomic<const void *> kernel{nullptr};
    std::atomic<int> bytes{0};
};
constexpr int kSmemEntries = 256;
SmemEntry g_smem_set[kMaxDevices][kSmemEntries];
}  // namespace

cudaError_t ensure_smem_limit(const void *kernel, int bytes) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    SmemEntry *slot = nullptr;
    if (dev >= 0 && dev < kMaxDevices) {
        const size_t h = (reinterpret_cast<uintptr_t>(kernel) >> 4) % kSmemEntries;
        for (size_t i = 0; i < kSmemEntries; ++i) {
            SmemEntry &en = g_smem_set[dev][(h + i) % kSmemEntries];
            const void *k = en.kernel.load(std::memory_order_acquire);
            if (k == kernel) {
                if (en.bytes.load(std::memory_order_acquire) >= bytes) return cudaSuccess;
                slot = &en;
                break;
            }
            if (k == nullptr) {
                const void *expected = nullptr;
                if (en.kernel.compare_exchange_strong(expected, kernel) || expected == kernel) {
                    slot = &en;
                    break;
                }
            }
        }
    }
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && slot) {
        int cur = slot->bytes.load(std::memory_order_relaxed);
        while (cur < bytes && !slot->bytes.compare_exchange_weak(cur, bytes)) {
        }
    }
    return e;
}

cudaError_t symbol_address_cached(const void *symbol, std::atomic<uint32_t *> *cache, uint32_t **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < kMaxDevices) {
        uint32_t *known = cache[dev].load(std::memory_order_acquire);
        if (known) {
            *out = known;
            return cudaSuccess;
        }
    }
    e = cudaGetSymbolAddress(reinterpret_cast<void **>(out), symbol);
    if (e == cudaSuccess && dev >= 0 && dev < kMaxDevices) cache[dev].store(*out, std::memory_order_release);
    return e;
}
int max_smem_per_block() { return device_attr(g_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, 48 * 1024); }
int max_smem_per_sm() { return device_attr(g_smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, 0); }

}  // namespace damp

using namespace damp;

extern "C" {

damp_status damp_validate_layout(const damp_layout *layout) { return check_layout(layout); }

size_t damp_record_bytes(const damp_layout *layout) {
    if (check_layout(layout) != DAMP_OK) return 0;
    return (size_t)rec_geom(layout->d_k, layout->k_hi, layout->lo_format).bytes;
}

size_t damp_slot_bytes(const damp_layout *layout) {
    if (check_layout(layout) != DAMP_OK) return 0;
    return (size_t)slot_bytes_of(layout);
}

double damp_bits_per_value(const damp_layout *L) {
    if (check_layout(L) != DAMP_OK) return -1.0;
    const double hi = 16.0 * L->k_hi * L->d_v;
    const double lo = L->lo_format == DAMP_LO_S8_ABSMAX_ROW
                          ? (8.0 * L->d_v + 32.0) * (double)(L->d_k - L->k_hi)  // int8 + one FP32 scale
                          : (fmt_code_bits(L->lo_format) + 32.0 / 32.0) * (double)(L->d_k - L->k_hi) *
                                L->d_v;  // codes + 32 bits of metadata per 32 values
    return (hi + lo) / ((double)L->d_k * L->d_v);
}

damp_status damp_gdn_decode_step(const damp_layout *layout, void *state, int64_t num_slots, const int32_t *slot_idx,
                                 int32_t batch, const uint8_t *perm, const void *q, const void *k, const void *v,
                                 const float *g, const float *beta, float *o, int32_t in_dtype, void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, perm, q, k, v, g, beta, o, in_dtype, stream, false, true,
                false);
}

damp_status damp_kda_decode_step(const damp_layout *layout, void *state, int64_t num_slots, const int32_t *slot_idx,
                                 int32_t batch, const uint8_t *perm, const void *q, const void *k, const void *v,
                                 const float *g, const float *beta, float *o, int32_t in_dtype, void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, perm, q, k, v, g, beta, o, in_dtype, stream, true, true,
                false);
}

damp_status damp_gdn_decode_step_groups(const damp_layout *layouts, int32_t n_groups, void *const *states,
                                        const int64_t *num_slots, const uint8_t *const *perms,
                                        const int32_t *slot_idx, int32_t batch, const void *q, const void *k,
                                        const void *v, const float *g, const float *beta, float *o,
                                        int32_t in_dtype, void *stream) {
    return step_groups(layouts, n_groups, states, num_slots, perms, slot_idx, batch, q, k, v, g, beta, o, in_dtype,
                       stream, false);
}

damp_status damp_kda_decode_step_groups(const damp_layout *layouts, int32_t n_groups, void *const *states,
                                        const int64_t *num_slots, const uint8_t *const *perms,
                                        const int32_t *slot_idx, int32_t batch, const void *q, const void *k,
                                        const void *v, const float *g, const float *beta, float *o,
                                        int32_t in_dtype, void *stream) {
    return step_groups(layouts, n_groups, states, num_slots, perms, slot_idx, batch, q, k, v, g, beta, o, in_dtype,
                       stream, true);
}

damp_status damp_test_kda_wait_timeout(const damp_layout *layout, void *state, int64_t num_slots,
                                       const int32_t *slot_idx, int32_t batch, const uint8_t *perm, const void *q,
                                       const void *k, const void *v, const float *g, const float *beta, float *o,
                                       int32_t in_dtype, void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, perm, q, k, v, g, beta, o, in_dtype, stream, true, true,
                false, true);
}

damp_status damp_u8_gdn_decode_step(const damp_layout *layout, void *state, int64_t num_slots,
                                    const int32_t *slot_idx, int32_t batch, const uint8_t *perm, const void *q,
                                    const void *k, const void *v, const float *g, const float *beta, float *o,
                                    int32_t in_dtype, void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, perm, q, k, v, g, beta, o, in_dtype, stream, false, true,
                true);
}

damp_status damp_u8_kda_decode_step(const damp_layout *layout, void *state, int64_t num_slots,
                                    const int32_t *slot_idx, int32_t batch, const uint8_t *perm, const void *q,
                                    const void *k, const void *v, const float *g, const float *beta, float *o,
                                    int32_t in_dtype, void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, perm, q, k, v, g, beta, o, in_dtype, stream, true, true,
                true);
}

damp_status damp_fp32_gdn_decode_step(const damp_layout *layout, float *state, int64_t num_slots,
                                      const int32_t *slot_idx, int32_t batch, const void *q, const void *k,
                                      const void *v, const float *g, const float *beta, float *o, int32_t in_dtype,
                                      void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, nullptr, q, k, v, g, beta, o, in_dtype, stream, false,
                false, false);
}

damp_status damp_fp32_kda_decode_step(const damp_layout *layout, float *state, int64_t num_slots,
                                      const int32_t *slot_idx, int32_t batch, const void *q, const void *k,
                                      const void *v, const float *g, const float *beta, float *o, int32_t in_dtype,
                                      void *stream) {
    return step(layout, state, num_slots, slot_idx, batch, nullptr, q, k, v, g, beta, o, in_dtype, stream, true,
                false, false);
}

damp_status damp_gdn_prefill_chunk(const damp_layout *layout, void *state, int64_t num_slots, const int32_t *slot_idx,
                                   int32_t batch, int32_t chunk_len, const int32_t *lengths, const uint8_t *perm,
                                   const void *q, const void *k, const void *v, const float *g, const float *beta,
                                   float *o, int32_t in_dtype, void *stream) {
    return prefill(layout, state, num_slots, slot_idx, batch, chunk_len, lengths, perm, q, k, v, g, beta, o, in_dtype,
                   stream, false);
}

damp_status damp_kda_prefill_chunk(const damp_layout *layout, void *state, int64_t num_slots, const int32_t *slot_idx,
                                   int32_t batch, int32_t chunk_len, const int32_t *lengths, const uint8_t *perm,
                                   const void *q, const void *k, const void *v, const float *g, const float *beta,
                                   float *o, int32_t in_dtype, void *stream) {
    return prefill(layout, state, num_slots, slot_idx, batch, chunk_len, lengths, perm, q, k, v, g, beta, o, in_dtype,
                   stream, true);
}

damp_status damp_quantize_state(const damp_layout *layout, const float *S, const uint8_t *perm, void *state,
                                int64_t num_slots, const int32_t *slot_idx, int32_t batch, void *stream) {
    return convert(layout, state, num_slots, slot_idx, batch, perm, const_cast<float *>(S), nullptr, nullptr,
                   nullptr, stream, kQ);
}

damp_status damp_dequantize_state(const damp_layout *layout, const void *state, int64_t num_slots,
                                  const int32_t *slot_idx, int32_t batch, const uint8_t *perm, float *S,
                                  void *stream) {
    return convert(layout, const_cast<void *>(state), num_slots, slot_idx, batch, perm, S, nullptr, nullptr, nullptr,
                   stream, kDQ);
}

damp_status damp_pack_tiers(const damp_layout *layout, const uint16_t *hi, const uint8_t *codes, const uint16_t *meta,
                            void *state, int64_t num_slots, const int32_t *slot_idx, int32_t batch, void *stream) {
    return convert(layout, state, num_slots, slot_idx, batch, nullptr, nullptr, const_cast<uint16_t *>(hi),
                   const_cast<uint8_t *>(codes), const_cast<uint16_t *>(meta), stream, kPack);
}

damp_status damp_unpack_tiers(const damp_layout *layout, const void *state, int64_t num_slots,
                              const int32_t *slot_idx, int32_t batch, uint16_t *hi, uint8_t *codes, uint16_t *meta,
                              void *stream) {
    return convert(layout, const_cast<void *>(state), num_slots, slot_idx, batch, nullptr, nullptr, hi, codes, meta,
                   stream, kUnpack);
}

damp_status damp_calib_error_energy(const damp_layout *layout, const float *S, int32_t batch, float *E_acc,
                                    void *stream) {
    damp_status st = check_layout(layout);
    if (st != DAMP_OK) return st;
    if (batch < 0) return DAMP_ERR_SHAPE;
    if (!E_acc) return DAMP_ERR_NULL;
    if (batch == 0) return DAMP_OK;
    if (!S) return DAMP_ERR_NULL;
    if (!aligned(S, 16) || !aligned(E_acc, 4)) return DAMP_ERR_ALIGN;
    const int64_t H = layout->num_heads, Hm = model_heads_of(layout), dk = layout->d_k, dv = layout->d_v;
    if (overlap(range_of(S, (int64_t)batch * Hm * dk * dv * 4), range_of(E_acc, Hm * dk * 4))) return DAMP_ERR_ALIAS;
    return launch_calib_error_energy(S, batch, (int32_t)H, (int32_t)Hm, layout->head_map, (int32_t)dk, (int32_t)dv,
                                     layout->lo_format, E_acc, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAMP_OK
               : DAMP_ERR_CUDA;
}

damp_status damp_calib_log_decay(const damp_layout *layout, const float *g, int32_t batch, int32_t kda, float *G_acc,
                                 void *stream) {
    damp_status st = check_layout(layout);
    if (st != DAMP_OK) return st;
    if (batch < 0) return DAMP_ERR_SHAPE;
    if (!G_acc) return DAMP_ERR_NULL;
    if (batch == 0) return DAMP_OK;
    if (!g) return DAMP_ERR_NULL;
    if (!aligned(g, 4) || !aligned(G_acc, 4)) return DAMP_ERR_ALIGN;
    const int64_t H = layout->num_heads, Hm = model_heads_of(layout), dk = layout->d_k;
    if (overlap(range_of(g, (int64_t)batch * Hm * (kda ? dk : 1) * 4), range_of(G_acc, Hm * dk * 4)))
        return DAMP_ERR_ALIAS;
    return launch_calib_log_decay(g, batch, (int32_t)H, (int32_t)Hm, layout->head_map, (int32_t)dk, kda ? 1 : 0,
                                  G_acc, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAMP_OK
               : DAMP_ERR_CUDA;
}

damp_status damp_calib_accumulate(const damp_layout *layout, float *S, int32_t n_docs, int32_t n_tokens,
                                  const void *q, const void *k, const void *v, const float *g, const float *beta,
                                  int32_t in_dtype, int32_t kda, int32_t every, float *E_acc, float *G_acc,
                                  void *stream) {
    damp_status st = check_layout(layout);
    if (st != DAMP_OK) return st;
    if (layout->head_map) return DAMP_ERR_SHAPE;  // the trajectories hold every head of the layer
    if (in_dtype != DAMP_IN_BF16 && in_dtype != DAMP_IN_FP32) return DAMP_ERR_FORMAT;
    if (n_docs < 0 || n_tokens < 0 || every < 1) return DAMP_ERR_SHAPE;
    if (!E_acc || !G_acc) return DAMP_ERR_NULL;
    if (n_docs == 0 || n_tokens == 0) return DAMP_OK;
    if (!S || !q || !k || !v || !g || !beta) return DAMP_ERR_NULL;
    if (!aligned(S, 16) || !aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(g, kda ? 16 : 4) ||
        !aligned(beta, 4) || !aligned(E_acc, 4) || !aligned(G_acc, 4))
        return DAMP_ERR_ALIGN;
    const int64_t B = n_docs, T = n_tokens, H = layout->num_heads, Hq = layout->num_qk_heads, dk = layout->d_k,
                  dv = layout->d_v;
    if (B * T > INT32_MAX) return DAMP_ERR_SHAPE;  // the log-decay call takes the (token, document) rows
    const int64_t esz = in_dtype == DAMP_IN_BF16 ? 2 : 4;
    const int64_t sq = B * Hq * dk * esz, sv = B * H * dv * esz, sg = B * H * (kda ? dk : 1) * 4, sb = B * H * 4;
    const Range rs = range_of(S, B * H * dk * dv * 4), re = range_of(E_acc, H * dk * 4), rg = range_of(G_acc, H * dk * 4);
    const Range inputs[] = {range_of(q, T * sq), range_of(k, T * sq), range_of(v, T * sv), range_of(g, T * sg),
                            range_of(beta, T * sb)};
    if (overlap(rs, re) || overlap(rs, rg) || overlap(re, rg)) return DAMP_ERR_ALIAS;
    for (const Range &r : inputs)
        if (overlap(rs, r) || overlap(re, r) || overlap(rg, r)) return DAMP_ERR_ALIAS;
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    StepArgs a{};
    a.H = (int32_t)H;
    a.Hqk = (int32_t)Hq;
    a.Hm = (int32_t)H;
    a.dk = (int32_t)dk;
    a.dv = (int32_t)dv;
    a.state = S;
    a.num_slots = B;
    a.batch = n_docs;
    a.o = nullptr;  // the trajectories' outputs are not needed
    a.in_bf16 = in_dtype == DAMP_IN_BF16;
    a.kda = kda ? 1 : 0;
    for (int64_t t = 0; t < T; ++t) {
        a.q = static_cast<const uint8_t *>(q) + t * sq;
        a.k = static_cast<const uint8_t *>(k) + t * sq;
        a.v = static_cast<const uint8_t *>(v) + t * sv;
        a.g = reinterpret_cast<const float *>(reinterpret_cast<const uint8_t *>(g) + t * sg);
        a.beta = reinterpret_cast<const float *>(reinterpret_cast<const uint8_t *>(beta) + t * sb);
        if (launch_fp32_step(a, s) != cudaSuccess) return DAMP_ERR_CUDA;
        if ((t + 1) % every == 0 &&
            launch_calib_error_energy(S, n_docs, (int32_t)H, (int32_t)H, nullptr, (int32_t)dk, (int32_t)dv,
                                      layout->lo_format, E_acc, s) != cudaSuccess)
            return DAMP_ERR_CUDA;
    }
    // the log-decay sums of every (token, document) row: the stacked gates as one batch
    return launch_calib_log_decay(g, (int32_t)(B * T), (int32_t)H, (int32_t)H, nullptr, (int32_t)dk, kda ? 1 : 0,
                                  G_acc, s) == cudaSuccess
               ? DAMP_OK
               : DAMP_ERR_CUDA;
}

damp_status damp_calib_select(const damp_layout *layout, const float *E_acc, int64_t n_samples, const float *G_acc,
                              int64_t n_tokens, float tau, float *C_out, uint8_t *perm_out, void *stream) {
    damp_status st = check_layout(layout);
    if (st != DAMP_OK) return st;
    if (!E_acc || !G_acc || !C_out || !perm_out) return DAMP_ERR_NULL;
    if (n_samples < 1 || n_tokens < 1 || !(tau > 0.0f) || !(tau <= 1.0f)) return DAMP_ERR_SHAPE;
    if (!aligned(E_acc, 4) || !aligned(G_acc, 4) || !aligned(C_out, 4)) return DAMP_ERR_ALIGN;
    const int64_t H = layout->num_heads, Hm = model_heads_of(layout), dk = layout->d_k;
    const Range rc = range_of(C_out, H * dk * 4), rp = range_of(perm_out, H * dk);
    const Range ins[] = {range_of(E_acc, Hm * dk * 4), range_of(G_acc, Hm * dk * 4)};
    if (overlap(rc, rp)) return DAMP_ERR_ALIAS;
    for (const Range &r : ins)
        if (overlap(r, rc) || overlap(r, rp)) return DAMP_ERR_ALIAS;
    return launch_calib_select(E_acc, n_samples, G_acc, n_tokens, tau, (int32_t)H, (int32_t)Hm, layout->head_map,
                               (int32_t)dk, layout->k_hi, C_out, perm_out,
                               static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAMP_OK
               : DAMP_ERR_CUDA;
}

damp_status damp_device_status(uint32_t *status) {
    if (!status) return DAMP_ERR_NULL;
    // Kernels on non-blocking streams do not order with the copies below: wait for
    // all of them first, so a bit set by a kernel in flight is not cleared unread.
    if (cudaDeviceSynchronize() != cudaSuccess) return DAMP_ERR_CUDA;
    uint32_t all = 0, bits = 0;
    if (take_status_packed_gdn(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_packed_kda(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_packed_gdn_u4(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_packed_kda_u4(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_packed_gdn_f8(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_packed_kda_f8(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_groups_gdn(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_groups_kda(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_quad_gdn(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_quad_kda(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_fp32(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_convert(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_rowabs(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_prefill_gdn(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_prefill_kda(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_prefill_gdn_x(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_prefill_kda_x(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    if (take_status_calib(&bits) != cudaSuccess) return DAMP_ERR_CUDA;
    all |= bits;
    *status = all;
    return DAMP_OK;
}

const char *damp_status_string(damp_status s) {
    switch (s) {
        case DAMP_OK: return "DAMP_OK";
        case DAMP_ERR_NULL: return "DAMP_ERR_NULL: a required pointer is NULL";
        case DAMP_ERR_SHAPE: return "DAMP_ERR_SHAPE: a size is outside what the kernels support";
        case DAMP_ERR_ALIGN: return "DAMP_ERR_ALIGN: a pointer is not aligned as documented";
        case DAMP_ERR_ALIAS: return "DAMP_ERR_ALIAS: an output overlaps the state pool or another argument";
        case DAMP_ERR_FORMAT: return "DAMP_ERR_FORMAT: unknown or unsupported lo_format / in_dtype";
        case DAMP_ERR_CUDA: return "DAMP_ERR_CUDA: the CUDA runtime reported an error while enqueueing";
    }
    return "unknown damp_status";
}

int32_t damp_version(void) { return 100; }

}  // extern "C"
