/*
 * damp.h -- C ABI of libdamp: the decode-time recurrent-state update of Gated
 * DeltaNet (GDN) and Kimi Delta Attention (KDA) over a DAMP mixed-precision
 * packed state, on one NVIDIA GB300 GPU (sm_103a).
 *
 * Method: "DAMP: Decay-Aware Mixed-Precision Recurrent-State Quantization"
 * (arxiv 2608.27513).  One decode step of one linear-attention layer, for every
 * request slot of a decode batch and every value head h, computes (Sec. 3.1):
 *
 *     S_bar = Lambda_t S_{t-1}                decay (GDN: alpha_t I; KDA: diag(exp(g_t)))
 *     delta = v_t - S_bar^T k_t               delta-rule read
 *     S_t   = S_bar + beta_t k_t delta^T      Eq. delta_update
 *     o_t   = S_t^T q_t                       output read (scale 1, FP32 post-update state)
 *
 * in FP32, on a state stored as (Sec. 5.2; App. A.5, Eq. packed_state_layout):
 *
 *     S_hi  FP16  [K_hi][d_v]                  the K_hi protected key channels
 *     Q_lo  UINT8 [d_k-K_hi][d_v]              the other channels, block-32 Hadamard
 *                                              transformed, asymmetric affine codes
 *     M_lo  FP16  [d_k-K_hi][d_v/32][2]        per 32-group scale s and zero point z
 *
 * with the key channels in the calibrated order pi_{l,h} (protected first), and
 * requantizes once per step (Sec. 3.3, Eq. quantized_recurrence):
 *     s = (x_max - x_min)/255 -> FP16,  z = round(-x_min/s) -> FP16,
 *     q_i = sat_[0,255](round(x_i/s) + z),  Q(x_i) = s (q_i - z)   (Eq. integer_quantizer).
 * round() is round-half-to-even; s and z are rounded to FP16 first and the codes
 * are encoded with the stored values; a block whose s rounds to 0 widens its
 * range to contain 0 (and uses s = 1, z = 0 if s is still 0).
 *
 * Conventions for every call:
 *   - Every array pointer is a CUDA device pointer owned by the caller.  libdamp
 *     never allocates or frees, and never synchronizes except in
 *     damp_device_status (below).  Work is enqueued on `stream`
 *     (a cudaStream_t passed as void*; NULL means the legacy default stream)
 *     and is ordered with the caller's other work on that stream.
 *   - Every argument check runs on the host before anything is enqueued.  A
 *     failed check returns a DAMP_ERR_* status and enqueues nothing.  A launch
 *     failure returns DAMP_ERR_CUDA.
 *   - A kernel never traps.  A slot index outside [0, num_slots) makes the kernel
 *     skip that batch row (its state and outputs are left untouched) and sets
 *     DAMP_DEV_BAD_SLOT in the device status word; a bounded wait inside a kernel
 *     that runs out sets DAMP_DEV_WAIT_TIMEOUT.  damp_device_status() reads and
 *     clears the word.
 *   - Operands are in natural key-channel order; the kernels apply pi.  Inputs
 *     q, k (and v) are read-only; the state is updated in place; o is written.
 *     Batch rows that name the same slot race: slot indices of one call must be
 *     distinct.
 *   - No C++ exception crosses the ABI.  The library keeps no per-call state;
 *     calls may come from several host threads.
 */
#ifndef DAMP_H
#define DAMP_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define DAMP_API __attribute__((visibility("default")))
#else
#define DAMP_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DAMP_OK = 0,
    DAMP_ERR_NULL = 1,    /* a required pointer is NULL */
    DAMP_ERR_SHAPE = 2,   /* a size is outside what the kernels support (see damp_layout) */
    DAMP_ERR_ALIGN = 3,   /* a pointer is not aligned as documented for its argument */
    DAMP_ERR_ALIAS = 4,   /* an output overlaps the state pool or another argument */
    DAMP_ERR_FORMAT = 5,  /* unknown lo_format or in_dtype, or one this call does not take */
    DAMP_ERR_CUDA = 6     /* the CUDA runtime reported an error while enqueueing */
} damp_status;

/* Low-precision tier formats (App. A.1, Tab. quantizer_specs). */
typedef enum {
    DAMP_LO_U8_AFFINE_G32_H32 = 0, /* UINT8 affine, G = 32 along d_v, FP16 (s, z), H_32 first:
                                      the paper's DAMP low tier ("INT8+Hadamard", 9.0 bits) */
    DAMP_LO_U8_AFFINE_G32 = 1,     /* the same without H_32 (the paper's "INT8" row, 9.0 bits) */
    DAMP_LO_S8_ABSMAX_ROW = 2,     /* per-row symmetric absmax INT8, one FP32 scale per row over
                                      all d_v values: s = max|x|/127, q = sat_[-127,127](rne(x/s)),
                                      s = 0 -> q = 0; no H_32 (8 + 32/d_v bits).  A fallback
                                      for a low tier whose scales are left open, not the paper's
                                      format.  Its row scale spans every value block of a head:
                                      for d_v <= 128 a step is a one-token chunk whose warps share
                                      each row's maximum; larger d_v sweep each head twice. */
    DAMP_LO_U4_AFFINE_G32_H32 = 3, /* UINT4 affine (b = 4), G = 32, FP16 (s, z), H_32 first (5.0 bits) */
    DAMP_LO_U4_AFFINE_G32 = 4,     /* the same without H_32 (the paper's "INT4" row, 5.0 bits) */
    DAMP_LO_FP8_E4M3_G32 = 5       /* FP8 E4M3, G = 32, one FP32 scale per group, natural domain:
                                      s = max(max|x|, 1e-10)/448, q = E4M3(clip(x/s, +-448)) (9.0 bits).
                                      Formats 3-5 are the paper's comparison tiers (App. A.1); their
                                      decode step is the same fused step as formats 0 and 1. */
} damp_lo_format;

/* Element type of q, k and v. */
typedef enum { DAMP_IN_BF16 = 0, DAMP_IN_FP32 = 1 } damp_in_dtype;

/* Device status bits (damp_device_status). */
#define DAMP_DEV_WAIT_TIMEOUT 1u
#define DAMP_DEV_BAD_SLOT 2u
#define DAMP_DEV_BAD_HEAD 4u

/*
 * Shape of one linear-attention layer's state (Sec. 3.1; Sec. 5.1 "Key-channel budget").
 *   num_heads     H      value heads held in the pool; one state per (slot, head)
 *   num_qk_heads  H_qk   q/k heads of the operand tensors
 *   d_k, d_v             state is d_k x d_v; d_k in {32, 64, 128}; d_v a multiple of 32, <= 1024
 *   k_hi          K_hi   FP16 key channels per head, 0 <= K_hi <= d_k (same for every head
 *                        of the pool)
 *   lo_format            damp_lo_format of the other d_k - K_hi channels
 *   model_heads   H_m    value heads of the operand and output tensors (v, g, beta, o, S,
 *                        calibration accumulators); 0 means H_m = H
 *   head_map             device int32 [H]: the model head (0 .. H_m-1) of each held head,
 *                        or NULL for the identity (then H_m must equal H)
 * Held head h is model head m = head_map[h] (or h); it reads q/k head floor(m*H_qk/H_m)
 * (GQA; H_m must be a multiple of H_qk), and its per-head operands and outputs are row m
 * of [*][H_m][...] tensors, while its permutation and packed records are row h of the pool.
 *
 * Head groups.  A layer whose heads protect different numbers of key channels (the
 * decay-tiered allocation of App. E: fast- and slow-decay heads with different K_hi)
 * is a set of layouts, one per K_hi, whose head maps partition 0 .. H_m-1; each group
 * has its own pool and permutation table, and one call per group -- or one
 * damp_*_decode_step_groups call for all groups -- updates the layer (the groups write
 * disjoint rows of o).  A head_map entry outside 0 .. H_m-1 sets
 * DAMP_DEV_BAD_HEAD in the device status word and that head is skipped.
 */
typedef struct {
    int32_t num_heads;
    int32_t num_qk_heads;
    int32_t d_k;
    int32_t d_v;
    int32_t k_hi;
    int32_t lo_format;
    int32_t model_heads;
    const int32_t *head_map;
} damp_layout;

/* Checks a layout; DAMP_OK or DAMP_ERR_NULL / DAMP_ERR_SHAPE / DAMP_ERR_FORMAT. Host only. */
DAMP_API damp_status damp_validate_layout(const damp_layout *layout);

/*
 * Physical packed state.  A pool holds num_slots slots; a slot holds H heads;
 * a head holds d_v/32 value-block records (the value-block-major organization of
 * App. A.5, which co-locates every 32-value code tile with its scale and zero
 * point).  Record (slot, h, c) starts at byte
 *     slot * damp_slot_bytes + (h * d_v/32 + c) * damp_record_bytes
 * and holds, for value columns 32c .. 32c+31 of all d_k packed rows:
 *     [ceil(K_hi/2) FP16 row pairs x 128 B][(d_k-K_hi) x 32 codes][(d_k-K_hi) x 4 B metadata]
 *     [padding to 16 B]
 * FP16 row pair i interleaves rows 2i and 2i+1 column by column; code rows are stored
 * chunk-major (16-byte chunk m of every row, then chunk m + 1), so that a warp's
 * 128-bit accesses to one chunk of 32 consecutive rows are contiguous.  The
 * metadata word of a row is its (s, z) FP16 pair (formats 0, 1, 3, 4), the FP32 group
 * scale (format 5) or its FP32 row scale (format 2, the same value in each of the
 * head's d_v/32 records).  4-bit formats store a code row in 16 bytes (value 2i in the
 * low nibble of byte i).  The byte order inside a record is private to libdamp: move logical
 * tiers in and out with damp_pack_tiers / damp_unpack_tiers.
 * The pool pointer must be 16-byte aligned.
 */
DAMP_API size_t damp_record_bytes(const damp_layout *layout); /* 0 if the layout is invalid */
DAMP_API size_t damp_slot_bytes(const damp_layout *layout);   /* 0 if the layout is invalid */

/* Storage bits per state value counted from the logical tiers (FP16 rows, codes and
 * metadata; record padding excluded).  Equals Eq. budgeted_allocation,
 * b(K_hi) = b_lo + (K_hi/d_k)(b_hi - b_lo) with b_hi = 16 and b_lo = 8 + 32/32 = 9:
 * 9.875 at K_hi = 16, d_k = 128 (Sec. 5.1).  Format 2 counts one FP32 scale per row
 * (b_lo = 8 + 32/d_v), although its records hold d_v/32 copies of it.
 * Returns -1.0 for an invalid layout. */
DAMP_API double damp_bits_per_value(const damp_layout *layout);

/*
 * One GDN decode step (Sec. 3.1 with Lambda_t = alpha_t I) of `batch` request
 * slots on the packed state, in place.
 *   state      [num_slots] packed slots (layout above), 16-B aligned, updated in place
 *   num_slots  slots in the pool (bounds slot indices; >= batch when slot_idx is NULL)
 *   slot_idx   int32 [batch]: batch row b updates slot slot_idx[b]; NULL means slot b.
 *              4-B aligned.  Indices must be distinct.
 *   batch      B >= 0 (0 enqueues nothing)
 *   perm       uint8 [H][d_k]: pi_h, packed row i holds key channel perm[h][i]
 *              (protected channels first).  16-B aligned.  Must be a permutation
 *              (not checked on the device).
 *   q, k       [B][H_qk][d_k] of in_dtype, natural key order, 16-B aligned
 *   v          [B][H_m][d_v] of in_dtype, 16-B aligned
 *   g          float [B][H_m]: log-decay, alpha = exp(g).  4-B aligned.
 *   beta       float [B][H_m]: delta-rule step size.  4-B aligned.
 *   o          float [B][H_m][d_v]: output S_t^T q_t from the FP32 post-update state,
 *              before requantization.  4-B aligned; must not overlap the pool.  Only
 *              the rows of the layout's heads are written (H_m = H without a head map).
 * (Per-head rows are indexed by model head, see damp_layout.)
 *   in_dtype   damp_in_dtype of q, k, v
 * Any lo_format; DAMP_LO_S8_ABSMAX_ROW runs the two-sweep step of that format.
 */
DAMP_API damp_status damp_gdn_decode_step(const damp_layout *layout, void *state, int64_t num_slots,
                                 const int32_t *slot_idx, int32_t batch, const uint8_t *perm,
                                 const void *q, const void *k, const void *v, const float *g,
                                 const float *beta, float *o, int32_t in_dtype, void *stream);

/*
 * One KDA decode step (Sec. 3.1 with Lambda_t = diag(exp(g_t))), as
 * damp_gdn_decode_step except:
 *   g          float [B][H_m][d_k]: per-key-channel log-decay in natural key order,
 *              a_u = exp(g_u).  16-B aligned.
 */
DAMP_API damp_status damp_kda_decode_step(const damp_layout *layout, void *state, int64_t num_slots,
                                 const int32_t *slot_idx, int32_t batch, const uint8_t *perm,
                                 const void *q, const void *k, const void *v, const float *g,
                                 const float *beta, float *o, int32_t in_dtype, void *stream);

/*
 * One decode step of a layer stored as head groups (App. E, "Common Per-Head Budget for
 * GDN": per-head protected-channel counts as budget-specific kernel groups; the
 * decay-tiered allocations of Tab. gdn_head_budget give half the heads K_fast and half
 * K_slow channels).  Group i is layouts[i] with its own pool states[i] (num_slots[i]
 * slots) and permutation table perms[i] (uint8 [layouts[i].num_heads][d_k]); every
 * group has a head map, and the head maps must partition 0 .. model_heads - 1 (not
 * checked on the device).  The operands q, k, v, g, beta, o, slot_idx, batch and
 * in_dtype are shared by the groups, with the shapes and alignment of
 * damp_gdn_decode_step (indexed by model head).
 *   n_groups   1 .. 8; all groups have the same model_heads, num_qk_heads, d_k, d_v
 *              (DAMP_ERR_SHAPE otherwise) and lo_format (DAMP_ERR_FORMAT otherwise);
 *              pools must not overlap each other, the operands or o (DAMP_ERR_ALIAS).
 * Two groups with d_k = 128, BF16 operands, lo_format 0 or 1 and K_hi pairs 12/20,
 * 8/24 or 4/28 run as one launch whose CTAs are split between the groups in proportion
 * to their records; other groups run one launch per group.  Results are the same as
 * one damp_gdn_decode_step call per group (the records up to the rounding of a rare
 * float-ordering tie: the one-launch form runs compile-time record layouts), except that in the one-launch form a lost record copy of the first
 * group also leaves the second group's records unwritten (DAMP_DEV_WAIT_TIMEOUT is set).
 * Every argument check runs before anything is enqueued.
 */
DAMP_API damp_status damp_gdn_decode_step_groups(const damp_layout *layouts, int32_t n_groups, void *const *states,
                                                 const int64_t *num_slots, const uint8_t *const *perms,
                                                 const int32_t *slot_idx, int32_t batch, const void *q,
                                                 const void *k, const void *v, const float *g, const float *beta,
                                                 float *o, int32_t in_dtype, void *stream);
/* The KDA step of a layer stored as head groups: as damp_gdn_decode_step_groups, with the
 * KDA operands of damp_kda_decode_step. */
DAMP_API damp_status damp_kda_decode_step_groups(const damp_layout *layouts, int32_t n_groups, void *const *states,
                                                 const int64_t *num_slots, const uint8_t *const *perms,
                                                 const int32_t *slot_idx, int32_t batch, const void *q,
                                                 const void *k, const void *v, const float *g, const float *beta,
                                                 float *o, int32_t in_dtype, void *stream);

/*
 * Uniform-INT8 baselines (the paper's INT8 / INT8+Hadamard rows of Tab. main):
 * the same steps with no FP16 tier.  layout->k_hi must be 0.
 */
DAMP_API damp_status damp_u8_gdn_decode_step(const damp_layout *layout, void *state, int64_t num_slots,
                                    const int32_t *slot_idx, int32_t batch, const uint8_t *perm,
                                    const void *q, const void *k, const void *v, const float *g,
                                    const float *beta, float *o, int32_t in_dtype, void *stream);
DAMP_API damp_status damp_u8_kda_decode_step(const damp_layout *layout, void *state, int64_t num_slots,
                                    const int32_t *slot_idx, int32_t batch, const uint8_t *perm,
                                    const void *q, const void *k, const void *v, const float *g,
                                    const float *beta, float *o, int32_t in_dtype, void *stream);

/*
 * FP32-state baselines: the deployment baseline of Sec. 6.1 ("default FP32
 * recurrent-state storage"), the same step on an FP32 state in natural key order.
 *   state  float [num_slots][H][d_k][d_v], 16-B aligned, updated in place
 * layout->k_hi and layout->lo_format are ignored; no permutation is taken.
 * Other arguments as in damp_gdn_decode_step / damp_kda_decode_step.
 */
DAMP_API damp_status damp_fp32_gdn_decode_step(const damp_layout *layout, float *state, int64_t num_slots,
                                      const int32_t *slot_idx, int32_t batch,
                                      const void *q, const void *k, const void *v, const float *g,
                                      const float *beta, float *o, int32_t in_dtype, void *stream);
DAMP_API damp_status damp_fp32_kda_decode_step(const damp_layout *layout, float *state, int64_t num_slots,
                                      const int32_t *slot_idx, int32_t batch,
                                      const void *q, const void *k, const void *v, const float *g,
                                      const float *beta, float *o, int32_t in_dtype, void *stream);

/*
 * One GDN prefill chunk on the packed state (App. A.5, "Prefill path"): for each
 * batch row, the packed slot is reconstructed, the recurrence runs in FP32 over the
 * chunk's tokens (Sec. 3.1 Eq. delta_update per token, o_t = S_t^T q_t) and the
 * chunk-final state is quantized once, in place, into the same packed cache that
 * decode steps and later chunks read.  An all-zero slot is the zero state (start of
 * a sequence).
 *   chunk_len  T >= 0 tokens per row (0 enqueues nothing)
 *   lengths    int32 [batch]: row b runs its first min(max(lengths[b], 0), T) tokens;
 *              NULL means T for every row.  A row with length 0 keeps its state.
 *              4-B aligned.
 *   q, k       [B][T][H_qk][d_k] of in_dtype, natural key order, 16-B aligned
 *   v          [B][T][H_m][d_v] of in_dtype, 16-B aligned
 *   g          float [B][T][H_m]: log-decay per token, 4-B aligned
 *   beta       float [B][T][H_m], 4-B aligned
 *   o          float [B][T][H_m][d_v]: o_t from the FP32 state after token t; rows past
 *              a row's length are not written.  Must not overlap the pool or inputs.
 *              4-B aligned; when it is 16-B aligned, chunks of T >= 32 tokens on the
 *              UINT8 tiers (formats 0, 1; d_k 64 or 128) run a kernel with less work per
 *              token, and chunks of T >= 32 tokens with d_k = d_v = 128, bf16 inputs and
 *              a UINT8 or UINT4 tier (formats 0, 1, 3, 4) run the chunkwise closed form of
 *              the delta rule on the tensor cores (pieces of up to 64 tokens; KDA pieces
 *              are cut shorter where a channel's decay within a piece would leave FP32).
 *              The results differ only in FP32 rounding order.
 * Other arguments as in damp_gdn_decode_step.  Any lo_format; the row-absmax format
 * (2) needs d_v <= 128 (DAMP_ERR_SHAPE otherwise): its row scale spans the value blocks
 * of a head, which four warps then share.
 */
DAMP_API damp_status damp_gdn_prefill_chunk(const damp_layout *layout, void *state, int64_t num_slots,
                                            const int32_t *slot_idx, int32_t batch, int32_t chunk_len,
                                            const int32_t *lengths, const uint8_t *perm, const void *q,
                                            const void *k, const void *v, const float *g, const float *beta,
                                            float *o, int32_t in_dtype, void *stream);

/* One KDA prefill chunk, as damp_gdn_prefill_chunk except
 *   g          float [B][T][H_m][d_k]: per-key-channel log-decay per token, 16-B aligned. */
DAMP_API damp_status damp_kda_prefill_chunk(const damp_layout *layout, void *state, int64_t num_slots,
                                            const int32_t *slot_idx, int32_t batch, int32_t chunk_len,
                                            const int32_t *lengths, const uint8_t *perm, const void *q,
                                            const void *k, const void *v, const float *g, const float *beta,
                                            float *o, int32_t in_dtype, void *stream);

/*
 * Write FP32 states into the packed cache: the hand-off from an FP32 prefix
 * state (App. A.5 "Prefill path": the chunk-final state is written directly into
 * the packed cache).  Row i of packed head h takes natural row perm[h][i];
 * rows < K_hi are rounded to FP16, the others H_32-transformed (format 0) and
 * quantized as their lo_format says.
 *   S      float [batch][H_m][d_k][d_v], natural key order, 16-B aligned, read only
 *          (the rows of the layout's heads)
 *   state, num_slots, slot_idx, batch, perm as in damp_gdn_decode_step
 */
DAMP_API damp_status damp_quantize_state(const damp_layout *layout, const float *S, const uint8_t *perm,
                                void *state, int64_t num_slots, const int32_t *slot_idx,
                                int32_t batch, void *stream);

/* Reconstruct FP32 states from the packed cache (the inverse map: FP16 rows widened,
 * codes dequantized s (q - z) (format 2: s q) and H_32-transformed back for format 0).
 *   S      float [batch][H_m][d_k][d_v] output, natural key order, 16-B aligned (the
 *          rows of the layout's heads are written) */
DAMP_API damp_status damp_dequantize_state(const damp_layout *layout, const void *state, int64_t num_slots,
                                  const int32_t *slot_idx, int32_t batch, const uint8_t *perm,
                                  float *S, void *stream);

/*
 * Copy logical tiers into / out of packed slots, bit for bit (no arithmetic).  The
 * tiers are indexed by the pool's own heads (no head map).
 *   hi     uint16 [batch][H][K_hi][d_v]            FP16 bit patterns (S_hi)
 *   codes  uint8  [batch][H][d_k-K_hi][d_v]        UINT8 codes (Q_lo); int8 for format 2,
 *                                                   E4M3 bit patterns for format 5,
 *          uint8  [batch][H][d_k-K_hi][d_v/2]      two UINT4 codes per byte for formats 3, 4
 *   meta   uint16 [batch][H][d_k-K_hi][d_v/32][2]  FP16 (s, z) (M_lo); for format 2
 *          float  [batch][H][d_k-K_hi]             FP32 row scales, for format 5
 *          float  [batch][H][d_k-K_hi][d_v/32]     FP32 group scales, through the same pointer
 * All three 4-B aligned.  NULL is allowed for an empty tier.  Unpacking format 2
 * returns the scale copy of each row's first record.
 */
DAMP_API damp_status damp_pack_tiers(const damp_layout *layout, const uint16_t *hi, const uint8_t *codes,
                            const uint16_t *meta, void *state, int64_t num_slots,
                            const int32_t *slot_idx, int32_t batch, void *stream);
DAMP_API damp_status damp_unpack_tiers(const damp_layout *layout, const void *state, int64_t num_slots,
                              const int32_t *slot_idx, int32_t batch, uint16_t *hi, uint8_t *codes,
                              uint16_t *meta, void *stream);

/*
 * Offline key-channel selection (Sec. 5.1 Eq. error_energy, persistence,
 * budgeted_selection; App. A.2 Eq. empirical_error_energy, empirical_persistence;
 * Algorithm 1), run on the GPU over calibration trajectories the caller produces
 * (for example with damp_fp32_*_decode_step on calibration documents).
 *
 * damp_calib_error_energy: E_acc[h][u] += sum_b || Q_lo(S_b,h)_{u:} - S_b,h,u: ||^2,
 *   the squared round-trip error of every key-channel row of the sampled FP32 states
 *   under layout->lo_format (H_32 + UINT8 G32, UINT8 G32, or row absmax INT8).
 *   S      float [batch][H_m][d_k][d_v] natural key order, 16-B aligned, read only
 *   E_acc  float [H_m][d_k], 4-B aligned, accumulated (the caller zeroes it first)
 * damp_calib_log_decay: G_acc[h][u] += sum_b g_b,h,u (KDA, g float [batch][H_m][d_k]) or
 *   sum_b g_b,h (GDN, g float [batch][H_m]: the head's log-decay counts for every channel).
 *   G_acc  float [H_m][d_k], 4-B aligned, accumulated
 * (S, g, E_acc and G_acc rows are model heads: row head_map[h] for held head h.)
 * damp_calib_select: E = E_acc / n_samples, a_eff = exp(G_acc / n_tokens),
 *   P = 1 / max(1 - a_eff^2, tau), C = E P (FP32), H = TopK_{K_hi}(C) with ties to the
 *   lower channel index, pi = the protected channels in ascending order, then the rest
 *   in ascending order.
 *   C_out     float [H][d_k] the scores of the held heads (4-B aligned)
 *   perm_out  uint8 [H][d_k] pi per held head, ready for the decode and prefill calls
 *   (E_acc and G_acc are read at the model-head rows of the held heads)
 *   tau       the persistence cap, 0 < tau <= 1 (the paper uses 1e-4)
 * Each accumulator entry has one writer and a fixed summation order: repeated runs
 * give identical bits.  No call allocates or uses global scratch memory.
 */
DAMP_API damp_status damp_calib_error_energy(const damp_layout *layout, const float *S, int32_t batch, float *E_acc,
                                             void *stream);
DAMP_API damp_status damp_calib_log_decay(const damp_layout *layout, const float *g, int32_t batch, int32_t kda,
                                          float *G_acc, void *stream);
/*
 * The accumulation of a calibration run in one call (App. A.2, Calibration Protocol;
 * Algorithm 1's statistics): the FP32 trajectories of n_docs calibration documents over
 * n_tokens tokens (one FP32-state step per token, Sec. 3.1, outputs not written), the
 * error energy of the states after tokens every, 2 every, ... (damp_calib_error_energy)
 * and the log-decay sums of every token (damp_calib_log_decay), enqueued by the library
 * instead of one call per token.
 *   layout     holds every head of the layer (no head map: DAMP_ERR_SHAPE); lo_format
 *              chooses the round trip of the error energy
 *   S          float [n_docs][H][d_k][d_v]: the trajectories' FP32 states (the initial
 *              states on entry, the final ones on return), 16-B aligned
 *   q, k       [n_tokens][n_docs][H_qk][d_k] of in_dtype, 16-B aligned
 *   v          [n_tokens][n_docs][H][d_v] of in_dtype, 16-B aligned
 *   g          float [n_tokens][n_docs][H][d_k] (kda != 0, 16-B aligned) or
 *              [n_tokens][n_docs][H] (GDN, 4-B aligned)
 *   beta       float [n_tokens][n_docs][H], 4-B aligned
 *   every      sampling period of the error energy, >= 1
 *   E_acc, G_acc  float [H][d_k], accumulated (the caller zeroes them first), 4-B aligned
 * Afterwards n_samples = n_docs * (n_tokens / every) and n_tokens * n_docs log-decay rows
 * go to damp_calib_select.  The results equal the per-token calls in the same order, bit for
 * bit.  Inputs, S and the accumulators must not overlap (DAMP_ERR_ALIAS).
 */
DAMP_API damp_status damp_calib_accumulate(const damp_layout *layout, float *S, int32_t n_docs, int32_t n_tokens,
                                           const void *q, const void *k, const void *v, const float *g,
                                           const float *beta, int32_t in_dtype, int32_t kda, int32_t every,
                                           float *E_acc, float *G_acc, void *stream);
DAMP_API damp_status damp_calib_select(const damp_layout *layout, const float *E_acc, int64_t n_samples,
                                       const float *G_acc, int64_t n_tokens, float tau, float *C_out,
                                       uint8_t *perm_out, void *stream);

/*
 * Test hook for the bounded waits (no counterpart in the paper; not part of the decode
 * path).  Runs the KDA packed step's kernel in a variant whose stage barriers expect 16
 * bytes more than each record copy delivers, with the wait limit cut to ~1 ms: every
 * warp's first wait runs out, the kernel settles the missing bytes itself, waits for
 * its copies in flight to land and returns.  No record and no row of o is written;
 * DAMP_DEV_WAIT_TIMEOUT is set in the device status word.  It lets a test check the
 * timeout path without a fault or a hang.  Arguments as damp_kda_decode_step; only the
 * layout d_k = d_v = 128, K_hi = 10, DAMP_LO_U8_AFFINE_G32_H32, BF16 inputs and no head map
 * (DAMP_ERR_SHAPE otherwise).
 */
DAMP_API damp_status damp_test_kda_wait_timeout(const damp_layout *layout, void *state, int64_t num_slots,
                                                const int32_t *slot_idx, int32_t batch, const uint8_t *perm,
                                                const void *q, const void *k, const void *v, const float *g,
                                                const float *beta, float *o, int32_t in_dtype, void *stream);

/* Reads and clears the device status word of the current device (DAMP_DEV_* bits).
 * It first waits for all work on the current device (cudaDeviceSynchronize: the one
 * call of libdamp that synchronizes), so every kernel enqueued before the call, on
 * any stream, has reported before the word is read; a bit is never cleared without
 * being returned.  DAMP_ERR_NULL if status is NULL; DAMP_ERR_CUDA if the wait or a
 * copy fails. */
DAMP_API damp_status damp_device_status(uint32_t *status);

/* Human-readable name of a status code (static string). */
DAMP_API const char *damp_status_string(damp_status status);

/* ABI version: 100 * major + minor. */
DAMP_API int32_t damp_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DAMP_H */
