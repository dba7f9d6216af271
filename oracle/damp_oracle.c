/*
 * damp_oracle.c -- plain, slow CPU oracle for the DAMP decode-step state update.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path (the CUDA library and
 * its Python binding) includes, links or calls this file.  It is used by the
 * tests, by __graft_entry__.smoke() and by the CPU-baseline leg of bench.py.
 *
 * Every function follows the paper (arxiv 2608.27513, "DAMP: Decay-Aware
 * Mixed-Precision Recurrent-State Quantization") in its own notation and
 * order, with no blocking, fusion or reordering:
 *   - the GDN/KDA delta-rule update and output read     (Sec. 3.1, Eq. delta_update)
 *   - the asymmetric affine block quantizer, UINT8, G=32,
 *     FP16 scale and zero point                          (Sec. 3.2, Eq. integer_quantizer;
 *                                                         App. A.1, Tab. quantizer_specs)
 *   - the normalized block-32 Hadamard transform H_32    (Sec. 4.1; App. A.1)
 *   - the packed mixed-precision state (S_hi, Q_lo, M_lo)
 *     in permuted key-channel order                      (Sec. 5.2; App. A.5, Eq. packed_state_layout)
 *   - one quantized recurrence step S^q_t = Q(A_t S^q_{t-1} + beta k v^T)
 *                                                        (Sec. 3.3, Eq. quantized_recurrence)
 *
 * Arithmetic is FP32 because the paper evaluates the recurrence in FP32
 * (Sec. 3.2; App. A.5 "Fused decode executor"); the FP16 conversions are
 * IEEE-754 binary16 round-to-nearest-even written out from the format's
 * definition.  Compile with -ffp-contract=off so that no multiply-add is
 * fused behind the reader's back.
 *
 * Readings where the paper is silent (each one is listed with its reason in
 * the design notes of the repository):
 *   round()      = round half to even, for z and for the codes;
 *   s, z         = computed in FP32, rounded to FP16, and the codes are then
 *                  encoded with the stored (FP16-rounded) s and z;
 *   s == 0       = widen [x_min, x_max] to contain 0 and recompute; if s is
 *                  still 0 use s = 1, z = 0;
 *   H_32         = Sylvester order (H_2n = [[H, H], [H, -H]]), entries
 *                  (-1)^popcount(i & j), scaled by fp32(1/sqrt(32)) after the sum;
 *   o_t          = S_t^T q_t on the FP32 post-update state, before requantization.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define DOR_G 32 /* group size along d_v (App. A.1) */

enum { DOR_FMT_U8_H32 = 0, DOR_FMT_U8 = 1, DOR_FMT_S8_ROW = 2, DOR_FMT_U4_H32 = 3, DOR_FMT_U4 = 4, DOR_FMT_E4M3 = 5 };
enum { DOR_GDN = 0, DOR_KDA = 1 };

/* ------------------------------------------------------------------------- */
/* IEEE-754 binary16 <-> binary32, round to nearest even.                     */
/* ------------------------------------------------------------------------- */

static uint32_t f32_bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }
static float bits_f32(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }

uint16_t dor_f32_to_f16(float f)
{
    uint32_t x = f32_bits(f);
    uint32_t sign = (x >> 16) & 0x8000u;
    uint32_t ax = x & 0x7FFFFFFFu;
    if (ax >= 0x7F800000u) { /* inf or NaN (NaN keeps a quiet payload bit) */
        if (ax == 0x7F800000u) return (uint16_t)(sign | 0x7C00u);
        return (uint16_t)(sign | 0x7E00u | ((ax >> 13) & 0x3FFu));
    }
    if (ax >= 0x477FF000u) /* >= 65520: rounds to infinity */
        return (uint16_t)(sign | 0x7C00u);
    if (ax < 0x38800000u) { /* below 2^-14: binary16 subnormal or zero */
        if (ax < 0x33000000u) return (uint16_t)sign; /* below 2^-25 (ties to even 0 at 2^-25) */
        uint32_t e = ax >> 23;
        uint32_t m = (ax & 0x7FFFFFu) | 0x800000u;
        uint32_t shift = 126u - e; /* value / 2^-24 = m * 2^(e-126) */
        uint32_t q = m >> shift;
        uint32_t rem = m & ((1u << shift) - 1u);
        uint32_t half = 1u << (shift - 1u);
        if (rem > half || (rem == half && (q & 1u))) q++;
        return (uint16_t)(sign | q);
    }
    uint32_t h = ((((ax >> 23) - 112u)) << 10) | ((ax & 0x7FFFFFu) >> 13);
    uint32_t rem = ax & 0x1FFFu;
    if (rem > 0x1000u || (rem == 0x1000u && (h & 1u))) h++; /* a carry may reach the exponent */
    return (uint16_t)(sign | h);
}

float dor_f16_to_f32(uint16_t h)
{
    uint32_t sign = ((uint32_t)h & 0x8000u) << 16;
    uint32_t e = ((uint32_t)h >> 10) & 0x1Fu;
    uint32_t m = (uint32_t)h & 0x3FFu;
    if (e == 0) {
        float v = (float)m * 5.9604644775390625e-8f; /* m * 2^-24, exact */
        return bits_f32(f32_bits(v) | sign);
    }
    if (e == 31) return bits_f32(sign | 0x7F800000u | (m << 13));
    return bits_f32(sign | ((e + 112u) << 23) | (m << 13));
}

void dor_f32_to_f16_array(const float *x, uint16_t *h, int64_t n)
{
    for (int64_t i = 0; i < n; i++) h[i] = dor_f32_to_f16(x[i]);
}

void dor_f16_to_f32_array(const uint16_t *h, float *x, int64_t n)
{
    for (int64_t i = 0; i < n; i++) x[i] = dor_f16_to_f32(h[i]);
}

static float f16_round(float x) { return dor_f16_to_f32(dor_f32_to_f16(x)); }

/* ------------------------------------------------------------------------- */
/* Normalized block-32 Hadamard transform (Sec. 4.1; App. A.1).              */
/* y_i = (1/sqrt 32) * sum_j (-1)^popcount(i & j) x_j ; H_32 is its own       */
/* inverse, so the same routine is the forward and the inverse transform.    */
/* ------------------------------------------------------------------------- */

static int popcount5(int v)
{
    int c = 0;
    for (int b = 0; b < 5; b++) c += (v >> b) & 1;
    return c;
}

void dor_hadamard32(const float *x, float *y)
{
    const float scale = (float)(1.0 / sqrt(32.0));
    for (int i = 0; i < DOR_G; i++) {
        float acc = 0.0f;
        for (int j = 0; j < DOR_G; j++) {
            if (popcount5(i & j) & 1) acc = acc - x[j];
            else acc = acc + x[j];
        }
        y[i] = acc * scale;
    }
}

/* ------------------------------------------------------------------------- */
/* Asymmetric affine UINT8 quantizer for one group of G = 32 values          */
/* (Sec. 3.2, Eq. integer_quantizer with b = 8; App. A.1: FP16 s and z,       */
/* codes saturate to the unsigned range).                                    */
/*   s = (x_max - x_min) / (2^b - 1),  z = round(-x_min / s),                */
/*   q_i = round(x_i / s) + z,         Q(x_i) = s * (q_i - z).               */
/* sz[0] = s, sz[1] = z, both binary16 bit patterns.                         */
/* ------------------------------------------------------------------------- */

/* The affine rule for b-bit codes (levels = 2^b - 1); q receives the codes as ints. */
static void quant_group_affine(const float *x, float levels, int *q, uint16_t *sz)
{
    float x_min = x[0], x_max = x[0];
    for (int i = 1; i < DOR_G; i++) {
        if (x[i] < x_min) x_min = x[i];
        if (x[i] > x_max) x_max = x[i];
    }
    float s = f16_round((x_max - x_min) / levels);
    if (s == 0.0f) { /* degenerate block: widen the range to contain 0 */
        if (x_min > 0.0f) x_min = 0.0f;
        if (x_max < 0.0f) x_max = 0.0f;
        s = f16_round((x_max - x_min) / levels);
    }
    if (s == 0.0f) s = 1.0f; /* all (near-)zero block */
    uint16_t z16 = dor_f32_to_f16(rintf(-x_min / s));
    float z = dor_f16_to_f32(z16);
    for (int i = 0; i < DOR_G; i++) {
        float t = rintf(x[i] / s) + z;
        if (t < 0.0f) t = 0.0f;
        if (t > levels) t = levels;
        q[i] = (int)t;
    }
    sz[0] = dor_f32_to_f16(s);
    sz[1] = z16;
}

void dor_quant_group_u8(const float *x, uint8_t *q, uint16_t *sz)
{
    int c[DOR_G];
    quant_group_affine(x, 255.0f, c, sz);
    for (int i = 0; i < DOR_G; i++) q[i] = (uint8_t)c[i];
}

void dor_dequant_group_u8(const uint8_t *q, const uint16_t *sz, float *x)
{
    float s = dor_f16_to_f32(sz[0]);
    float z = dor_f16_to_f32(sz[1]);
    for (int i = 0; i < DOR_G; i++) x[i] = s * ((float)q[i] - z);
}

/* UINT4 variant (Eq. integer_quantizer with b = 4, App. A.1): levels 0..15, FP16
 * (s, z); the 32 codes are packed two per byte, value 2i in the low nibble of q[i]. */
void dor_quant_group_u4(const float *x, uint8_t *q, uint16_t *sz)
{
    int c[DOR_G];
    quant_group_affine(x, 15.0f, c, sz);
    for (int i = 0; i < DOR_G / 2; i++) q[i] = (uint8_t)(c[2 * i] | (c[2 * i + 1] << 4));
}

void dor_dequant_group_u4(const uint8_t *q, const uint16_t *sz, float *x)
{
    float s = dor_f16_to_f32(sz[0]);
    float z = dor_f16_to_f32(sz[1]);
    for (int i = 0; i < DOR_G; i++) x[i] = s * ((float)((q[i / 2] >> (4 * (i & 1))) & 15) - z);
}

/* ------------------------------------------------------------------------- */
/* FP8 E4M3: sign, 4 exponent bits (bias 7), 3 mantissa bits.  Exponent field */
/* e = 1..15 gives 2^(e-7) (1 + m/8), e = 0 the subnormals 2^-6 (m/8); e = 15 */
/* with m = 7 is NaN, so the largest finite magnitude is 448; no infinities.  */
/* ------------------------------------------------------------------------- */

float dor_e4m3_to_f32(uint8_t b)
{
    int sign = b >> 7, e = (b >> 3) & 15, m = b & 7;
    double v;
    if (e == 15 && m == 7) return NAN;
    if (e == 0) v = ldexp(m / 8.0, -6);
    else v = ldexp(1.0 + m / 8.0, e - 7);
    return (float)(sign ? -v : v);
}

/* Nearest E4M3 value of a finite float, ties to the even mantissa, magnitudes of
 * 448 and above saturating to 448. */
uint8_t dor_f32_to_e4m3(float x)
{
    int sign = signbit(x) ? 1 : 0;
    double a = fabs((double)x);
    if (a >= 448.0) return (uint8_t)(sign << 7 | 0x7E);
    int e = -6;                       /* binade of a (values below 2^-6 share the subnormal spacing) */
    while (e < 8 && a >= ldexp(1.0, e + 1)) e++;
    double quantum = ldexp(1.0, e - 3); /* spacing of E4M3 values in [2^e, 2^(e+1)) */
    double v = nearbyint(a / quantum) * quantum; /* a / quantum is exact; ties to even */
    if (v == 0.0) return (uint8_t)(sign << 7);
    int ev = -6;
    while (ev < 8 && v >= ldexp(1.0, ev + 1)) ev++;
    int field, m;
    if (v < ldexp(1.0, -6)) {
        field = 0;
        m = (int)(v / ldexp(1.0, -9));
    } else {
        field = ev + 7;
        m = (int)((v / ldexp(1.0, ev) - 1.0) * 8.0);
    }
    return (uint8_t)(sign << 7 | field << 3 | m);
}

/* FP8 group quantizer (App. A.1, Eq. fp8_storage): one FP32 scale per 32 values,
 *   s = max(max_i |x_i|, 1e-10) / 448,  q_i = E4M3(clip(x_i / s, -448, 448)),
 *   Q(x_i) = s * FP32(q_i). */
void dor_quant_group_e4m3(const float *x, uint8_t *q, float *s_out)
{
    float amax = 0.0f;
    for (int i = 0; i < DOR_G; i++) {
        float a = fabsf(x[i]);
        if (a > amax) amax = a;
    }
    float s = (amax > 1e-10f ? amax : 1e-10f) / 448.0f;
    for (int i = 0; i < DOR_G; i++) {
        float t = x[i] / s;
        if (t < -448.0f) t = -448.0f;
        if (t > 448.0f) t = 448.0f;
        q[i] = dor_f32_to_e4m3(t);
    }
    *s_out = s;
}

void dor_dequant_group_e4m3(const uint8_t *q, float s, float *x)
{
    for (int i = 0; i < DOR_G; i++) x[i] = s * dor_e4m3_to_f32(q[i]);
}

/* Per-row symmetric absmax INT8 with an FP32 scale and round-to-nearest-even:
 * the fallback quantizer for a low tier the paper would leave open.
 *   s = max_i |x_i| / 127,  q_i = sat_[-127,127](round(x_i / s)),  s = 0 -> q = 0. */
void dor_quant_row_s8(const float *x, int n, int8_t *q, float *s_out)
{
    float amax = 0.0f;
    for (int i = 0; i < n; i++) {
        float a = fabsf(x[i]);
        if (a > amax) amax = a;
    }
    float s = amax / 127.0f;
    for (int i = 0; i < n; i++) {
        float t = (s == 0.0f) ? 0.0f : rintf(x[i] / s);
        if (t < -127.0f) t = -127.0f;
        if (t > 127.0f) t = 127.0f;
        q[i] = (int8_t)t;
    }
    *s_out = s;
}

void dor_dequant_row_s8(const int8_t *q, int n, float s, float *x)
{
    for (int i = 0; i < n; i++) x[i] = s * (float)q[i];
}

/* ------------------------------------------------------------------------- */
/* Q_lo on one natural-domain row of d_v values: quantize, then reconstruct  */
/* (the deployed low-tier mapping of App. A.1 / App. A.2).                   */
/* ------------------------------------------------------------------------- */

static int code_bits(int fmt) { return fmt == DOR_FMT_U4_H32 || fmt == DOR_FMT_U4 ? 4 : 8; }
static int uses_h32(int fmt) { return fmt == DOR_FMT_U8_H32 || fmt == DOR_FMT_U4_H32; }

static void lo_encode_row(int dv, int fmt, const float *x, void *codes_row, void *meta_row)
{
    if (fmt == DOR_FMT_S8_ROW) {
        dor_quant_row_s8(x, dv, (int8_t *)codes_row, (float *)meta_row);
        return;
    }
    for (int g = 0; g < dv / DOR_G; g++) {
        float xt[DOR_G];
        if (uses_h32(fmt)) dor_hadamard32(x + g * DOR_G, xt);
        else memcpy(xt, x + g * DOR_G, sizeof xt);
        uint8_t *cg = (uint8_t *)codes_row + g * DOR_G * code_bits(fmt) / 8;
        if (fmt == DOR_FMT_E4M3) dor_quant_group_e4m3(xt, cg, (float *)meta_row + g);
        else if (code_bits(fmt) == 4) dor_quant_group_u4(xt, cg, (uint16_t *)meta_row + 2 * g);
        else dor_quant_group_u8(xt, cg, (uint16_t *)meta_row + 2 * g);
    }
}

static void lo_decode_row(int dv, int fmt, const void *codes_row, const void *meta_row, float *x)
{
    if (fmt == DOR_FMT_S8_ROW) {
        dor_dequant_row_s8((const int8_t *)codes_row, dv, *(const float *)meta_row, x);
        return;
    }
    for (int g = 0; g < dv / DOR_G; g++) {
        float xt[DOR_G];
        const uint8_t *cg = (const uint8_t *)codes_row + g * DOR_G * code_bits(fmt) / 8;
        if (fmt == DOR_FMT_E4M3) dor_dequant_group_e4m3(cg, ((const float *)meta_row)[g], xt);
        else if (code_bits(fmt) == 4) dor_dequant_group_u4(cg, (const uint16_t *)meta_row + 2 * g, xt);
        else dor_dequant_group_u8(cg, (const uint16_t *)meta_row + 2 * g, xt);
        if (uses_h32(fmt)) dor_hadamard32(xt, x + g * DOR_G);
        else memcpy(x + g * DOR_G, xt, sizeof xt);
    }
}

static int64_t meta_row_bytes(int dv, int fmt)
{
    return fmt == DOR_FMT_S8_ROW ? 4 : (int64_t)(dv / DOR_G) * 4;
}

static int64_t code_row_bytes(int dv, int fmt) { return (int64_t)dv * code_bits(fmt) / 8; }

void dor_qdq_rows(int64_t n_rows, int dv, int fmt, const float *x, float *out)
{
    uint8_t codes[4096];
    uint8_t meta[1024];
    for (int64_t r = 0; r < n_rows; r++) {
        lo_encode_row(dv, fmt, x + r * dv, codes, meta);
        lo_decode_row(dv, fmt, codes, meta, out + r * dv);
    }
}

/* ------------------------------------------------------------------------- */
/* Packed mixed-precision state of one head (Sec. 5.2; App. A.5).            */
/* Packed row i holds key channel perm[i]; rows 0..K-1 are the FP16 tier     */
/* S_hi[K][d_v]; rows K..d_k-1 are the low tier Q_lo[d_k-K][d_v] with        */
/* metadata M_lo[d_k-K][d_v/G][2] (s, z).  S is the natural-order FP32 state. */
/* Returns 0, or -1 if perm is not a permutation of 0..d_k-1 or a size is    */
/* outside what the oracle supports.                                         */
/* ------------------------------------------------------------------------- */

static int check_args(int dk, int dv, int K, int fmt, const uint8_t *perm)
{
    if (dk <= 0 || dk > 256 || dv <= 0 || dv > 4096 || dv % DOR_G) return -1;
    if (K < 0 || K > dk || fmt < 0 || fmt > 5) return -1;
    int seen[256] = {0};
    for (int i = 0; i < dk; i++) {
        if (perm[i] >= dk || seen[perm[i]]) return -1;
        seen[perm[i]] = 1;
    }
    return 0;
}

int dor_pack_head(int dk, int dv, int K, int fmt, const uint8_t *perm, const float *S,
                  uint16_t *hi, void *codes, void *meta)
{
    if (check_args(dk, dv, K, fmt, perm)) return -1;
    int64_t mrow = meta_row_bytes(dv, fmt);
    for (int i = 0; i < dk; i++) {
        const float *row = S + (int64_t)perm[i] * dv;
        if (i < K) {
            for (int j = 0; j < dv; j++) hi[(int64_t)i * dv + j] = dor_f32_to_f16(row[j]);
        } else {
            int r = i - K;
            lo_encode_row(dv, fmt, row, (uint8_t *)codes + r * code_row_bytes(dv, fmt), (uint8_t *)meta + r * mrow);
        }
    }
    return 0;
}

int dor_unpack_head(int dk, int dv, int K, int fmt, const uint8_t *perm, const uint16_t *hi,
                    const void *codes, const void *meta, float *S)
{
    if (check_args(dk, dv, K, fmt, perm)) return -1;
    int64_t mrow = meta_row_bytes(dv, fmt);
    for (int i = 0; i < dk; i++) {
        float *row = S + (int64_t)perm[i] * dv;
        if (i < K) {
            for (int j = 0; j < dv; j++) row[j] = dor_f16_to_f32(hi[(int64_t)i * dv + j]);
        } else {
            int r = i - K;
            lo_decode_row(dv, fmt, (const uint8_t *)codes + r * code_row_bytes(dv, fmt), (const uint8_t *)meta + r * mrow, row);
        }
    }
    return 0;
}

/* ------------------------------------------------------------------------- */
/* One delta-rule step on a natural-order FP32 state (Sec. 3.1).             */
/*   S_bar = Lambda_t S_{t-1}          (row u scaled by a[u])                */
/*   r     = S_bar^T k                 (the current key reads the state)     */
/*   delta = v - r                                                           */
/*   S_t   = S_bar + beta k delta^T    (Eq. delta_update)                    */
/*   o     = S_t^T q                   (output read, scale 1)                */
/* GDN passes a[u] = alpha for every u; KDA passes a[u] = exp(g_u).          */
/* ------------------------------------------------------------------------- */

void dor_delta_step(int dk, int dv, float *S, const float *q, const float *k, const float *v,
                    const float *a, float beta, float *o)
{
    float r[4096];
    for (int u = 0; u < dk; u++)
        for (int j = 0; j < dv; j++) S[(int64_t)u * dv + j] = a[u] * S[(int64_t)u * dv + j];
    for (int j = 0; j < dv; j++) {
        float acc = 0.0f;
        for (int u = 0; u < dk; u++) acc = acc + S[(int64_t)u * dv + j] * k[u];
        r[j] = acc;
    }
    for (int u = 0; u < dk; u++) {
        float bk = beta * k[u];
        for (int j = 0; j < dv; j++) {
            float delta = v[j] - r[j];
            S[(int64_t)u * dv + j] = S[(int64_t)u * dv + j] + bk * delta;
        }
    }
    for (int j = 0; j < dv; j++) {
        float acc = 0.0f;
        for (int u = 0; u < dk; u++) acc = acc + S[(int64_t)u * dv + j] * q[u];
        o[j] = acc;
    }
}

/* Decay of one head from its log-decay input: GDN g is one scalar per head
 * (alpha = exp(g)), KDA g is one value per key channel (a_u = exp(g_u)). */
static void decay_from_log(int kind, int dk, const float *g, float *a)
{
    for (int u = 0; u < dk; u++) a[u] = expf(kind == DOR_GDN ? g[0] : g[u]);
}

/* ------------------------------------------------------------------------- */
/* One quantized recurrence step of one head on the packed state             */
/* (Sec. 3.3, Eq. quantized_recurrence): reconstruct the packed state,      */
/* run the FP32 delta step, requantize once, write both tiers back.         */
/* ------------------------------------------------------------------------- */

int dor_mixed_step(int dk, int dv, int K, int fmt, int kind, const uint8_t *perm,
                   uint16_t *hi, void *codes, void *meta,
                   const float *q, const float *k, const float *v, const float *g, float beta, float *o)
{
    static float S[256 * 4096];
    float a[256];
    if (check_args(dk, dv, K, fmt, perm)) return -1;
    if (dor_unpack_head(dk, dv, K, fmt, perm, hi, codes, meta, S)) return -1;
    decay_from_log(kind, dk, g, a);
    dor_delta_step(dk, dv, S, q, k, v, a, beta, o);
    return dor_pack_head(dk, dv, K, fmt, perm, S, hi, codes, meta);
}

/* ------------------------------------------------------------------------- */
/* One prefill chunk of one head (App. A.5, "Prefill path"): reconstruct the */
/* packed state, evaluate the exact FP32 recurrence over the chunk's T       */
/* tokens (Eq. delta_update per token, o_t = S_t^T q_t), then quantize the   */
/* chunk-final state once into the packed tiers.  T = 0 leaves the tiers     */
/* untouched.  Token t reads q + t*dk, k + t*dk, v + t*dv, g + t*gdim and    */
/* beta[t]; o receives T rows of d_v values.                                 */
/* ------------------------------------------------------------------------- */

int dor_prefill_chunk(int dk, int dv, int K, int fmt, int kind, const uint8_t *perm,
                      uint16_t *hi, void *codes, void *meta, int T,
                      const float *q, const float *k, const float *v, const float *g, const float *beta,
                      float *o)
{
    static float S[256 * 4096];
    float a[256];
    int gdim = kind == DOR_GDN ? 1 : dk;
    if (check_args(dk, dv, K, fmt, perm)) return -1;
    if (T <= 0) return 0;
    if (dor_unpack_head(dk, dv, K, fmt, perm, hi, codes, meta, S)) return -1;
    for (int t = 0; t < T; t++) {
        decay_from_log(kind, dk, g + (int64_t)t * gdim, a);
        dor_delta_step(dk, dv, S, q + (int64_t)t * dk, k + (int64_t)t * dk, v + (int64_t)t * dv, a, beta[t],
                       o + (int64_t)t * dv);
    }
    return dor_pack_head(dk, dv, K, fmt, perm, S, hi, codes, meta);
}

/* ------------------------------------------------------------------------- */
/* Plain loops over n independent heads (each head: its own permutation,     */
/* operands and state).  Arrays are dense, head-major.                       */
/* ------------------------------------------------------------------------- */

int dor_mixed_step_heads(int64_t n, int dk, int dv, int K, int fmt, int kind, const uint8_t *perm,
                         uint16_t *hi, void *codes, void *meta,
                         const float *q, const float *k, const float *v, const float *g,
                         const float *beta, float *o)
{
    int64_t code_b = (int64_t)(dk - K) * code_row_bytes(dv, fmt);
    int64_t meta_b = (int64_t)(dk - K) * meta_row_bytes(dv, fmt);
    int64_t gdim = kind == DOR_GDN ? 1 : dk;
    for (int64_t h = 0; h < n; h++) {
        int rc = dor_mixed_step(dk, dv, K, fmt, kind, perm + h * dk, hi + h * (int64_t)K * dv,
                                (uint8_t *)codes + h * code_b, (uint8_t *)meta + h * meta_b,
                                q + h * dk, k + h * dk, v + h * dv, g + h * gdim, beta[h], o + h * dv);
        if (rc) return rc;
    }
    return 0;
}

/* n heads, each with its own chunk length T[h] <= Tmax: operands head-major
 * [n][Tmax][...], o [n][Tmax][dv] (rows t >= T[h] untouched). */
int dor_prefill_chunk_heads(int64_t n, int dk, int dv, int K, int fmt, int kind, const uint8_t *perm,
                            uint16_t *hi, void *codes, void *meta, int Tmax, const int32_t *T,
                            const float *q, const float *k, const float *v, const float *g,
                            const float *beta, float *o)
{
    int64_t code_b = (int64_t)(dk - K) * code_row_bytes(dv, fmt);
    int64_t meta_b = (int64_t)(dk - K) * meta_row_bytes(dv, fmt);
    int64_t gdim = kind == DOR_GDN ? 1 : dk;
    for (int64_t h = 0; h < n; h++) {
        if (T[h] < 0 || T[h] > Tmax) return -1;
        int rc = dor_prefill_chunk(dk, dv, K, fmt, kind, perm + h * dk, hi + h * (int64_t)K * dv,
                                   (uint8_t *)codes + h * code_b, (uint8_t *)meta + h * meta_b, T[h],
                                   q + h * Tmax * dk, k + h * Tmax * dk, v + h * Tmax * dv,
                                   g + h * Tmax * gdim, beta + h * Tmax, o + h * Tmax * dv);
        if (rc) return rc;
    }
    return 0;
}

void dor_delta_step_heads(int64_t n, int dk, int dv, int kind, float *S,
                          const float *q, const float *k, const float *v, const float *g,
                          const float *beta, float *o)
{
    float a[256];
    int64_t gdim = kind == DOR_GDN ? 1 : dk;
    for (int64_t h = 0; h < n; h++) {
        decay_from_log(kind, dk, g + h * gdim, a);
        dor_delta_step(dk, dv, S + h * (int64_t)dk * dv, q + h * dk, k + h * dk, v + h * dv, a,
                       beta[h], o + h * dv);
    }
}

int dor_pack_heads(int64_t n, int dk, int dv, int K, int fmt, const uint8_t *perm, const float *S,
                   uint16_t *hi, void *codes, void *meta)
{
    int64_t code_b = (int64_t)(dk - K) * code_row_bytes(dv, fmt);
    int64_t meta_b = (int64_t)(dk - K) * meta_row_bytes(dv, fmt);
    for (int64_t h = 0; h < n; h++) {
        int rc = dor_pack_head(dk, dv, K, fmt, perm + h * dk, S + h * (int64_t)dk * dv,
                               hi + h * (int64_t)K * dv, (uint8_t *)codes + h * code_b,
                               (uint8_t *)meta + h * meta_b);
        if (rc) return rc;
    }
    return 0;
}

int dor_unpack_heads(int64_t n, int dk, int dv, int K, int fmt, const uint8_t *perm, const uint16_t *hi,
                     const void *codes, const void *meta, float *S)
{
    int64_t code_b = (int64_t)(dk - K) * code_row_bytes(dv, fmt);
    int64_t meta_b = (int64_t)(dk - K) * meta_row_bytes(dv, fmt);
    for (int64_t h = 0; h < n; h++) {
        int rc = dor_unpack_head(dk, dv, K, fmt, perm + h * dk, hi + h * (int64_t)K * dv,
                                 (const uint8_t *)codes + h * code_b, (const uint8_t *)meta + h * meta_b,
                                 S + h * (int64_t)dk * dv);
        if (rc) return rc;
    }
    return 0;
}
