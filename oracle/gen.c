/*
 * Oracle: seeded input generation, plain C (TEST INFRASTRUCTURE ONLY).
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
 * arm may load this code.  It shares nothing with the CUDA path: both sides
 * implement the same published counter-based generator from its definition.
 *
 * What it computes.  A benchmarking command generates seeded inputs before the
 * check and the timed loop (paper Section 2.1, "Benchmarking command"; Section
 * 1).  The paper names no generator, so the workload definition fixes it:
 * SplitMix64(seed, index) mapped to U[-1,1] rounded to bf16 for GEMM operands,
 * and N(0, 4) via Box-Muller in fp32 for the softmax input.  Where that
 * definition is silent this code takes these readings: each tensor has its own
 * stream key; one 64-bit draw feeds an element pair (bits 63..40 and 31..8);
 * fp16 GEMM operands take the same 24-bit values rounded RNE to IEEE binary16;
 * "N(0, 4)" means variance 4 (sigma = 2); Box-Muller's ln and sincos are the
 * fp32 series routines below, evaluated operation by operation.
 *
 * SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014; constants as published by Vigna):
 *     state_{j+1} = state_j + GAMMA,  output_j = mix64(state_{j+1}).
 *
 * Build flags matter for bit-exactness: -ffp-contract=off, no -ffast-math,
 * IEEE fp32 arithmetic (FLT_EVAL_METHOD == 0 on x86-64 SSE and AArch64).
 * Every fused multiply-add below is an explicit fmaf() call.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#if defined(FLT_EVAL_METHOD) && FLT_EVAL_METHOD != 0
#error "oracle needs FLT_EVAL_METHOD == 0 (IEEE single-precision arithmetic)"
#endif

#define GAMMA 0x9E3779B97F4A7C15ull

/* ---------------------------------------------------------------- hash ---- */

/* SplitMix64 output mix (Stafford's "Mix13" variant as used by SplitMix64). */
uint64_t oracle_mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* Per-tensor stream key: SplitMix64 seeded with `seed`, advanced tensor_id+1
 * steps; its output starts that tensor's own stream. */
uint64_t oracle_stream_key(uint64_t seed, uint32_t tensor_id)
{
    return oracle_mix64(seed + ((uint64_t)tensor_id + 1ull) * GAMMA);
}

/* Draw j of a stream: SplitMix64 state after j+1 steps from `key`, mixed. */
uint64_t oracle_draw(uint64_t key, uint64_t j)
{
    return oracle_mix64(key + (j + 1ull) * GAMMA);
}

/* ------------------------------------------------------------ bf16 ------- */

static uint32_t f32_bits(float x) { uint32_t u; memcpy(&u, &x, 4); return u; }
static float bits_f32(uint32_t u) { float x; memcpy(&x, &u, 4); return x; }

/* IEEE round-to-nearest-even from fp32 to bf16 (finite inputs only). */
uint16_t oracle_f32_to_bf16_rne(float x)
{
    uint32_t u = f32_bits(x);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

float oracle_bf16_to_f32(uint16_t h) { return bits_f32((uint32_t)h << 16); }

/* ------------------------------------------------------ uniform U[-1,1] --- */

/* Element e of a uniform bf16 tensor.  Elements 2j and 2j+1 share draw j:
 * element 2j takes bits 63..40, element 2j+1 takes bits 31..8.  A 24-bit
 * value b maps to x = (b - 2^23) * 2^-23, exact in fp32 and in [-1, 1); the
 * bf16 result is RNE(x), which can round up to +1.0. */
uint16_t oracle_uniform_bf16_at(uint64_t key, uint64_t e)
{
    uint64_t z = oracle_draw(key, e >> 1);
    uint32_t b = (e & 1u) ? (uint32_t)((z >> 8) & 0xFFFFFFu) : (uint32_t)(z >> 40);
    float x = (float)((int32_t)b - (int32_t)(1 << 23)) * 0x1p-23f;
    return oracle_f32_to_bf16_rne(x);
}

/* ------------------------------------------------------------ fp16 ------- */

/* IEEE binary16 round-to-nearest-even from fp32, subnormals included.  With
 * x = m 2^(e-23) (m the 24-bit significand), a normal binary16 keeps 11
 * significant bits, quantum 2^(e-10), for e >= -14; below, the quantum is the
 * subnormal step 2^-24.  Magnitudes past the largest binary16 give infinity;
 * NaN stays NaN (quiet). */
uint16_t oracle_f32_to_f16_rne(float x)
{
    uint32_t u = f32_bits(x);
    uint16_t sign = (uint16_t)((u >> 16) & 0x8000u);
    uint32_t a = u & 0x7FFFFFFFu;
    if (a >= 0x7F800000u) return (uint16_t)(sign | 0x7C00u | (a > 0x7F800000u ? 0x200u : 0u));
    int32_t e;
    uint32_t m;
    if (a >= 0x00800000u) {
        e = (int32_t)(a >> 23) - 127;
        m = (a & 0x7FFFFFu) | 0x800000u;
    } else {
        e = -126;
        m = a;
    }
    int32_t shift = (e >= -14) ? 13 : (-1 - e);
    if (shift > 24) return sign;  /* below half the smallest subnormal */
    uint32_t q = m >> shift;
    uint32_t rem = m & ((1u << shift) - 1u);
    uint32_t half = 1u << (shift - 1);
    if (rem > half || (rem == half && (q & 1u))) q += 1u;
    if (e >= -14) {
        int32_t E = e + 15;
        if (q == 0x800u) {  /* rounding carried into the next binade */
            q = 0x400u;
            E += 1;
        }
        if (E >= 31) return (uint16_t)(sign | 0x7C00u);
        return (uint16_t)(sign | (uint32_t)(E << 10) | (q & 0x3FFu));
    }
    return (uint16_t)(sign | q);  /* q == 0x400 is the smallest normal: same encoding */
}

/* Element e of a uniform fp16 tensor: the same 24-bit value as the bf16 form,
 * x = (b - 2^23) 2^-23 exact in fp32, rounded RNE to binary16. */
uint16_t oracle_uniform_f16_at(uint64_t key, uint64_t e)
{
    uint64_t z = oracle_draw(key, e >> 1);
    uint32_t b = (e & 1u) ? (uint32_t)((z >> 8) & 0xFFFFFFu) : (uint32_t)(z >> 40);
    float x = (float)((int32_t)b - (int32_t)(1 << 23)) * 0x1p-23f;
    return oracle_f32_to_f16_rne(x);
}

void oracle_f32_to_f16_many(const float *x, int64_t n, uint16_t *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_f32_to_f16_rne(x[i]);
}

/* ------------------------------------------------ fp32 ln and sincos ----- */
/* Both routines are written from textbook series (no library math is used in
 * the value path); each fp32 operation is one IEEE round-to-nearest step.
 * Their coefficients are the fp32 roundings of closed forms, computed here
 * from those closed forms in double precision. */

static float C_ATANH[4];   /* 1/3, 1/5, 1/7, 1/9 */
static float C_SIN[5];     /* (-1)^k (pi/2)^(2k+1) / (2k+1)!, k = 0..4 */
static float C_COS[5];     /* (-1)^k (pi/2)^(2k) / (2k)!,     k = 1..5 */
static float LN2_F;        /* RN32(ln 2) */
static float SQRT2_F;      /* RN32(sqrt 2) */
static int   coeffs_ready;

static void init_coeffs(void)
{
    if (coeffs_ready) return;
    const double pio2 = 1.5707963267948966192313216916398;
    for (int k = 0; k < 4; ++k) C_ATANH[k] = (float)(1.0 / (double)(2 * k + 3));
    for (int k = 0; k < 5; ++k) {
        int n = 2 * k + 1;
        double t = 1.0;
        for (int i = 1; i <= n; ++i) t *= pio2 / (double)i;
        C_SIN[k] = (float)((k & 1) ? -t : t);
    }
    for (int k = 1; k <= 5; ++k) {
        int n = 2 * k;
        double t = 1.0;
        for (int i = 1; i <= n; ++i) t *= pio2 / (double)i;
        C_COS[k - 1] = (float)((k & 1) ? -t : t);
    }
    LN2_F = (float)0.69314718055994530941723212145818;
    SQRT2_F = (float)1.4142135623730950488016887242097;
    coeffs_ready = 1;
}

/* Coefficients as used (for the pin tests). order: atanh[4], sin[5], cos[5], ln2, sqrt2 */
void oracle_coefficients(float out[16])
{
    init_coeffs();
    for (int k = 0; k < 4; ++k) out[k] = C_ATANH[k];
    for (int k = 0; k < 5; ++k) out[4 + k] = C_SIN[k];
    for (int k = 0; k < 5; ++k) out[9 + k] = C_COS[k];
    out[14] = LN2_F;
    out[15] = SQRT2_F;
}

/* ln(u1) for u1 = n1 * 2^-24, n1 in [1, 2^24].
 * n1 = 2^e * m with m in [1,2) (exact); if m > sqrt2, m /= 2 and e += 1, so
 * m in (sqrt(1/2), sqrt2].  ln m = 2 atanh(s), s = (m-1)/(m+1), |s| <= 0.1716;
 * atanh(s) = s + s^3/3 + s^5/5 + s^7/7 + s^9/9 + O(s^11) (series truncated
 * where the next term is below 2^-28 relative).  ln u1 = (e-24) ln2 + ln m. */
float oracle_ln_u1(uint32_t n1)
{
    init_coeffs();
    uint32_t fb = f32_bits((float)n1);                       /* exact: n1 <= 2^24 */
    int e = (int)((fb >> 23) & 0xFFu) - 127;                 /* floor(log2 n1) */
    float m = bits_f32((fb & 0x007FFFFFu) | 0x3F800000u);    /* n1 * 2^-e, exact */
    if (m > SQRT2_F) { m = m * 0.5f; e = e + 1; }
    float f = m - 1.0f;                                      /* exact (Sterbenz) */
    float d = 2.0f + f;
    float s = f / d;
    float w = s * s;
    float q = C_ATANH[3];
    q = fmaf(q, w, C_ATANH[2]);
    q = fmaf(q, w, C_ATANH[1]);
    q = fmaf(q, w, C_ATANH[0]);
    float sw = s * w;
    float at = fmaf(sw, q, s);                               /* atanh(s) */
    float lnm = 2.0f * at;
    float k = (float)(e - 24);
    return fmaf(k, LN2_F, lnm);
}

/* sin and cos of the angle 2*pi*b2*2^-24, b2 in [0, 2^24).
 * In turns: t = 4*b2*2^-24, quadrant q = floor(t), f = t - q in [0,1) (exact).
 * With g = f (f <= 1/2) or g = 1 - f (f > 1/2), x = (pi/2) g is in [0, pi/4];
 * sin x and cos x come from their Taylor series in g (odd terms to g^9, even
 * terms to g^10), then the quadrant and the f > 1/2 reflection swap or negate. */
void oracle_sincos_turns(uint32_t b2, float *sn, float *cs)
{
    init_coeffs();
    uint32_t q = (b2 >> 22) & 3u;
    float f = (float)(b2 & 0x3FFFFFu) * 0x1p-22f;            /* exact */
    int refl = f > 0.5f;
    float g = refl ? 1.0f - f : f;                           /* exact */
    float g2 = g * g;
    float ps = C_SIN[4];
    ps = fmaf(ps, g2, C_SIN[3]);
    ps = fmaf(ps, g2, C_SIN[2]);
    ps = fmaf(ps, g2, C_SIN[1]);
    ps = fmaf(ps, g2, C_SIN[0]);
    float sg = g * ps;                                       /* sin((pi/2) g) */
    float pc = C_COS[4];
    pc = fmaf(pc, g2, C_COS[3]);
    pc = fmaf(pc, g2, C_COS[2]);
    pc = fmaf(pc, g2, C_COS[1]);
    pc = fmaf(pc, g2, C_COS[0]);
    float cg = fmaf(g2, pc, 1.0f);                           /* cos((pi/2) g) */
    float s1 = refl ? cg : sg;                               /* sin((pi/2) f) */
    float c1 = refl ? sg : cg;                               /* cos((pi/2) f) */
    switch (q) {
    case 0:  *sn = s1;  *cs = c1;  break;
    case 1:  *sn = c1;  *cs = -s1; break;
    case 2:  *sn = -s1; *cs = -c1; break;
    default: *sn = -c1; *cs = s1;  break;
    }
}

/* ------------------------------------------------------- normal N(0,s^2) - */

/* Box-Muller pair j: u1 = (hi24 + 1) 2^-24 in (0,1], u2 = lo24 2^-24 in [0,1);
 * r = sqrt(-2 ln u1); y0 = sigma (r cos 2 pi u2), y1 = sigma (r sin 2 pi u2). */
void oracle_normal_pair(uint64_t key, uint64_t j, float sigma, float out[2])
{
    uint64_t z = oracle_draw(key, j);
    uint32_t n1 = (uint32_t)(z >> 40) + 1u;
    uint32_t b2 = (uint32_t)((z >> 8) & 0xFFFFFFu);
    float L = oracle_ln_u1(n1);
    float r = sqrtf(-2.0f * L);
    float sn, cs;
    oracle_sincos_turns(b2, &sn, &cs);
    out[0] = sigma * (r * cs);
    out[1] = sigma * (r * sn);
}

float oracle_normal_f32_at(uint64_t key, uint64_t e, float sigma)
{
    float p[2];
    oracle_normal_pair(key, e >> 1, sigma, p);
    return p[e & 1u];
}

/* ------------------------------------------------------- bulk helpers ---- */

/* Row-major rows x cols tensor, element index e = r*cols + c, stored with
 * leading dimension ld (elements). */
void oracle_fill_uniform_bf16(uint64_t seed, uint32_t tensor_id, int64_t rows,
                              int64_t cols, int64_t ld, uint16_t *out)
{
    uint64_t key = oracle_stream_key(seed, tensor_id);
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c)
            out[r * ld + c] = oracle_uniform_bf16_at(key, (uint64_t)(r * cols + c));
}

void oracle_fill_uniform_f16(uint64_t seed, uint32_t tensor_id, int64_t rows,
                             int64_t cols, int64_t ld, uint16_t *out)
{
    uint64_t key = oracle_stream_key(seed, tensor_id);
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c)
            out[r * ld + c] = oracle_uniform_f16_at(key, (uint64_t)(r * cols + c));
}

void oracle_fill_normal_f32(uint64_t seed, uint32_t tensor_id, float sigma,
                            int64_t rows, int64_t cols, int64_t ld, float *out)
{
    uint64_t key = oracle_stream_key(seed, tensor_id);
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c)
            out[r * ld + c] = oracle_normal_f32_at(key, (uint64_t)(r * cols + c), sigma);
}

/* Gather: out[i] = element idx[i] (logical row-major index) of the tensor. */
void oracle_gather_uniform_bf16(uint64_t seed, uint32_t tensor_id,
                                const int64_t *idx, int64_t n, uint16_t *out)
{
    uint64_t key = oracle_stream_key(seed, tensor_id);
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_uniform_bf16_at(key, (uint64_t)idx[i]);
}

void oracle_gather_uniform_f16(uint64_t seed, uint32_t tensor_id,
                               const int64_t *idx, int64_t n, uint16_t *out)
{
    uint64_t key = oracle_stream_key(seed, tensor_id);
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_uniform_f16_at(key, (uint64_t)idx[i]);
}

void oracle_gather_normal_f32(uint64_t seed, uint32_t tensor_id, float sigma,
                              const int64_t *idx, int64_t n, float *out)
{
    uint64_t key = oracle_stream_key(seed, tensor_id);
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_normal_f32_at(key, (uint64_t)idx[i], sigma);
}

/* Vector forms of the fp32 routines, for exhaustive pin tests. */
void oracle_ln_u1_many(const uint32_t *n1, int64_t n, float *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_ln_u1(n1[i]);
}

void oracle_sincos_turns_many(const uint32_t *b2, int64_t n, float *sn, float *cs)
{
    for (int64_t i = 0; i < n; ++i) oracle_sincos_turns(b2[i], &sn[i], &cs[i]);
}

void oracle_draw_many(uint64_t key, uint64_t j0, int64_t n, uint64_t *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_draw(key, j0 + (uint64_t)i);
}
