// K1 / K2: seeded input generation on the GPU (paper Section 2.1: a
// benchmarking command generates its inputs before the check and the timed
// loop).  Counter-based SplitMix64, so any element can be produced by any
// thread: the output is bit-identical for every launch shape.
//
//   draw j of a stream   z_j = mix64(key + (j+1) * G)
//   uniform element e    bits 63..40 (e even) / 31..8 (e odd) of z_{e/2},
//                        x = (b - 2^23) 2^-23 (exact), bf16 = RNE(x)
//                        (fp16 operands: binary16 = RNE(x))
//   normal pair j        u1 = (hi24 + 1) 2^-24, u2 = lo24 2^-24,
//                        (y0, y1) = sigma * sqrt(-2 ln u1) * (cos, sin)(2 pi u2)
//
// The fp32 ln and sincos are this file's own series evaluations (atanh series
// for ln, Taylor series in quarter turns for sin/cos), written operation by
// operation with explicit round-to-nearest intrinsics so no contraction or
// approximate instruction changes a bit.  Coefficients are the fp32 roundings
// of 1/(2k+1) and (pi/2)^n / n!.
//
// Layout: one thread writes 16 bytes per step (8 bf16 = 4 draws, or 4 fp32 =
// 2 Box-Muller pairs); rows of a strided buffer are handled by a 2-D grid.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "common.cuh"

namespace krex {
namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// ---------------------------------------------------------------- uniform --

// Draw j's two 24-bit fields, each in bits 31..8 of a word with the low byte
// clear: bits 63..40 of z_j (element 2j) and bits 31..8 (element 2j+1), from
// the draw's state s = key + (j+1) G.  The last step of mix64 (z ^= z >> 31)
// changes only bit 0 of the high word, and xors the high word shifted left by
// one (plus one bit into bit 0) into the low word; so bits 31..8 of the final
// words are those of hi and of lo ^ (hi << 1) before that step.
__device__ __forceinline__ void draw_fields(uint64_t s, uint32_t &wh, uint32_t &wl) {
    uint64_t z = (s ^ (s >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    const uint32_t hi = (uint32_t)(z >> 32), lo = (uint32_t)z;
    wh = hi & 0xFFFFFF00u;
    wl = (lo ^ (hi << 1)) & 0xFFFFFF00u;
}

// A field w = b 2^8 (b its 24-bit value) -> (b - 2^23) 2^-23, exactly: w
// converts to fp32 without rounding (24 significant bits), and w 2^-31 - 1 =
// (b - 2^23) 2^-23 is representable, so the fused multiply-add is exact.
__device__ __forceinline__ float field_to_pm1(uint32_t w) {
    return __fmaf_rn(__uint2float_rn(w), 0x1p-31f, -1.0f);
}

// Elements 2j (low half) and 2j+1 (high half) from the state of draw j,
// rounded to bf16 or (F16) to IEEE binary16, both round-to-nearest-even.
template <bool F16>
__device__ __forceinline__ uint32_t uniform_16x2(uint64_t s) {
    uint32_t wh, wl;
    draw_fields(s, wh, wl);
    const float x0 = field_to_pm1(wh), x1 = field_to_pm1(wl);
    if constexpr (F16) {
        __half2 h = __floats2half2_rn(x0, x1);
        return *reinterpret_cast<uint32_t *>(&h);
    } else {
        __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
        return *reinterpret_cast<uint32_t *>(&h);
    }
}

template <bool F16>
__device__ __forceinline__ uint16_t uniform_16_at(uint64_t key, uint64_t e) {
    uint32_t p = uniform_16x2<F16>(key + ((e >> 1) + 1ull) * kGamma);
    return (uint16_t)((e & 1ull) ? (p >> 16) : (p & 0xFFFFu));
}

// Contiguous rows (ld == cols) are treated as one row of rows*cols elements.
// Vector path: cols % 8 == 0 within each row of a strided buffer, or any
// length for a contiguous buffer (the scalar tail is done by thread 0).
template <bool F16>
__global__ void __launch_bounds__(256)
fill_uniform_16_vec(uint64_t key, uint16_t *__restrict__ out, int64_t rows, int64_t cols,
                    int64_t ld) {
    const int64_t groups = cols >> 3;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t r = blockIdx.y; r < rows; r += gridDim.y) {
        uint16_t *row = out + r * ld;
        const uint64_t e_row = (uint64_t)(r * cols);
        for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups; g += stride) {
            uint64_t s = key + (((e_row + (uint64_t)(g << 3)) >> 1) + 1ull) * kGamma;
            uint4 v;
            v.x = uniform_16x2<F16>(s);
            s += kGamma;
            v.y = uniform_16x2<F16>(s);
            s += kGamma;
            v.z = uniform_16x2<F16>(s);
            s += kGamma;
            v.w = uniform_16x2<F16>(s);
            *reinterpret_cast<uint4 *>(row + (g << 3)) = v;
        }
        if (blockIdx.x == 0 && threadIdx.x == 0) {
            for (int64_t c = groups << 3; c < cols; ++c)
                row[c] = uniform_16_at<F16>(key, e_row + (uint64_t)c);
        }
    }
}

// ----------------------------------------------------------------- normal --

constexpr float kAt3 = 0x1.555556p-2f;   // 1/3
constexpr float kAt5 = 0x1.99999ap-3f;   // 1/5
constexpr float kAt7 = 0x1.24924ap-3f;   // 1/7
constexpr float kAt9 = 0x1.c71c72p-4f;   // 1/9
constexpr float kS1 = 0x1.921fb6p+0f;    //  (pi/2)^1 / 1!
constexpr float kS3 = -0x1.4abbcep-1f;   // -(pi/2)^3 / 3!
constexpr float kS5 = 0x1.466bc6p-4f;    //  (pi/2)^5 / 5!
constexpr float kS7 = -0x1.32d2ccp-8f;   // -(pi/2)^7 / 7!
constexpr float kS9 = 0x1.507834p-13f;   //  (pi/2)^9 / 9!
constexpr float kC2 = -0x1.3bd3ccp+0f;   // -(pi/2)^2 / 2!
constexpr float kC4 = 0x1.03c1f0p-2f;    //  (pi/2)^4 / 4!
constexpr float kC6 = -0x1.55d3c8p-6f;   // -(pi/2)^6 / 6!
constexpr float kC8 = 0x1.e1f506p-11f;   //  (pi/2)^8 / 8!
constexpr float kC10 = -0x1.a6d1f2p-16f; // -(pi/2)^10 / 10!
constexpr float kLn2 = 0x1.62e430p-1f;   // ln 2
constexpr float kSqrt2 = 0x1.6a09e6p+0f; // sqrt 2

// ln(n1 * 2^-24) for n1 in [1, 2^24]: n1 = 2^e m, m in (sqrt(1/2), sqrt 2],
// ln m = 2 atanh((m-1)/(m+1)) by its series to s^9.
__device__ __forceinline__ float ln_u1(uint32_t n1) {
    uint32_t fb = __float_as_uint(__uint2float_rn(n1));  // exact
    int e = (int)((fb >> 23) & 0xFFu) - 127;
    float m = __uint_as_float((fb & 0x007FFFFFu) | 0x3F800000u);
    if (m > kSqrt2) {
        m = __fmul_rn(m, 0.5f);
        e += 1;
    }
    float f = __fsub_rn(m, 1.0f);
    float d = __fadd_rn(2.0f, f);
    float s = __fdiv_rn(f, d);
    float w = __fmul_rn(s, s);
    float q = kAt9;
    q = __fmaf_rn(q, w, kAt7);
    q = __fmaf_rn(q, w, kAt5);
    q = __fmaf_rn(q, w, kAt3);
    float sw = __fmul_rn(s, w);
    float at = __fmaf_rn(sw, q, s);
    float lnm = __fmul_rn(2.0f, at);
    float k = __int2float_rn(e - 24);
    return __fmaf_rn(k, kLn2, lnm);
}

// sin and cos of 2 pi b2 2^-24 evaluated in quarter turns.
__device__ __forceinline__ void sincos_turns(uint32_t b2, float &sn, float &cs) {
    uint32_t q = (b2 >> 22) & 3u;
    float f = __fmul_rn(__uint2float_rn(b2 & 0x3FFFFFu), 0x1p-22f);  // exact
    bool refl = f > 0.5f;
    float g = refl ? __fsub_rn(1.0f, f) : f;
    float g2 = __fmul_rn(g, g);
    float ps = kS9;
    ps = __fmaf_rn(ps, g2, kS7);
    ps = __fmaf_rn(ps, g2, kS5);
    ps = __fmaf_rn(ps, g2, kS3);
    ps = __fmaf_rn(ps, g2, kS1);
    float sg = __fmul_rn(g, ps);
    float pc = kC10;
    pc = __fmaf_rn(pc, g2, kC8);
    pc = __fmaf_rn(pc, g2, kC6);
    pc = __fmaf_rn(pc, g2, kC4);
    pc = __fmaf_rn(pc, g2, kC2);
    float cg = __fmaf_rn(g2, pc, 1.0f);
    float s1 = refl ? cg : sg;
    float c1 = refl ? sg : cg;
    switch (q) {
    case 0: sn = s1; cs = c1; break;
    case 1: sn = c1; cs = -s1; break;
    case 2: sn = -s1; cs = -c1; break;
    default: sn = -c1; cs = s1; break;
    }
}

__device__ __forceinline__ float2 normal_pair(uint64_t z, float sigma) {
    uint32_t hi = (uint32_t)(z >> 32), lo = (uint32_t)z;
    float L = ln_u1((hi >> 8) + 1u);
    float r = __fsqrt_rn(__fmul_rn(-2.0f, L));
    float sn, cs;
    sincos_turns(lo >> 8, sn, cs);
    return make_float2(__fmul_rn(sigma, __fmul_rn(r, cs)), __fmul_rn(sigma, __fmul_rn(r, sn)));
}

__global__ void __launch_bounds__(256)
fill_normal_f32_vec(uint64_t key, float sigma, float *__restrict__ out, int64_t rows,
                    int64_t cols, int64_t ld) {
    const int64_t groups = cols >> 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t r = blockIdx.y; r < rows; r += gridDim.y) {
        float *row = out + r * ld;
        const uint64_t e_row = (uint64_t)(r * cols);
        for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups; g += stride) {
            uint64_t s = key + (((e_row + (uint64_t)(g << 2)) >> 1) + 1ull) * kGamma;
            float2 p0 = normal_pair(mix64(s), sigma);
            float2 p1 = normal_pair(mix64(s + kGamma), sigma);
            *reinterpret_cast<float4 *>(row + (g << 2)) = make_float4(p0.x, p0.y, p1.x, p1.y);
        }
        if (blockIdx.x == 0 && threadIdx.x == 0) {
            for (int64_t c = groups << 2; c < cols; ++c) {
                uint64_t e = e_row + (uint64_t)c;
                float2 p = normal_pair(mix64(key + ((e >> 1) + 1ull) * kGamma), sigma);
                row[c] = (e & 1ull) ? p.y : p.x;
            }
        }
    }
}

// Measurement probe: each fill kernel's loop (the same grid-stride walk over
// 16-byte groups of a contiguous buffer of n elements, the same per-draw device
// functions) with every group folded into one word instead of stored, to
// measure the rate at which this GPU computes the generator: the fills'
// compute ceiling.  The fold is stored only if it equals a value no run
// produces in practice (it keeps the arithmetic live; `sink` must hold one
// word per thread anyway).
template <int DIST>
__global__ void __launch_bounds__(256)
generator_probe(uint64_t key, int64_t n, float sigma, uint32_t *sink) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    uint32_t acc = 0;
    if constexpr (DIST == KREX_DIST_UNIFORM_PM1) {
        for (int64_t g = t; g < (n >> 3); g += stride) {
            uint64_t s = key + (((uint64_t)(g << 3) >> 1) + 1ull) * kGamma;
            uint32_t v = uniform_16x2<false>(s);
            s += kGamma;
            v ^= uniform_16x2<false>(s);
            s += kGamma;
            v ^= uniform_16x2<false>(s);
            s += kGamma;
            v ^= uniform_16x2<false>(s);
            acc ^= v;
        }
    } else {
        for (int64_t g = t; g < (n >> 2); g += stride) {
            uint64_t s = key + (((uint64_t)(g << 2) >> 1) + 1ull) * kGamma;
            float2 p0 = normal_pair(mix64(s), sigma);
            float2 p1 = normal_pair(mix64(s + kGamma), sigma);
            acc ^= __float_as_uint(p0.x) ^ __float_as_uint(p0.y) ^ __float_as_uint(p1.x) ^ __float_as_uint(p1.y);
        }
    }
    if (acc == 0x5EED5EEDu) sink[t] = acc;
}

// Any layout: one element per thread step (each element recomputes its draw).
template <bool F16>
__global__ void __launch_bounds__(256)
fill_uniform_16_scalar(uint64_t key, uint16_t *__restrict__ out, int64_t rows, int64_t cols,
                       int64_t ld) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t r = blockIdx.y; r < rows; r += gridDim.y)
        for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < cols; c += stride)
            out[r * ld + c] = uniform_16_at<F16>(key, (uint64_t)(r * cols + c));
}

__global__ void __launch_bounds__(256)
fill_normal_f32_scalar(uint64_t key, float sigma, float *__restrict__ out, int64_t rows,
                       int64_t cols, int64_t ld) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t r = blockIdx.y; r < rows; r += gridDim.y)
        for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < cols; c += stride) {
            uint64_t e = (uint64_t)(r * cols + c);
            float2 p = normal_pair(mix64(key + ((e >> 1) + 1ull) * kGamma), sigma);
            out[r * ld + c] = (e & 1ull) ? p.y : p.x;
        }
}

// Grid: enough blocks to cover the vector groups of one (logical) row, capped
// at a few waves of resident blocks; rows go to gridDim.y (capped at 65535,
// grid-stride beyond).
dim3 fill_grid(int64_t rows, int64_t per_row_items) {
    int64_t cap = (int64_t)sm_count() * 8;
    int64_t bx = (per_row_items + 255) / 256;
    int64_t by = rows < 65535 ? rows : 65535;
    if (bx < 1) bx = 1;
    if (by < 1) by = 1;
    // total blocks ~ cap: split between x and y
    if (bx * by > cap) {
        if (by >= cap) {
            by = cap;
            bx = 1;
        } else {
            bx = (cap + by - 1) / by;
        }
    }
    return dim3((unsigned)bx, (unsigned)by, 1);
}

template <bool F16>
void launch_uniform(uint64_t key, uint16_t *p, bool aligned, int64_t rows, int64_t cols, int64_t ld,
                    cudaStream_t s) {
    if (aligned && ld == cols) {
        // one logical row of rows*cols elements
        int64_t n = rows * cols;
        fill_uniform_16_vec<F16><<<fill_grid(1, n >> 3), 256, 0, s>>>(key, p, 1, n, n);
    } else if (aligned && (cols & 7) == 0 && (ld & 7) == 0) {
        fill_uniform_16_vec<F16><<<fill_grid(rows, cols >> 3), 256, 0, s>>>(key, p, rows, cols, ld);
    } else {
        fill_uniform_16_scalar<F16><<<fill_grid(rows, cols), 256, 0, s>>>(key, p, rows, cols, ld);
    }
}

}  // namespace

cudaError_t launch_generator_probe(int32_t dist, uint64_t key, int64_t n, float sigma, int blocks, uint32_t *sink,
                                   cudaStream_t s) {
    if (dist == KREX_DIST_UNIFORM_PM1)
        generator_probe<KREX_DIST_UNIFORM_PM1><<<blocks, 256, 0, s>>>(key, n, sigma, sink);
    else
        generator_probe<KREX_DIST_NORMAL><<<blocks, 256, 0, s>>>(key, n, sigma, sink);
    return cudaGetLastError();
}

cudaError_t launch_fill_uniform_16(uint64_t key, bool f16, void *out, int64_t rows, int64_t cols,
                                   int64_t ld, cudaStream_t s) {
    if (rows == 0 || cols == 0) return cudaSuccess;
    uint16_t *p = static_cast<uint16_t *>(out);
    bool aligned = (reinterpret_cast<uintptr_t>(out) & 15u) == 0;
    if (f16)
        launch_uniform<true>(key, p, aligned, rows, cols, ld, s);
    else
        launch_uniform<false>(key, p, aligned, rows, cols, ld, s);
    return cudaGetLastError();
}

cudaError_t launch_fill_normal_f32(uint64_t key, float sigma, float *out, int64_t rows,
                                   int64_t cols, int64_t ld, cudaStream_t s) {
    if (rows == 0 || cols == 0) return cudaSuccess;
    bool aligned = (reinterpret_cast<uintptr_t>(out) & 15u) == 0;
    if (aligned && ld == cols) {
        int64_t n = rows * cols;
        fill_normal_f32_vec<<<fill_grid(1, n >> 2), 256, 0, s>>>(key, sigma, out, 1, n, n);
    } else if (aligned && (cols & 3) == 0 && (ld & 3) == 0) {
        fill_normal_f32_vec<<<fill_grid(rows, cols >> 2), 256, 0, s>>>(key, sigma, out, rows, cols, ld);
    } else {
        fill_normal_f32_scalar<<<fill_grid(rows, cols), 256, 0, s>>>(key, sigma, out, rows, cols, ld);
    }
    return cudaGetLastError();
}

}  // namespace krex
