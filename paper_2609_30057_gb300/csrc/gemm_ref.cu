// K7: the reference GEMM the check compares the candidate against (paper
// Section 2.1: the command checks the candidate against a reference).  CUDA
// cores only (the tcgen05 candidate is the only tensor-core path):
// C[i,j] = sum_k A[i,k] B[k,j] with bf16 (or binary16) inputs widened exactly to fp32,
// fp32 fused multiply-add accumulation in k order, fp32 output.
//
// Shared-memory tiling on the FP32 pipe: a 128x128 output tile per 256-thread
// block, K in slices of 16 staged as fp32 in two shared-memory buffers (the
// next slice is fetched from global memory into registers while the current
// one is multiplied).  Each thread owns an 8x8 block made of the four 4x4
// blocks at rows {ty*4, 64+ty*4} x cols {tx*4, 64+tx*4}, so its per-k operand
// reads are four conflict-free 16-byte shared loads for 64 FMAs.  Any M, N, K;
// loads outside the matrix read as zero and stores are guarded.
#include <cuda_fp16.h>

#include "common.cuh"

namespace krex {
namespace {

constexpr int TM = 128, TN = 128, TK = 16;

// 8 consecutive bf16 at (r, c..c+7) of a row-major matrix as raw 16-bit words
// packed in a uint4, zero outside [0,R)x[0,C).
__device__ __forceinline__ uint4 load8(const uint16_t *__restrict__ p, int64_t ld, int64_t R, int64_t C, int64_t r,
                                       int64_t c, bool vec_ok) {
    if (vec_ok && r < R && c + 8 <= C) return __ldg(reinterpret_cast<const uint4 *>(p + r * ld + c));
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t lo = (r < R && c + 2 * i < C) ? __ldg(p + r * ld + c + 2 * i) : 0u;
        const uint32_t hi = (r < R && c + 2 * i + 1 < C) ? __ldg(p + r * ld + c + 2 * i + 1) : 0u;
        w[i] = lo | (hi << 16);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// Exact widening of the low / high 16-bit element of a word: bf16 is the top
// half of an fp32; binary16 goes through the hardware conversion (exact).
template <bool F16>
__device__ __forceinline__ float lo_f32(uint32_t w) {
    if constexpr (F16) return __half2float(__ushort_as_half((unsigned short)(w & 0xFFFFu)));
    return __uint_as_float(w << 16);
}
template <bool F16>
__device__ __forceinline__ float hi_f32(uint32_t w) {
    if constexpr (F16) return __half2float(__ushort_as_half((unsigned short)(w >> 16)));
    return __uint_as_float(w & 0xFFFF0000u);
}

template <bool F16>
__global__ void __launch_bounds__(256)
gemm_ref_simt(const uint16_t *__restrict__ A, int64_t lda, const uint16_t *__restrict__ B, int64_t ldb,
              float *__restrict__ C, int64_t ldc, int64_t M, int64_t N, int64_t K, bool a_vec, bool b_vec,
              bool c_vec) {
    __shared__ __align__(16) float As[2][TK][TM];  // As[buf][k][m]
    __shared__ __align__(16) float Bs[2][TK][TN];  // Bs[buf][k][n]
    const int t = threadIdx.x;
    const int tx = t & 15, ty = t >> 4;
    const int64_t m0 = (int64_t)blockIdx.y * TM, n0 = (int64_t)blockIdx.x * TN;
    // load slots: A row t/2, k (t&1)*8..+7; B k-row t/16, cols (t&15)*8..+7
    const int a_row = t >> 1, a_k = (t & 1) * 8;
    const int b_k = t >> 4, b_n = (t & 15) * 8;
    auto stage = [&](int nb, const uint4 &ua, const uint4 &ub) {
        const uint32_t wa[4] = {ua.x, ua.y, ua.z, ua.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            As[nb][a_k + 2 * i][a_row] = lo_f32<F16>(wa[i]);
            As[nb][a_k + 2 * i + 1][a_row] = hi_f32<F16>(wa[i]);
        }
        *reinterpret_cast<float4 *>(&Bs[nb][b_k][b_n]) =
            make_float4(lo_f32<F16>(ub.x), hi_f32<F16>(ub.x), lo_f32<F16>(ub.y), hi_f32<F16>(ub.y));
        *reinterpret_cast<float4 *>(&Bs[nb][b_k][b_n + 4]) =
            make_float4(lo_f32<F16>(ub.z), hi_f32<F16>(ub.z), lo_f32<F16>(ub.w), hi_f32<F16>(ub.w));
    };

    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;

    uint4 ua = load8(A, lda, M, K, m0 + a_row, a_k, a_vec);
    uint4 ub = load8(B, ldb, K, N, b_k, n0 + b_n, b_vec);
    stage(0, ua, ub);
    __syncthreads();

    int buf = 0;
    for (int64_t k0 = 0; k0 < K; k0 += TK) {
        const bool more = k0 + TK < K;
        if (more) {  // fetch the next slice while this one is multiplied
            ua = load8(A, lda, M, K, m0 + a_row, k0 + TK + a_k, a_vec);
            ub = load8(B, ldb, K, N, k0 + TK + b_k, n0 + b_n, b_vec);
        }
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            const float4 a0 = *reinterpret_cast<const float4 *>(&As[buf][k][ty * 4]);
            const float4 a1 = *reinterpret_cast<const float4 *>(&As[buf][k][64 + ty * 4]);
            const float4 b0 = *reinterpret_cast<const float4 *>(&Bs[buf][k][tx * 4]);
            const float4 b1 = *reinterpret_cast<const float4 *>(&Bs[buf][k][64 + tx * 4]);
            const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        if (more) {
            const int nb = buf ^ 1;
            stage(nb, ua, ub);
            __syncthreads();
            buf = nb;
        }
    }

#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t r = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
        if (r >= M) continue;
        float *cr = C + r * ldc;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int64_t c = n0 + h * 64 + tx * 4;
            const float *v = &acc[i][4 * h];
            if (c_vec && c + 4 <= N) {
                *reinterpret_cast<float4 *>(cr + c) = make_float4(v[0], v[1], v[2], v[3]);
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (c + j < N) cr[c + j] = v[j];
            }
        }
    }
}

}  // namespace

cudaError_t launch_gemm_ref(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb, float *c, int64_t ldc,
                            int64_t M, int64_t N, int64_t K, bool f16, cudaStream_t s) {
    if (M == 0 || N == 0) return cudaSuccess;
    const bool a_vec = ((reinterpret_cast<uintptr_t>(a) & 15u) == 0) && (lda % 8 == 0);
    const bool b_vec = ((reinterpret_cast<uintptr_t>(b) & 15u) == 0) && (ldb % 8 == 0);
    const bool c_vec = ((reinterpret_cast<uintptr_t>(c) & 15u) == 0) && (ldc % 4 == 0);
    dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
    if (f16)
        gemm_ref_simt<true><<<grid, 256, 0, s>>>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec);
    else
        gemm_ref_simt<false><<<grid, 256, 0, s>>>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec);
    return cudaGetLastError();
}

}  // namespace krex
