// K7: the reference GEMM the check compares the candidate against (paper
// Section 2.1: the command checks the candidate against a reference).  CUDA
// cores only (the tcgen05 candidate is the only tensor-core path):
// C[i,j] = sum_k A[i,k] B[k,j] with bf16 inputs widened exactly to fp32,
// fp32 fused multiply-add accumulation in k order, fp32 output.
//
// Classic shared-memory tiling: a 128x128 output tile per 256-thread block,
// 8x8 outputs per thread, K in slices of 16 staged as fp32 (A transposed so a
// thread's 8 rows are one 32-byte read).  Any M, N, K; loads outside the
// matrix read as zero and stores are guarded.
#include "common.cuh"

namespace krex {
namespace {

constexpr int TM = 128, TN = 128, TK = 16, PAD = 4;

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

// 8 consecutive bf16 of row `r` starting at column `c` (zero outside [0,R)x[0,C)).
__device__ __forceinline__ void load8(const uint16_t *__restrict__ p, int64_t ld, int64_t R,
                                      int64_t C, int64_t r, int64_t c, bool vec_ok, float *out) {
    if (r < R && c + 8 <= C && vec_ok) {
        uint4 u = __ldg(reinterpret_cast<const uint4 *>(p + r * ld + c));
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            out[2 * k] = __uint_as_float(w[k] << 16);
            out[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
        }
    } else {
#pragma unroll
        for (int k = 0; k < 8; ++k)
            out[k] = (r < R && c + k < C) ? bf16_to_f32(__ldg(p + r * ld + c + k)) : 0.0f;
    }
}

__global__ void __launch_bounds__(256)
gemm_ref_simt(const uint16_t *__restrict__ A, int64_t lda, const uint16_t *__restrict__ B,
              int64_t ldb, float *__restrict__ C, int64_t ldc, int64_t M, int64_t N, int64_t K,
              bool a_vec, bool b_vec, bool c_vec) {
    __shared__ __align__(16) float As[TK][TM + PAD];  // As[k][m]
    __shared__ __align__(16) float Bs[TK][TN + PAD];  // Bs[k][n]
    const int t = threadIdx.x;
    const int tx = t & 15, ty = t >> 4;
    const int64_t m0 = (int64_t)blockIdx.y * TM, n0 = (int64_t)blockIdx.x * TN;

    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;

    // this thread's load slots: A row (t>>1), k half (t&1)*8; B k-row (t>>4), n chunk (t&15)*8
    const int a_row = t >> 1, a_k = (t & 1) * 8;
    const int b_k = t >> 4, b_n = (t & 15) * 8;

    for (int64_t k0 = 0; k0 < K; k0 += TK) {
        float av[8], bv[8];
        load8(A, lda, M, K, m0 + a_row, k0 + a_k, a_vec, av);
        load8(B, ldb, K, N, k0 + b_k, n0 + b_n, b_vec, bv);
#pragma unroll
        for (int i = 0; i < 8; ++i) As[a_k + i][a_row] = av[i];
        *reinterpret_cast<float4 *>(&Bs[b_k][b_n]) = make_float4(bv[0], bv[1], bv[2], bv[3]);
        *reinterpret_cast<float4 *>(&Bs[b_k][b_n + 4]) = make_float4(bv[4], bv[5], bv[6], bv[7]);
        __syncthreads();
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            float4 a0 = *reinterpret_cast<const float4 *>(&As[k][ty * 8]);
            float4 a1 = *reinterpret_cast<const float4 *>(&As[k][ty * 8 + 4]);
            float4 b0 = *reinterpret_cast<const float4 *>(&Bs[k][tx * 8]);
            float4 b1 = *reinterpret_cast<const float4 *>(&Bs[k][tx * 8 + 4]);
            const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }

#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t r = m0 + ty * 8 + i;
        if (r >= M) continue;
        const int64_t c = n0 + tx * 8;
        float *cr = C + r * ldc;
        if (c_vec && c + 8 <= N) {
            *reinterpret_cast<float4 *>(cr + c) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
            *reinterpret_cast<float4 *>(cr + c + 4) = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (c + j < N) cr[c + j] = acc[i][j];
        }
    }
}

}  // namespace

cudaError_t launch_gemm_ref(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb,
                            float *c, int64_t ldc, int64_t M, int64_t N, int64_t K,
                            cudaStream_t s) {
    if (M == 0 || N == 0) return cudaSuccess;
    const bool a_vec = ((reinterpret_cast<uintptr_t>(a) & 15u) == 0) && (lda % 8 == 0);
    const bool b_vec = ((reinterpret_cast<uintptr_t>(b) & 15u) == 0) && (ldb % 8 == 0);
    const bool c_vec = ((reinterpret_cast<uintptr_t>(c) & 15u) == 0) && (ldc % 4 == 0);
    dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
    gemm_ref_simt<<<grid, 256, 0, s>>>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec);
    return cudaGetLastError();
}

}  // namespace krex
