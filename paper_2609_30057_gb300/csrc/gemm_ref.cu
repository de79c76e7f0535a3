// K7: the reference GEMM the check compares the candidate against (paper
// Section 2.1: the command checks the candidate against a reference).  CUDA
// cores only (the tcgen05 candidate is the only tensor-core path):
// C[i,j] = sum_k A[i,k] B[k,j] with bf16 (or binary16) inputs widened exactly to fp32,
// fp32 fused multiply-add accumulation in k order, fp32 output.
//
// Shared-memory tiling on the FP32 pipe: a 128 x (64*NG) output tile per
// 256-thread block, K in slices of TK staged as fp32 in two shared-memory
// buffers (the next slice is fetched from global memory into registers while
// the current one is multiplied).  Each thread owns an 8 x (4*NG) block made
// of 4x4 blocks at rows {ty*4, 64+ty*4} x cols {g*64 + tx*4 : g < NG}, so its
// per-k operand reads are conflict-free 16-byte shared loads (two for A, NG
// for B) for 32*NG FMAs.  Any M, N, K; loads outside the matrix read as zero
// and stores are guarded.  GEMMs of a few tiles use a one-output-per-thread
// kernel instead, with the same k-order chains (identical bits).
#include <cuda_fp16.h>

#include "common.cuh"

namespace krex {
namespace {

constexpr int TM = 128;

// 8 consecutive 16-bit elements at (r, c..c+7) of a row-major matrix as raw
// words packed in a uint4, zero outside [0,R)x[0,C).
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

// NG: 64-column groups per block (tile 128 x 64*NG); TK: K per shared slice;
// MINB: resident blocks per SM the register budget is sized for.  Any shape
// and row strides (bounds-checked loads and stores).
template <bool F16, int NG, int TK, int MINB>
__global__ void __launch_bounds__(256, MINB)
gemm_ref_simt(const uint16_t *__restrict__ A, int64_t lda, const uint16_t *__restrict__ B, int64_t ldb,
              float *__restrict__ C, int64_t ldc, int64_t M, int64_t N, int64_t K, bool a_vec, bool b_vec,
              bool c_vec) {
    constexpr int TN = 64 * NG;
    constexpr int A_LOADS = TM * TK / 8 / 256;  // uint4 (8 elements) per thread and slice
    constexpr int B_LOADS = TK * TN / 8 / 256;
    static_assert(A_LOADS >= 1 && B_LOADS >= 1, "slice too small for 256 threads");
    extern __shared__ __align__(16) float smem[];
    float *As = smem;                  // [2][TK][TM]
    float *Bs = smem + 2 * TK * TM;    // [2][TK][TN]
    const int t = threadIdx.x;
    const int tx = t & 15, ty = t >> 4;
    const int64_t m0 = (int64_t)blockIdx.y * TM, n0 = (int64_t)blockIdx.x * TN;
    // load slots s = t + 256 i: A row s / (TK/8), k offset 8 (s % (TK/8));
    //                           B k-row s / (TN/8), cols 8 (s % (TN/8))
    uint4 ua[A_LOADS], ub[B_LOADS];
    auto fetch = [&](int64_t k0) {
#pragma unroll
        for (int i = 0; i < A_LOADS; ++i) {
            const int s = t + 256 * i;
            ua[i] = load8(A, lda, M, K, m0 + s / (TK / 8), k0 + 8 * (s % (TK / 8)), a_vec);
        }
#pragma unroll
        for (int i = 0; i < B_LOADS; ++i) {
            const int s = t + 256 * i;
            ub[i] = load8(B, ldb, K, N, k0 + s / (TN / 8), n0 + 8 * (s % (TN / 8)), b_vec);
        }
    };
    auto stage = [&](int nb) {
        float *as = As + nb * TK * TM;
        float *bs = Bs + nb * TK * TN;
#pragma unroll
        for (int i = 0; i < A_LOADS; ++i) {
            const int s = t + 256 * i;
            const int row = s / (TK / 8), kk = 8 * (s % (TK / 8));
            const uint32_t wa[4] = {ua[i].x, ua[i].y, ua[i].z, ua[i].w};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                as[(kk + 2 * j) * TM + row] = lo_f32<F16>(wa[j]);
                as[(kk + 2 * j + 1) * TM + row] = hi_f32<F16>(wa[j]);
            }
        }
#pragma unroll
        for (int i = 0; i < B_LOADS; ++i) {
            const int s = t + 256 * i;
            const int kr = s / (TN / 8), col = 8 * (s % (TN / 8));
            float *dst = bs + kr * TN + col;
            *reinterpret_cast<float4 *>(dst) =
                make_float4(lo_f32<F16>(ub[i].x), hi_f32<F16>(ub[i].x), lo_f32<F16>(ub[i].y), hi_f32<F16>(ub[i].y));
            *reinterpret_cast<float4 *>(dst + 4) =
                make_float4(lo_f32<F16>(ub[i].z), hi_f32<F16>(ub[i].z), lo_f32<F16>(ub[i].w), hi_f32<F16>(ub[i].w));
        }
    };

    float acc[8][4 * NG];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4 * NG; ++j) acc[i][j] = 0.0f;

    fetch(0);
    stage(0);
    __syncthreads();

    int buf = 0;
    for (int64_t k0 = 0; k0 < K; k0 += TK) {
        const bool more = k0 + TK < K;
        if (more) fetch(k0 + TK);  // the next slice comes in while this one is multiplied
        const float *as = As + buf * TK * TM;
        const float *bs = Bs + buf * TK * TN;
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            const float4 a0 = *reinterpret_cast<const float4 *>(as + k * TM + ty * 4);
            const float4 a1 = *reinterpret_cast<const float4 *>(as + k * TM + 64 + ty * 4);
            float b[4 * NG];
#pragma unroll
            for (int g = 0; g < NG; ++g) {
                const float4 bg = *reinterpret_cast<const float4 *>(bs + k * TN + g * 64 + tx * 4);
                b[4 * g] = bg.x;
                b[4 * g + 1] = bg.y;
                b[4 * g + 2] = bg.z;
                b[4 * g + 3] = bg.w;
            }
            const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 4 * NG; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        if (more) {
            const int nb = buf ^ 1;
            stage(nb);
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
        for (int g = 0; g < NG; ++g) {
            const int64_t c = n0 + g * 64 + tx * 4;
            const float *v = &acc[i][4 * g];
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

// The same tiling for GEMMs made of whole tiles (M % 128 = N % 128 = K % 16 =
// 0, 16-byte aligned rows), the sizes of the benchmark workloads.  Operands
// stay 16-bit in shared memory (the A slice transposed to k-major, the B
// slice as loaded), and the outer product uses the mixed-precision FMA
// (fma.rn.f32.bf16 / .f16: 16-bit a and b, fp32 c and d), which widens both
// factors exactly and rounds once like fmaf on the widened values: each
// output is the same k-order FMA chain as in gemm_ref_simt (identical bits),
// with half the shared-memory traffic and fragment registers and no
// conversion in the slice staging.  No bounds checks, one 16-byte load of A
// and one of B per thread and slice, a 32-bit K loop.  Each thread owns 8
// consecutive rows x 8 consecutive columns, so its per-k operands are one
// 16-byte shared load of A (two distinct addresses per warp) and one of B
// (256 contiguous bytes per warp), swept column by column.  Measured on GB300
// in one process (TFLOP/s at 4096^3 / 16384^3, L2 flushed): 65.5 / 68.7,
// against 64.3 / 67.4 with the 4x4-block ownership of gemm_ref_simt (two
// 8-byte loads of each operand per k), 58.8 / 60.4 with operands widened to
// fp32 in shared memory and 55.0 / 57.0 for gemm_ref_simt.  Also measured and
// dropped here: 128x256 and 256x128 tiles with 8x16 / 16x8 outputs per thread
// (one block per SM: 52-55 / 61-65), 32-deep slices (58-60 / 61-64), raster
// groups of 8 or 32 rows (no change), and the slices brought in by TMA
// through an mbarrier ring with operand rows kept m-major (no block barrier,
// no staging: 53 / 56).
template <bool F16>
__device__ __forceinline__ void fma_mixed(float &acc, unsigned short a, unsigned short b) {
    if constexpr (F16) asm("fma.rn.f32.f16 %0, %1, %2, %0;" : "+f"(acc) : "h"(a), "h"(b));
    else asm("fma.rn.f32.bf16 %0, %1, %2, %0;" : "+f"(acc) : "h"(a), "h"(b));
}
__device__ __forceinline__ void halves(uint32_t w, unsigned short &lo, unsigned short &hi) {
    asm("mov.b32 {%0, %1}, %2;" : "=h"(lo), "=h"(hi) : "r"(w));
}

// Tile rows per raster group of gemm_ref_whole.  Measured on GB300 at 16384^3:
// DRAM reads per launch 65.9 GB with plain row-major block order, 12.3 GB
// with groups of 16 rows, at the same speed (the kernel is bound by the FMA
// pipe; 4, 8, 16 and 32 rows all ran 67.6 TFLOP/s).
constexpr int kRefGroup = 16;

template <bool F16>
__global__ void __launch_bounds__(256, 2)
gemm_ref_whole(const uint16_t *__restrict__ A, int64_t lda, const uint16_t *__restrict__ B, int64_t ldb,
               float *__restrict__ C, int64_t ldc, int K, int tiles_m, int tiles_n) {
    constexpr int TK = 16, TN = 128;
    __shared__ __align__(16) uint16_t As[2][TK][TM];   // k-major
    __shared__ __align__(16) uint16_t Bs[2][TK][TN];
    const int t = threadIdx.x, tx = t & 15, ty = t >> 4;
    // grouped raster: blocks in launch order cover kRefGroup tile rows at a
    // time, column by column, so a wave of resident blocks (2 per SM) touches
    // kRefGroup A strips and about 19 B strips instead of every B strip
    int mb, nb;
    {
        const int b = blockIdx.x, per_group = kRefGroup * tiles_n, g = b / per_group, first = g * kRefGroup;
        const int gsize = min(tiles_m - first, kRefGroup), in_g = b - g * per_group;
        mb = first + in_g % gsize;
        nb = in_g / gsize;
    }
    const int64_t m0 = (int64_t)mb * TM, n0 = (int64_t)nb * TN;
    // one 16-byte load of A (row t / 2, k offset 8 (t % 2)) and one of B
    // (k-row t / 16, columns 8 (t % 16)) per thread and slice
    uint4 ua, ub;
    auto fetch = [&](int k0) {
        ua = __ldg(reinterpret_cast<const uint4 *>(A + (m0 + (t >> 1)) * lda + k0 + 8 * (t & 1)));
        ub = __ldg(reinterpret_cast<const uint4 *>(B + (int64_t)(k0 + (t >> 4)) * ldb + n0 + 8 * (t & 15)));
    };
    auto stage = [&](int nb) {
        const int row = t >> 1, kk = 8 * (t & 1);
        const uint32_t wa[4] = {ua.x, ua.y, ua.z, ua.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            As[nb][kk + 2 * j][row] = (uint16_t)(wa[j] & 0xFFFFu);
            As[nb][kk + 2 * j + 1][row] = (uint16_t)(wa[j] >> 16);
        }
        *reinterpret_cast<uint4 *>(&Bs[nb][t >> 4][8 * (t & 15)]) = ub;
    };
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.0f;
    fetch(0);
    stage(0);
    __syncthreads();
    int buf = 0;
    for (int k0 = 0; k0 < K; k0 += TK) {
        const bool more = k0 + TK < K;
        if (more) fetch(k0 + TK);  // the next slice comes in while this one is multiplied
#pragma unroll
        for (int k = 0; k < TK; ++k) {
            const uint4 av = *reinterpret_cast<const uint4 *>(&As[buf][k][ty * 8]);
            const uint4 bv = *reinterpret_cast<const uint4 *>(&Bs[buf][k][tx * 8]);
            unsigned short a[8], b[8];
            halves(av.x, a[0], a[1]);
            halves(av.y, a[2], a[3]);
            halves(av.z, a[4], a[5]);
            halves(av.w, a[6], a[7]);
            halves(bv.x, b[0], b[1]);
            halves(bv.y, b[2], b[3]);
            halves(bv.z, b[4], b[5]);
            halves(bv.w, b[6], b[7]);
#pragma unroll
            for (int j = 0; j < 8; ++j)
#pragma unroll
                for (int i = 0; i < 8; ++i) fma_mixed<F16>(acc[i][j], a[i], b[j]);
        }
        if (more) {
            const int nb = buf ^ 1;
            stage(nb);
            __syncthreads();
            buf = nb;
        }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        float *cr = C + (m0 + ty * 8 + i) * ldc + n0 + tx * 8;
        *reinterpret_cast<float4 *>(cr) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
        *reinterpret_cast<float4 *>(cr + 4) = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
    }
}

// Small GEMMs (a few 128x128 tiles would leave most SMs idle): one output per
// thread, 16x16 outputs per 256-thread block, K in 16-deep shared slices padded
// with zeros like the large tiling's, so each output is the same k-order FMA
// chain and both give identical bits.
template <bool F16>
__device__ __forceinline__ float widen16(const uint16_t *p, int64_t i) {
    const uint32_t w = p[i];
    if constexpr (F16) return __half2float(__ushort_as_half((unsigned short)w));
    return __uint_as_float(w << 16);
}

template <bool F16>
__global__ void __launch_bounds__(256)
gemm_ref_small(const uint16_t *__restrict__ A, int64_t lda, const uint16_t *__restrict__ B, int64_t ldb,
               float *__restrict__ C, int64_t ldc, int64_t M, int64_t N, int64_t K) {
    __shared__ float As[16][17], Bs[16][17];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int64_t row = (int64_t)blockIdx.y * 16 + ty, col = (int64_t)blockIdx.x * 16 + tx;
    float acc = 0.0f;
    for (int64_t k0 = 0; k0 < K; k0 += 16) {
        As[ty][tx] = (row < M && k0 + tx < K) ? widen16<F16>(A, row * lda + k0 + tx) : 0.0f;
        Bs[ty][tx] = (k0 + ty < K && col < N) ? widen16<F16>(B, (k0 + ty) * ldb + col) : 0.0f;
        __syncthreads();
#pragma unroll
        for (int k = 0; k < 16; ++k) acc = fmaf(As[ty][k], Bs[k][tx], acc);
        __syncthreads();
    }
    if (row < M && col < N) C[row * ldc + col] = acc;
}

template <bool F16>
cudaError_t launch_small(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb, float *c, int64_t ldc,
                         int64_t M, int64_t N, int64_t K, cudaStream_t s) {
    dim3 grid((unsigned)((N + 15) / 16), (unsigned)((M + 15) / 16));
    gemm_ref_small<F16><<<grid, 256, 0, s>>>(a, lda, b, ldb, c, ldc, M, N, K);
    return cudaGetLastError();
}

template <bool F16, int NG, int TK, int MINB>
cudaError_t launch_cfg(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb, float *c, int64_t ldc,
                       int64_t M, int64_t N, int64_t K, bool a_vec, bool b_vec, bool c_vec, cudaStream_t s) {
    constexpr int TN = 64 * NG;
    constexpr size_t smem = (size_t)2 * TK * (TM + TN) * sizeof(float);
    static const cudaError_t attr = cudaFuncSetAttribute(
        gemm_ref_simt<F16, NG, TK, MINB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (attr != cudaSuccess) return attr;
    dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
    gemm_ref_simt<F16, NG, TK, MINB><<<grid, 256, smem, s>>>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec);
    return cudaGetLastError();
}

// Whole tiles and aligned rows: the unchecked kernel (identical bits).
template <bool F16>
bool whole_tiles(int64_t M, int64_t N, int64_t K, bool a_vec, bool b_vec, bool c_vec) {
    return M % TM == 0 && N % 128 == 0 && K % 16 == 0 && K > 0 && K <= INT32_MAX - 16 && a_vec && b_vec && c_vec &&
           (M / TM) * (N / 128) <= INT32_MAX;
}

template <bool F16>
cudaError_t launch_whole(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb, float *c, int64_t ldc,
                         int64_t M, int64_t N, int64_t K, cudaStream_t s) {
    const int tm = (int)(M / TM), tn = (int)(N / 128);
    gemm_ref_whole<F16><<<(unsigned)(tm * tn), 256, 0, s>>>(a, lda, b, ldb, c, ldc, (int)K, tm, tn);
    return cudaGetLastError();
}

// Tiling of the reference (the tuning record's reference_tiling selects another
// for comparisons): 0 = 128x128, TK 16, one block per SM (143 registers); 1 =
// 128x256, TK 16; 2 = 128x128, TK 32; 3 = 128x256, TK 32; 4 = 128x128, TK 16
// with at most 128 registers, so two blocks share an SM.  Measured on GB300
// (TFLOP/s at 4096^3 / 8192^3, L2 flushed): 53.3/54.5, 49.9/56.6, 50.7/51.8,
// 43.0/49.0, 54.8/57.2,
// all bit-identical (each output is one k-order FMA chain).  Also measured and
// dropped: packed fp32x2 FMAs (with duplicated or diagonally paired operands:
// 47-55 at 16384^3), 32-deep slices with two blocks per SM, per-thread tiles of
// 4x16, 16x4, 8x16 and 16x8 (54-59 at 16384^3).  Default: 4, run as
// gemm_ref_whole when the GEMM is made of whole tiles, or 5 (the
// one-output-per-thread kernel) when the GEMM has at most 16 tiles of 128x128
// (L2 flushed: 256^3 30 -> 18 us, 512^3 53 -> 47 us; at 768^3, 36 tiles, the
// tiled form is faster).
int ref_tile(int64_t M, int64_t N) {
    const int v = tuning_snapshot().reference_tiling;
    if (v >= 0 && v <= 5) return v;
    return ((M + 127) / 128) * ((N + 127) / 128) <= 16 ? 5 : 4;
}

template <bool F16>
cudaError_t launch_ref(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb, float *c, int64_t ldc,
                       int64_t M, int64_t N, int64_t K, bool a_vec, bool b_vec, bool c_vec, cudaStream_t s) {
    switch (ref_tile(M, N)) {
    case 0: return launch_cfg<F16, 2, 16, 1>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s);
    case 1: return launch_cfg<F16, 4, 16, 1>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s);
    case 2: return launch_cfg<F16, 2, 32, 1>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s);
    case 3: return launch_cfg<F16, 4, 32, 1>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s);
    case 5: return launch_small<F16>(a, lda, b, ldb, c, ldc, M, N, K, s);
    default:
        if (whole_tiles<F16>(M, N, K, a_vec, b_vec, c_vec))
            return launch_whole<F16>(a, lda, b, ldb, c, ldc, M, N, K, s);
        return launch_cfg<F16, 2, 16, 2>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s);
    }
}

}  // namespace

cudaError_t launch_gemm_ref(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb, float *c, int64_t ldc,
                            int64_t M, int64_t N, int64_t K, bool f16, cudaStream_t s) {
    if (M == 0 || N == 0) return cudaSuccess;
    const bool a_vec = ((reinterpret_cast<uintptr_t>(a) & 15u) == 0) && (lda % 8 == 0);
    const bool b_vec = ((reinterpret_cast<uintptr_t>(b) & 15u) == 0) && (ldb % 8 == 0);
    const bool c_vec = ((reinterpret_cast<uintptr_t>(c) & 15u) == 0) && (ldc % 4 == 0);
    return f16 ? launch_ref<true>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s)
               : launch_ref<false>(a, lda, b, ldb, c, ldc, M, N, K, a_vec, b_vec, c_vec, s);
}

}  // namespace krex
