// K5: the bandwidth-bound candidate, a single-pass online row softmax, and
// K8: the three-pass reference softmax the check compares it against.
//
//   y_j = exp(x_j - m) / sum_k exp(x_k - m),   m = max_k x_k   (per row)
//
// K5 reads each row from HBM once into registers (one CTA per row, 16-byte
// loads), reduces a running (max, sum) pair with the online merge
//   (m, s) + (m', s') = (M, s e^(m-M) + s' e^(m'-M)),  M = max(m, m')
// across the warp with shuffles and across warps through shared memory, and
// writes each row once: one read and one write of HBM per element.  Rows too
// long for the register tile fall back to a two-read online kernel.
#include <math.h>

#include "common.cuh"

namespace krex {
namespace {

struct MS {
    float m, s;
};

__device__ __forceinline__ MS ms_merge(MS a, MS b) {
    float M = fmaxf(a.m, b.m);
    if (M == -INFINITY) return {M, 0.0f};
    float sa = (a.m == -INFINITY) ? 0.0f : a.s * expf(a.m - M);
    float sb = (b.m == -INFINITY) ? 0.0f : b.s * expf(b.m - M);
    return {M, sa + sb};
}

template <int THREADS>
__device__ __forceinline__ MS block_merge(MS v) {
    __shared__ float s_m[THREADS / 32], s_s[THREADS / 32];
    __shared__ MS s_out;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        MS w{__shfl_xor_sync(0xffffffffu, v.m, o), __shfl_xor_sync(0xffffffffu, v.s, o)};
        v = ms_merge(v, w);
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) {
        s_m[warp] = v.m;
        s_s[warp] = v.s;
    }
    __syncthreads();
    if (warp == 0) {
        MS u = lane < THREADS / 32 ? MS{s_m[lane], s_s[lane]} : MS{-INFINITY, 0.0f};
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            MS w{__shfl_xor_sync(0xffffffffu, u.m, o), __shfl_xor_sync(0xffffffffu, u.s, o)};
            u = ms_merge(u, w);
        }
        if (lane == 0) s_out = u;
    }
    __syncthreads();
    MS r = s_out;
    __syncthreads();  // s_out may be rewritten by the next row
    return r;
}

// Register-tiled single pass: row length <= THREADS * 4 * VPT, 16-byte aligned
// rows (cols % 4 == 0, ld % 4 == 0).  Thread t owns float4 chunks t, t+THREADS, ...
template <int THREADS, int VPT>
__global__ void __launch_bounds__(THREADS)
softmax_rows_reg(const float *__restrict__ x, int64_t ldx, float *__restrict__ y, int64_t ldy,
                 int64_t rows, int cols) {
    const int nchunk = cols >> 2;
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
        const float4 *xr = reinterpret_cast<const float4 *>(x + r * ldx);
        float4 *yr = reinterpret_cast<float4 *>(y + r * ldy);
        float4 v[VPT];
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            int c = threadIdx.x + k * THREADS;
            v[k] = c < nchunk ? __ldcs(xr + c) : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        }
        float m = -INFINITY;
#pragma unroll
        for (int k = 0; k < VPT; ++k) m = fmaxf(m, fmaxf(fmaxf(v[k].x, v[k].y), fmaxf(v[k].z, v[k].w)));
        // a thread whose elements are all masked (-inf) shifts by 0, so they
        // become exp(-inf) = 0 and its sum 0, with no -inf - -inf
        const float shift = (m == -INFINITY) ? 0.0f : m;
        float s = 0.0f;
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            v[k].x = expf(v[k].x - shift);
            v[k].y = expf(v[k].y - shift);
            v[k].z = expf(v[k].z - shift);
            v[k].w = expf(v[k].w - shift);
            s += (v[k].x + v[k].y) + (v[k].z + v[k].w);
        }
        MS tot = block_merge<THREADS>(MS{m, s});
        float scale = (m == -INFINITY) ? 0.0f : expf(m - tot.m) / tot.s;
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            int c = threadIdx.x + k * THREADS;
            if (c < nchunk)
                __stcs(yr + c, make_float4(v[k].x * scale, v[k].y * scale, v[k].z * scale, v[k].w * scale));
        }
    }
}

// Any length / layout: online (max, sum) pass, then a write pass (two reads).
template <int THREADS>
__global__ void __launch_bounds__(THREADS)
softmax_rows_online(const float *__restrict__ x, int64_t ldx, float *__restrict__ y, int64_t ldy,
                    int64_t rows, int64_t cols) {
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
        const float *xr = x + r * ldx;
        float *yr = y + r * ldy;
        MS acc{-INFINITY, 0.0f};
        for (int64_t c = threadIdx.x; c < cols; c += THREADS) {
            float xv = xr[c];
            if (xv > acc.m) {
                acc.s = (acc.m == -INFINITY ? 0.0f : acc.s * expf(acc.m - xv)) + 1.0f;
                acc.m = xv;
            } else if (xv != -INFINITY) {  // a masked -inf adds 0 (and -inf - -inf would be NaN)
                acc.s += expf(xv - acc.m);
            }
        }
        MS tot = block_merge<THREADS>(acc);
        float inv = 1.0f / tot.s;
        for (int64_t c = threadIdx.x; c < cols; c += THREADS) yr[c] = expf(xr[c] - tot.m) * inv;
    }
}

// K8 reference: max pass, sum pass, write pass, plain block reductions.
__global__ void __launch_bounds__(256)
softmax_rows_ref3(const float *__restrict__ x, int64_t ldx, float *__restrict__ y, int64_t ldy,
                  int64_t rows, int64_t cols) {
    __shared__ float red[256];
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
        const float *xr = x + r * ldx;
        float *yr = y + r * ldy;
        float m = -INFINITY;
        for (int64_t c = threadIdx.x; c < cols; c += 256) m = fmaxf(m, xr[c]);
        red[threadIdx.x] = m;
        __syncthreads();
        for (int o = 128; o > 0; o >>= 1) {
            if ((int)threadIdx.x < o) red[threadIdx.x] = fmaxf(red[threadIdx.x], red[threadIdx.x + o]);
            __syncthreads();
        }
        m = red[0];
        __syncthreads();
        float s = 0.0f;
        for (int64_t c = threadIdx.x; c < cols; c += 256) s += expf(xr[c] - m);
        red[threadIdx.x] = s;
        __syncthreads();
        for (int o = 128; o > 0; o >>= 1) {
            if ((int)threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
            __syncthreads();
        }
        s = red[0];
        __syncthreads();
        for (int64_t c = threadIdx.x; c < cols; c += 256) yr[c] = expf(xr[c] - m) / s;
    }
}

unsigned row_grid(int64_t rows) {
    int64_t cap = (int64_t)sm_count() * 64;
    return (unsigned)(rows < cap ? rows : cap);
}

}  // namespace

cudaError_t launch_softmax(const float *x, int64_t ldx, float *y, int64_t ldy, int64_t rows,
                           int64_t cols, cudaStream_t s) {
    if (rows == 0 || cols == 0) return cudaSuccess;
    const bool vec = ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15u) == 0 &&
                     (cols & 3) == 0 && (ldx & 3) == 0 && (ldy & 3) == 0;
    const unsigned g = row_grid(rows);
    if (vec && cols <= 256 * 4 * 1)
        softmax_rows_reg<256, 1><<<g, 256, 0, s>>>(x, ldx, y, ldy, rows, (int)cols);
    else if (vec && cols <= 256 * 4 * 2)
        softmax_rows_reg<256, 2><<<g, 256, 0, s>>>(x, ldx, y, ldy, rows, (int)cols);
    else if (vec && cols <= 256 * 4 * 4)
        softmax_rows_reg<256, 4><<<g, 256, 0, s>>>(x, ldx, y, ldy, rows, (int)cols);
    else if (vec && cols <= 256 * 4 * 8)
        softmax_rows_reg<256, 8><<<g, 256, 0, s>>>(x, ldx, y, ldy, rows, (int)cols);
    else if (vec && cols <= 512 * 4 * 8)
        softmax_rows_reg<512, 8><<<g, 512, 0, s>>>(x, ldx, y, ldy, rows, (int)cols);
    else
        softmax_rows_online<512><<<g, 512, 0, s>>>(x, ldx, y, ldy, rows, cols);
    return cudaGetLastError();
}

cudaError_t launch_softmax_ref(const float *x, int64_t ldx, float *y, int64_t ldy, int64_t rows,
                               int64_t cols, cudaStream_t s) {
    if (rows == 0 || cols == 0) return cudaSuccess;
    softmax_rows_ref3<<<row_grid(rows), 256, 0, s>>>(x, ldx, y, ldy, rows, cols);
    return cudaGetLastError();
}

}  // namespace krex
