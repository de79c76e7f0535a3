// Measurement probe for the CUDA-core reference GEMM's roofline (not part of
// the paper's method): the FP32 fused multiply-add pipe's rate on this GPU,
// measured rather than derived from unit counts and clocks.
#include "common.cuh"

namespace krex {
namespace {

// Measurement probe: the FP32 fused multiply-add pipe's rate on this GPU.
// Each thread runs `iters` rounds of 16 independent FMA chains (enough
// independent work per warp to keep the pipe busy at any occupancy), at
// values that stay normal and finite; the sum is stored only if it equals a
// value no run produces in practice (the store keeps the chains live).
__global__ void __launch_bounds__(256)
fma_probe(int iters, float x, float y, float *sink) {
    float a[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) a[j] = (float)(threadIdx.x + j) * 0x1p-20f;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int j = 0; j < 16; ++j) a[j] = fmaf(a[j], x, y);
    }
    float s = 0.0f;
#pragma unroll
    for (int j = 0; j < 16; ++j) s += a[j];
    if (s == -1.0f) sink[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

}  // namespace

cudaError_t launch_fma_probe(int iters, int blocks, float *sink, cudaStream_t s) {
    // x < 1 and y small: the chains converge to y / (1 - x), normal and finite
    fma_probe<<<blocks, 256, 0, s>>>(iters, 0.999f, 0x1p-10f, sink);
    return cudaGetLastError();
}

}  // namespace krex
