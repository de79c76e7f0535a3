// A command's inputs from the caller's page-locked host buffers (the end-to-end
// form of the command), read by the SMs over the host link instead of the
// copy engine.  On GB300's Grace host the two run at the same rate from
// memory backed by huge pages (about 200 GB/s), but from memory in 64 KiB
// pages (where the host grants no huge page) a copy-engine read that follows
// a copy back and a pause of a quarter second ran at 12-14 GB/s, while SM
// loads of the same buffer kept 64-87 GB/s (measured on GB300, 512 MiB per
// copy).  Writes to host memory showed no such effect, so the copy back stays
// on the copy engine.
#include <algorithm>

#include "common.cuh"

namespace krex {
namespace {

// Rows of w16 16-byte words: n = rows * w16 words, source and destination row
// pitches in words.  Four independent loads in flight per thread; the source
// is read once, so its lines are not kept in L2 (ld.global.cs).
template <bool CONTIG>
__global__ void __launch_bounds__(256)
copy_rows16(const uint4 *__restrict__ src, int64_t spitch, uint4 *__restrict__ dst, int64_t dpitch, int64_t w16,
            int64_t n) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    auto src_at = [&](int64_t j) { return CONTIG ? j : (j / w16) * spitch + j % w16; };
    auto dst_at = [&](int64_t j) { return CONTIG ? j : (j / w16) * dpitch + j % w16; };
    for (; i + 3 * stride < n; i += 4 * stride) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = __ldcs(src + src_at(i + u * stride));
#pragma unroll
        for (int u = 0; u < 4; ++u) dst[dst_at(i + u * stride)] = v[u];
    }
    for (; i < n; i += stride) dst[dst_at(i)] = __ldcs(src + src_at(i));
}

}  // namespace

cudaError_t launch_copy_rows_from_host(const void *src, size_t spitch, void *dst, size_t dpitch, size_t width,
                                       size_t rows, cudaStream_t s, bool *launched) {
    *launched = false;
    const uintptr_t a = reinterpret_cast<uintptr_t>(src), b = reinterpret_cast<uintptr_t>(dst);
    if ((a | b | spitch | dpitch | width) & 15u) return cudaSuccess;  // not whole 16-byte words
    if (width == 0 || rows == 0) {
        *launched = true;
        return cudaSuccess;
    }
    const int64_t w16 = (int64_t)(width / 16), n = w16 * (int64_t)rows;
    // 8 blocks of 256 threads per SM, fewer for small copies
    const int64_t blocks = std::min<int64_t>((int64_t)sm_count() * 8, (n + 1023) / 1024);
    const auto *s16 = static_cast<const uint4 *>(src);
    auto *d16 = static_cast<uint4 *>(dst);
    if (spitch == width && dpitch == width)
        copy_rows16<true><<<(unsigned)blocks, 256, 0, s>>>(s16, 0, d16, 0, n, n);
    else
        copy_rows16<false><<<(unsigned)blocks, 256, 0, s>>>(s16, (int64_t)(spitch / 16), d16, (int64_t)(dpitch / 16),
                                                            w16, n);
    *launched = true;
    return cudaGetLastError();
}

}  // namespace krex
