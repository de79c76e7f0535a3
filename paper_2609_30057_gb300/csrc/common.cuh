// Internal declarations shared by the translation units of libkrex.so.
// Not part of the public ABI (see include/krex.h).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "krex.h"

namespace krex {

// ---- device properties (cached per device) -------------------------------
int sm_count();                 // multiprocessors of the current device
size_t l2_bytes_current();      // L2 size of the current device

// ---- kernel launchers (return the launch error, never synchronise) --------

// K1: SplitMix64 -> U[-1,1] -> bf16 (f16: binary16), 16-byte stores.  `key`
// is the stream key.
cudaError_t launch_fill_uniform_16(uint64_t key, bool f16, void *out, int64_t rows, int64_t cols,
                                   int64_t ld, cudaStream_t s);
// K2: SplitMix64 -> Box-Muller -> N(0, sigma^2) fp32, 16-byte stores.
cudaError_t launch_fill_normal_f32(uint64_t key, float sigma, float *out, int64_t rows,
                                   int64_t cols, int64_t ld, cudaStream_t s);
// Probe: the fill kernel of `dist` over n contiguous elements on `blocks` x
// 256 threads, folding instead of storing (sink: one word per thread).
cudaError_t launch_generator_probe(int32_t dist, uint64_t key, int64_t n, float sigma, int blocks, uint32_t *sink,
                                   cudaStream_t s);
// Probe: `blocks` x 256 threads, each `iters` rounds of 16 independent fp32
// FMAs (2 x 16 x iters flops per thread).
cudaError_t launch_fma_probe(int iters, int blocks, float *sink, cudaStream_t s);
// Rows of `width` bytes from a host buffer the device reads directly (src is
// its device-side address) into device memory, by SM loads.  Launches only
// when src, dst, both pitches and width are multiples of 16 bytes; *launched
// tells the caller whether to copy another way.
cudaError_t launch_copy_rows_from_host(const void *src, size_t spitch, void *dst, size_t dpitch, size_t width,
                                       size_t rows, cudaStream_t s, bool *launched);
// K3: grid-stride writer of `bytes` bytes of `value`.
cudaError_t launch_flush(void *p, size_t bytes, uint32_t value, cudaStream_t s);
// K6: compare-and-reduce; result (16 bytes) lands in scratch, whose 32-byte
// header must be zero before its first use and is left ready by every call.
size_t check_scratch_bytes();
size_t check_header_bytes();
cudaError_t init_check_scratch(void *scratch, cudaStream_t s);
// Copy the result of the last check on `scratch` to *r (synchronises s);
// KREX_ERR_STATE if the header shows the scratch was not ready on entry.
krex_status read_check_header(const void *scratch, krex_check_result *r, cudaStream_t s);
cudaError_t launch_check(const void *out, int out_dtype, int64_t ldo, const void *ref,
                         int ref_dtype, int64_t ldr, int64_t rows, int64_t cols, float atol,
                         float rtol, void *scratch, cudaStream_t s);
// K5: single-pass online row softmax.
cudaError_t launch_softmax(const float *x, int64_t ldx, float *y, int64_t ldy, int64_t rows,
                           int64_t cols, cudaStream_t s);
// K8: three-pass reference softmax.
cudaError_t launch_softmax_ref(const float *x, int64_t ldx, float *y, int64_t ldy,
                               int64_t rows, int64_t cols, cudaStream_t s);
// K7: SIMT fp32 reference GEMM (bf16 or, with f16, binary16 in; fp32 out).
cudaError_t launch_gemm_ref(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb,
                            float *c, int64_t ldc, int64_t M, int64_t N, int64_t K, bool f16,
                            cudaStream_t s);
// K4: tcgen05 GEMM.  Returns KREX_OK or an error status with a message set.
// `workspace` (may be NULL) enables the split-K tail; see gemm_workspace_bytes.
// f16: binary16 A, B and C (else bf16).
krex_status launch_gemm_tcgen05(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb,
                                uint16_t *c, int64_t ldc, int64_t M, int64_t N, int64_t K, bool f16,
                                void *workspace, size_t workspace_bytes, cudaStream_t s);
size_t gemm_workspace_bytes();
// Device status word of the GEMM kernel's bounded waits (read and clear).
cudaError_t read_and_clear_device_status(uint32_t *code);
cudaError_t read_device_status_detail(unsigned long long *words);

// The process-wide tuning record (a copy; see krex_set_tuning).
krex_tuning tuning_snapshot();
// The failure-detection test hook of the GEMM's split-K hand-over.
void set_debug_stall_handover(bool on);

// Count kernels launched outside api.cu in krex_launch_count().
void note_launches(int n);

// ---- errors -----------------------------------------------------------------
krex_status set_error(krex_status st, const char *fmt, ...);
krex_status cuda_error(cudaError_t e, const char *what);
// KREX_OK, clearing the calling thread's last error string.
krex_status ok_status();
// Validation of a caller's buffer descriptor (dtype, shape, stride, pointer);
// sets the error string and returns KREX_ERR_INVALID on a bad one.
krex_status check_buf(const krex_buf &b, const char *name);

}  // namespace krex

#define KREX_CUDA_TRY(call)                                            \
    do {                                                               \
        cudaError_t _e = (call);                                       \
        if (_e != cudaSuccess) return ::krex::cuda_error(_e, #call);   \
    } while (0)
