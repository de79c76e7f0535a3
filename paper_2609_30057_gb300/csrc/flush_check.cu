// K3: the L2-flush writer and K6: the compare-and-reduce correctness check.
//
// Flush (paper Section 2.1: harnesses flush L2 between timed iterations;
// Section 4.2 step 5: region entry flushes L2 by writing an L2-sized buffer):
// a grid-stride loop of 16-byte stores of a per-call value.
//
// Check (Section 2.1: the command checks the candidate against the reference
// and returns a verdict).  Per element, IEEE fp32 without contraction:
//     d = |out - ref|,  violation iff !(d <= atol + rtol*|ref|)
// max |d| is reduced over the IEEE bit pattern as unsigned (valid ordering for
// non-negative floats; a NaN dominates and is reported as the canonical quiet
// NaN 0x7FC00000).  Warp reduction with __reduce_max_sync/__reduce_add_sync,
// then each block adds its count and maxes its bits into the call's result
// slot with two atomics and takes a ticket; the last block to take one
// prepares the other slot for the next call, re-arms the ticket and marks the
// call done.  Max and count are exact, so the result does not depend on the
// launch shape or the order of the atomics.
//
// The scratch is zeroed once (by the caller or krex_check_scratch_init) and
// every call leaves it ready for the next, so a check is one launch with no
// reset in front of it: calls alternate between two result slots (the slot of
// call g is g mod 2, g counted in the scratch), and a call's last block
// clears the slot the next call uses.  Block 0 clears the done word at its
// start; a scratch whose ticket was not zero on entry ends with done = 0 (no
// block saw itself last) or a non-zero ticket (a block saw itself last too
// early), and the host's fetch reports that instead of a result.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <type_traits>

#include <mutex>

#include <string.h>

#include "common.cuh"

namespace krex {
namespace {

// ------------------------------------------------------------------ flush --

__global__ void __launch_bounds__(512)
flush_kernel(uint4 *__restrict__ p, size_t n16, uint32_t value, uint8_t *tail, size_t ntail) {
    const uint4 v = make_uint4(value, value ^ 0x9E3779B9u, value + 1u, ~value);
    size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (; i + 3 * stride < n16; i += 4 * stride) {
        p[i] = v;
        p[i + stride] = v;
        p[i + 2 * stride] = v;
        p[i + 3 * stride] = v;
    }
    for (; i < n16; i += stride) p[i] = v;
    if (blockIdx.x == 0 && threadIdx.x < ntail) tail[threadIdx.x] = (uint8_t)value;
}

// ------------------------------------------------------------------ check --

constexpr int kCheckThreads = 256;
constexpr int kCheckMaxBlocks = 2048;
// Resident blocks per SM the check kernels are compiled for (their register
// budgets follow); the grid never exceeds what is resident at once, so no
// block waits for a second wave with too few loads in flight to keep HBM busy.
constexpr int kVecBlocksPerSM = 8;
constexpr int kGenericBlocksPerSM = 4;
constexpr uint32_t kCanonicalNaN = 0x7FC00000u;

// Scratch layout (device, caller-owned): two result slots and the call state,
// each on its own 128-byte line (the atomics of a call hit the slot's line and
// the ticket's line).
struct Slot {
    unsigned long long count;
    uint32_t max_bits;
    uint32_t pad[29];
};
struct CheckScratch {
    Slot slot[2];            // results of alternating calls
    unsigned int ticket;     // blocks that have added their results; 0 between calls
    unsigned int done;       // 1 once the last block has finished
    unsigned int gen;        // calls completed on this scratch (call g uses slot g % 2)
    unsigned int pad[29];
};
static_assert(sizeof(Slot) == 128 && sizeof(CheckScratch) == 384, "check scratch layout");
constexpr size_t kCheckHeaderBytes = sizeof(CheckScratch);

__device__ __forceinline__ float widen(const __nv_bfloat16 *p, int64_t i) {
    return __uint_as_float((uint32_t)(*reinterpret_cast<const uint16_t *>(p + i)) << 16);
}
__device__ __forceinline__ float widen(const __half *p, int64_t i) { return __half2float(p[i]); }
__device__ __forceinline__ float widen(const float *p, int64_t i) { return p[i]; }

struct Acc {
    uint32_t max_bits = 0;
    uint32_t count = 0;
    __device__ __forceinline__ void add(float o, float r, float atol, float rtol) {
        float d = fabsf(__fsub_rn(o, r));
        float thr = __fadd_rn(atol, __fmul_rn(rtol, fabsf(r)));
        count += !(d <= thr);
        uint32_t b = (d != d) ? kCanonicalNaN : __float_as_uint(d);
        max_bits = max(max_bits, b);
    }
};

// Eight packed 16-bit values widened exactly to fp32 (T: __nv_bfloat16 or
// __half).
template <typename T>
__device__ __forceinline__ void x8_to_f32(const uint4 &u, float *f) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if constexpr (std::is_same<T, __half>::value) {
            const float2 v = __half22float2(*reinterpret_cast<const __half2 *>(&w[k]));
            f[2 * k] = v.x;
            f[2 * k + 1] = v.y;
        } else {
            f[2 * k] = __uint_as_float(w[k] << 16);
            f[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
        }
    }
}

// Add the block's count and max into the call's slot; in the last block,
// prepare the next call's slot and mark this call done.
__device__ __forceinline__ void block_reduce_publish(Acc acc, CheckScratch *sc) {
    __shared__ uint32_t s_max[kCheckThreads / 32];
    __shared__ uint32_t s_cnt[kCheckThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t m = __reduce_max_sync(0xffffffffu, acc.max_bits);
    uint32_t c = __reduce_add_sync(0xffffffffu, acc.count);
    if (lane == 0) {
        s_max[warp] = m;
        s_cnt[warp] = c;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t bm = 0;
        unsigned long long bc = 0;
        for (int w = 0; w < kCheckThreads / 32; ++w) {
            bm = max(bm, s_max[w]);
            bc += s_cnt[w];
        }
        // gen changes only in the previous call's last block (stream order)
        const unsigned int g = __ldcg(&sc->gen);
        Slot &slot = sc->slot[g & 1u];
        if (bc) atomicAdd(&slot.count, bc);
        if (bm) atomicMax(&slot.max_bits, bm);
        __threadfence();
        const unsigned int t = atomicAdd(&sc->ticket, 1u);
        if (t == gridDim.x - 1) {
            // every block's atomics precede its ticket: this call's slot is
            // final; clear the next call's, re-arm, count the call, mark done
            __threadfence();
            Slot &next = sc->slot[(g + 1u) & 1u];
            next.count = 0ull;
            next.max_bits = 0u;
            sc->ticket = 0u;
            sc->gen = g + 1u;
            __threadfence();
            sc->done = 1u;
        }
    }
}

// Block 0 clears the done word before any block can take the last ticket
// (its own ticket comes after this store and a fence).
__device__ __forceinline__ void clear_done(CheckScratch *sc) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        sc->done = 0u;
        __threadfence();
    }
}

// Contiguous fast path: 16-bit out (bf16 or binary16) vs fp32 ref, 8
// elements per step.
template <typename T>
__global__ void __launch_bounds__(kCheckThreads, kVecBlocksPerSM)
check_16_f32_vec(const uint4 *__restrict__ out, const float4 *__restrict__ ref, int64_t n8,
                 const T *out_s, const float *ref_s, int64_t n, float atol,
                 float rtol, CheckScratch *sc) {
    Acc acc;
    clear_done(sc);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < n8; g += stride) {
        uint4 o = __ldcs(out + g);
        float4 r0 = __ldcs(ref + 2 * g);
        float4 r1 = __ldcs(ref + 2 * g + 1);
        float f[8];
        x8_to_f32<T>(o, f);
        acc.add(f[0], r0.x, atol, rtol);
        acc.add(f[1], r0.y, atol, rtol);
        acc.add(f[2], r0.z, atol, rtol);
        acc.add(f[3], r0.w, atol, rtol);
        acc.add(f[4], r1.x, atol, rtol);
        acc.add(f[5], r1.y, atol, rtol);
        acc.add(f[6], r1.z, atol, rtol);
        acc.add(f[7], r1.w, atol, rtol);
    }
    if (blockIdx.x == 0)
        for (int64_t i = n8 * 8 + threadIdx.x; i < n; i += blockDim.x)
            acc.add(widen(out_s, i), ref_s[i], atol, rtol);
    block_reduce_publish(acc, sc);
}

// Contiguous fast path: fp32 out vs fp32 ref, 4 elements per step, 2 steps unrolled.
__global__ void __launch_bounds__(kCheckThreads, kVecBlocksPerSM)
check_f32_f32_vec(const float4 *__restrict__ out, const float4 *__restrict__ ref, int64_t n4,
                  const float *out_s, const float *ref_s, int64_t n, float atol, float rtol,
                  CheckScratch *sc) {
    Acc acc;
    clear_done(sc);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (; g + stride < n4; g += 2 * stride) {
        float4 o0 = __ldcs(out + g), r0 = __ldcs(ref + g);
        float4 o1 = __ldcs(out + g + stride), r1 = __ldcs(ref + g + stride);
        acc.add(o0.x, r0.x, atol, rtol);
        acc.add(o0.y, r0.y, atol, rtol);
        acc.add(o0.z, r0.z, atol, rtol);
        acc.add(o0.w, r0.w, atol, rtol);
        acc.add(o1.x, r1.x, atol, rtol);
        acc.add(o1.y, r1.y, atol, rtol);
        acc.add(o1.z, r1.z, atol, rtol);
        acc.add(o1.w, r1.w, atol, rtol);
    }
    for (; g < n4; g += stride) {
        float4 o0 = __ldcs(out + g), r0 = __ldcs(ref + g);
        acc.add(o0.x, r0.x, atol, rtol);
        acc.add(o0.y, r0.y, atol, rtol);
        acc.add(o0.z, r0.z, atol, rtol);
        acc.add(o0.w, r0.w, atol, rtol);
    }
    if (blockIdx.x == 0)
        for (int64_t i = n4 * 4 + threadIdx.x; i < n; i += blockDim.x)
            acc.add(out_s[i], ref_s[i], atol, rtol);
    block_reduce_publish(acc, sc);
}

// Any layout / dtype pair: one element per step.
template <typename TO, typename TR>
__global__ void __launch_bounds__(kCheckThreads, kGenericBlocksPerSM)
check_generic(const TO *out, int64_t ldo, const TR *ref, int64_t ldr, int64_t rows,
              int64_t cols, float atol, float rtol, CheckScratch *sc) {
    Acc acc;
    clear_done(sc);
    const int64_t n = rows * cols;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        int64_t r = i / cols, c = i - r * cols;
        acc.add(widen(out, r * ldo + c), widen(ref, r * ldr + c), atol, rtol);
    }
    block_reduce_publish(acc, sc);
}

template <typename TO, typename TR>
void launch_generic(const void *out, int64_t ldo, const void *ref, int64_t ldr, int64_t rows, int64_t cols,
                    float atol, float rtol, CheckScratch *sc, int blocks, cudaStream_t s) {
    check_generic<TO, TR><<<blocks, kCheckThreads, 0, s>>>(static_cast<const TO *>(out), ldo,
                                                          static_cast<const TR *>(ref), ldr, rows, cols,
                                                          atol, rtol, sc);
}

template <typename TO>
void launch_generic_out(const void *out, int64_t ldo, const void *ref, int ref_dtype, int64_t ldr, int64_t rows,
                        int64_t cols, float atol, float rtol, CheckScratch *sc, int blocks, cudaStream_t s) {
    if (ref_dtype == KREX_F32)
        launch_generic<TO, float>(out, ldo, ref, ldr, rows, cols, atol, rtol, sc, blocks, s);
    else if (ref_dtype == KREX_BF16)
        launch_generic<TO, __nv_bfloat16>(out, ldo, ref, ldr, rows, cols, atol, rtol, sc, blocks, s);
    else
        launch_generic<TO, __half>(out, ldo, ref, ldr, rows, cols, atol, rtol, sc, blocks, s);
}

// Any layout and any pair of krex dtypes (validated by the caller).
void launch_check_generic(const void *out, int out_dtype, int64_t ldo, const void *ref, int ref_dtype,
                          int64_t ldr, int64_t rows, int64_t cols, float atol, float rtol, CheckScratch *sc,
                          int blocks, cudaStream_t s) {
    if (out_dtype == KREX_F32)
        launch_generic_out<float>(out, ldo, ref, ref_dtype, ldr, rows, cols, atol, rtol, sc, blocks, s);
    else if (out_dtype == KREX_BF16)
        launch_generic_out<__nv_bfloat16>(out, ldo, ref, ref_dtype, ldr, rows, cols, atol, rtol, sc, blocks, s);
    else
        launch_generic_out<__half>(out, ldo, ref, ref_dtype, ldr, rows, cols, atol, rtol, sc, blocks, s);
}

int check_blocks(int64_t items, int blocks_per_sm) {
    int64_t b = (items + kCheckThreads - 1) / kCheckThreads;
    int64_t cap = (int64_t)sm_count() * blocks_per_sm;
    if (cap > kCheckMaxBlocks) cap = kCheckMaxBlocks;
    if (b > cap) b = cap;
    if (b < 1) b = 1;
    return (int)b;
}

}  // namespace

size_t check_scratch_bytes() { return sizeof(CheckScratch); }

size_t check_header_bytes() { return kCheckHeaderBytes; }

cudaError_t init_check_scratch(void *scratch, cudaStream_t s) {
    return cudaMemsetAsync(scratch, 0, kCheckHeaderBytes, s);
}

krex_status read_check_header(const void *scratch, krex_check_result *r, cudaStream_t s) {
    CheckScratch h;
    cudaError_t e = cudaMemcpyAsync(&h, scratch, kCheckHeaderBytes, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return cuda_error(e, "cudaMemcpyAsync (check result)");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_error(e, "cudaStreamSynchronize (check result)");
    if (h.done != 1u || h.ticket != 0u)
        return set_error(KREX_ERR_STATE,
                         "check scratch was not ready (done %u, ticket %u): zero its %zu bytes once before its "
                         "first check (krex_check_scratch_init)",
                         h.done, h.ticket, kCheckHeaderBytes);
    const Slot &res = h.slot[(h.gen - 1u) & 1u];  // the call just completed
    memcpy(&r->max_abs_err, &res.max_bits, sizeof(float));
    r->reserved = 0;
    r->n_violations = res.count;
    return KREX_OK;
}

cudaError_t launch_flush(void *p, size_t bytes, uint32_t value, cudaStream_t s) {
    if (bytes == 0) return cudaSuccess;
    size_t n16 = bytes / 16, ntail = bytes % 16;
    int64_t blocks = (int64_t)((n16 + 511) / 512);
    int64_t cap = (int64_t)sm_count() * 4;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    flush_kernel<<<(unsigned)blocks, 512, 0, s>>>(static_cast<uint4 *>(p), n16, value,
                                                  static_cast<uint8_t *>(p) + n16 * 16, ntail);
    return cudaGetLastError();
}

cudaError_t launch_check(const void *out, int out_dtype, int64_t ldo, const void *ref,
                         int ref_dtype, int64_t ldr, int64_t rows, int64_t cols, float atol,
                         float rtol, void *scratch, cudaStream_t s) {
    CheckScratch *sc = static_cast<CheckScratch *>(scratch);
    const int64_t n = rows * cols;
    const bool contiguous = (ldo == cols && ldr == cols) || rows <= 1;
    const bool a16 = ((reinterpret_cast<uintptr_t>(out) | reinterpret_cast<uintptr_t>(ref)) & 15u) == 0;
    if (contiguous && a16 && out_dtype == KREX_BF16 && ref_dtype == KREX_F32) {
        int64_t n8 = n / 8;
        check_16_f32_vec<__nv_bfloat16><<<check_blocks(n8, kVecBlocksPerSM), kCheckThreads, 0, s>>>(
            static_cast<const uint4 *>(out), static_cast<const float4 *>(ref), n8,
            static_cast<const __nv_bfloat16 *>(out), static_cast<const float *>(ref), n, atol,
            rtol, sc);
    } else if (contiguous && a16 && out_dtype == KREX_F16 && ref_dtype == KREX_F32) {
        int64_t n8 = n / 8;
        check_16_f32_vec<__half><<<check_blocks(n8, kVecBlocksPerSM), kCheckThreads, 0, s>>>(
            static_cast<const uint4 *>(out), static_cast<const float4 *>(ref), n8,
            static_cast<const __half *>(out), static_cast<const float *>(ref), n, atol, rtol, sc);
    } else if (contiguous && a16 && out_dtype == KREX_F32 && ref_dtype == KREX_F32) {
        int64_t n4 = n / 4;
        check_f32_f32_vec<<<check_blocks(n4 / 2, kVecBlocksPerSM), kCheckThreads, 0, s>>>(
            static_cast<const float4 *>(out), static_cast<const float4 *>(ref), n4,
            static_cast<const float *>(out), static_cast<const float *>(ref), n, atol, rtol, sc);
    } else {
        launch_check_generic(out, out_dtype, ldo, ref, ref_dtype, ldr, rows, cols, atol, rtol, sc,
                             check_blocks(n, kGenericBlocksPerSM), s);
    }
    return cudaGetLastError();
}

}  // namespace krex

// --------------------------------------------------- allocation-free check
//
// krex_check with library-owned scratch, for callers that must not allocate
// device memory: code whose device memory is owned by another allocator with
// no room or permission to give (a framework's caching pool or a fixed memory
// budget), and timing harnesses in which a cudaMalloc/cudaFree would be a
// hazard because those calls can synchronise the whole device and disturb the
// measurement around them.  The scratch is a fixed static device array that
// each GPU loading this library keeps until the process exits.

// Capacity: room for the check's scratch (two result slots and the call
// state, 384 bytes) with a wide margin, fixed so the array's size does not
// change with the check's layout.
#define KREX_CHECK_NOALLOC_SCRATCH_BYTES 33024
static __device__ __align__(256) unsigned char g_check_noalloc_scratch[KREX_CHECK_NOALLOC_SCRATCH_BYTES];
static_assert(sizeof(krex::CheckScratch) <= KREX_CHECK_NOALLOC_SCRATCH_BYTES,
              "the static check scratch must hold the check's scratch layout");

namespace krex {
namespace {

typedef CUresult (*PfnCtxGetCurrent)(CUcontext *);
typedef CUresult (*PfnCtxGetId)(CUcontext, unsigned long long *);

// The driver's cuCtxGetCurrent / cuCtxGetId through the runtime's entry-point
// query (the library links no driver library).
void driver_ctx_fns(PfnCtxGetCurrent *get_current, PfnCtxGetId *get_id) {
    static PfnCtxGetCurrent gc = nullptr;
    static PfnCtxGetId gi = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            gc = reinterpret_cast<PfnCtxGetCurrent>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            gi = reinterpret_cast<PfnCtxGetId>(p);
    });
    *get_current = gc;
    *get_id = gi;
}

// Where the static array lives, per device ordinal, and in which context:
// a context that is destroyed and created again (a device reset, a new
// primary context) reloads the module and may move the array, so the address
// is resolved again whenever the current context's id differs.
struct NoallocSlot {
    unsigned long long ctx_id = 0;
    void *addr = nullptr;
};
std::mutex g_noalloc_mu;
NoallocSlot g_noalloc[64];

}  // namespace
}  // namespace krex

extern "C" krex_status krex_check_noalloc(krex_buf out, krex_buf ref, float atol, float rtol,
                                          krex_check_result *host_result, krex_stream_t stream) {
    using namespace krex;
    krex_status st;
    if ((st = check_buf(out, "check_noalloc: out")) || (st = check_buf(ref, "check_noalloc: ref"))) return st;
    if (out.rows != ref.rows || out.cols != ref.cols)
        return set_error(KREX_ERR_INVALID, "check_noalloc: out and ref shapes differ");
    if (!host_result) return set_error(KREX_ERR_INVALID, "check_noalloc: host_result is null");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) return set_error(KREX_ERR_UNSUPPORTED, "check_noalloc: device ordinal %d >= 64", dev);
    PfnCtxGetCurrent get_current = nullptr;
    PfnCtxGetId get_id = nullptr;
    driver_ctx_fns(&get_current, &get_id);
    if (!get_current || !get_id)
        return set_error(KREX_ERR_CUDA, "check_noalloc: the driver offers no cuCtxGetCurrent / cuCtxGetId");
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) {
        // no context bound to this thread yet: bind the device's primary one
        e = cudaSetDevice(dev);
        if (e != cudaSuccess) return cuda_error(e, "cudaSetDevice (check_noalloc)");
        if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr)
            return set_error(KREX_ERR_CUDA, "check_noalloc: no current context on device %d", dev);
    }
    unsigned long long ctx_id = 0;
    if (get_id(ctx, &ctx_id) != CUDA_SUCCESS)
        return set_error(KREX_ERR_CUDA, "check_noalloc: cuCtxGetId failed");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    void *scratch = nullptr;
    {
        // set-up, once per device and context: resolve the array's device
        // address in that context and zero the check's header there
        std::lock_guard<std::mutex> lk(g_noalloc_mu);
        NoallocSlot &slot = g_noalloc[dev];
        if (slot.addr == nullptr || slot.ctx_id != ctx_id) {
            void *p = nullptr;
            e = cudaGetSymbolAddress(&p, g_check_noalloc_scratch);
            if (e != cudaSuccess) return cuda_error(e, "cudaGetSymbolAddress (check_noalloc scratch)");
            e = init_check_scratch(p, s);
            if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync (check_noalloc scratch header)");
            slot.addr = p;
            slot.ctx_id = ctx_id;
        }
        scratch = slot.addr;
    }
    e = launch_check(out.ptr, out.dtype, out.ld, ref.ptr, ref.dtype, ref.ld, out.rows, out.cols, atol, rtol, scratch, s);
    if (e != cudaSuccess) return cuda_error(e, "check_noalloc launch");
    note_launches(1);
    krex_check_result r;
    if ((st = read_check_header(scratch, &r, s))) return st;
    *host_result = r;
    return ok_status();
}
