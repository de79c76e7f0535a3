// C ABI of libkrex.so (declared and documented in include/krex.h): argument
// validation, the critical region (paper Sections 4.1-4.2), the native timing
// loop and the whole benchmarking command (Section 2.1).  Host code only; the
// kernels live in the other translation units.
#include <pthread.h>
#include <sched.h>
#include <sys/mman.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>
#include <time.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <mutex>
#include <set>
#include <vector>

#include "common.cuh"

namespace krex {

// ------------------------------------------------------------------ errors --

static thread_local char t_err[512] = "";

krex_status set_error(krex_status st, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(t_err, sizeof(t_err), fmt, ap);
    va_end(ap);
    return st;
}

krex_status cuda_error(cudaError_t e, const char *what) {
    return set_error(KREX_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

static krex_status ok() {
    t_err[0] = '\0';
    return KREX_OK;
}

krex_status ok_status() { return ok(); }

// ------------------------------------------------------- device properties --

namespace {
constexpr int kMaxDev = 64;
std::atomic<int> g_sm[kMaxDev];
std::atomic<long long> g_l2[kMaxDev];
std::atomic<uint64_t> g_launches{0};
std::atomic<uint32_t> g_flush_value{0x5EED0001u};
}  // namespace

int sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return 152;
    int v = g_sm[dev].load(std::memory_order_relaxed);
    if (v <= 0) {
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) v = 152;
        g_sm[dev].store(v, std::memory_order_relaxed);
    }
    return v;
}

size_t l2_bytes_current() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return 0;
    long long v = g_l2[dev].load(std::memory_order_relaxed);
    if (v <= 0) {
        int a = 0;
        if (cudaDeviceGetAttribute(&a, cudaDevAttrL2CacheSize, dev) != cudaSuccess) return 0;
        v = a;
        g_l2[dev].store(v, std::memory_order_relaxed);
    }
    return (size_t)v;
}

static void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

// ------------------------------------------------------------------ tuning --

namespace {
std::mutex g_tuning_mu;
krex_tuning default_tuning() {
    krex_tuning t;
    memset(&t, 0, sizeof(t));
    t.gemm_tail_split = -1;
    t.gemm_split_k = -1;
    t.gemm_k_alternate = -1;
    t.reference_tiling = -1;
    return t;
}
krex_tuning g_tuning = default_tuning();

bool tuning_valid(const krex_tuning &t) {
    return (t.gemm_pair_tile_n == 0 || t.gemm_pair_tile_n == 128 || t.gemm_pair_tile_n == 192 ||
            t.gemm_pair_tile_n == 256 || t.gemm_pair_tile_n == 512) &&
           (t.gemm_stage_k == 0 || t.gemm_stage_k == 64 || t.gemm_stage_k == 128) &&
           (t.gemm_ring_stages == 0 ||
            (t.gemm_ring_stages >= 2 && t.gemm_ring_stages <= (t.gemm_stage_k == 64 ? 6 : 3))) &&
           (t.gemm_raster_group >= 0 && t.gemm_raster_group <= 64) &&
           (t.gemm_tail_split >= -1 && t.gemm_tail_split <= 1) && (t.gemm_split_k >= -1 && t.gemm_split_k <= 1) &&
           (t.gemm_k_alternate >= -1 && t.gemm_k_alternate <= 1) &&
           (t.reference_tiling >= -1 && t.reference_tiling <= 5) &&
           (t.wait_timeout_ms >= 0 && t.wait_timeout_ms <= 600000);
}
}  // namespace

krex_tuning tuning_snapshot() {
    std::lock_guard<std::mutex> lk(g_tuning_mu);
    return g_tuning;
}

void note_launches(int n) { count_launches(n); }

// ---------------------------------------------------------- host SplitMix64 --

static uint64_t host_mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static uint64_t stream_key(uint64_t seed, uint32_t tensor_id) {
    return host_mix64(seed + ((uint64_t)tensor_id + 1ull) * 0x9E3779B97F4A7C15ull);
}

// -------------------------------------------------------------- validation --

static size_t elem_size(int32_t dt) { return (dt == KREX_BF16 || dt == KREX_F16) ? 2 : (dt == KREX_F32 ? 4 : 0); }

static bool is_gemm(int32_t op) { return op == KREX_OP_GEMM_BF16 || op == KREX_OP_GEMM_F16; }

// dtype of a GEMM op's operands and output; fp32 for the softmax
static int32_t op_dtype(int32_t op) {
    return op == KREX_OP_GEMM_BF16 ? KREX_BF16 : (op == KREX_OP_GEMM_F16 ? KREX_F16 : KREX_F32);
}

krex_status check_buf(const krex_buf &b, const char *name) {
    if (elem_size(b.dtype) == 0) return set_error(KREX_ERR_INVALID, "%s: bad dtype %d", name, b.dtype);
    if (b.rows < 0 || b.cols < 0) return set_error(KREX_ERR_INVALID, "%s: negative shape", name);
    if (b.rows > 0 && b.ld < b.cols) return set_error(KREX_ERR_INVALID, "%s: ld %lld < cols %lld", name,
                                                     (long long)b.ld, (long long)b.cols);
    if (b.rows * b.cols > 0 && b.ptr == nullptr) return set_error(KREX_ERR_INVALID, "%s: null pointer", name);
    if (b.rows > 0 && b.cols > 0 && b.ld > (int64_t)1 << 40) return set_error(KREX_ERR_INVALID, "%s: ld too large", name);
    return KREX_OK;
}

static bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The optional GEMM workspace: NULL, or 16-byte aligned and large enough.
static krex_status check_gemm_workspace(const void *ws, size_t bytes) {
    if (!ws) return KREX_OK;
    if (!aligned16(ws)) return set_error(KREX_ERR_UNSUPPORTED, "GEMM workspace must be 16-byte aligned");
    if (bytes < gemm_workspace_bytes())
        return set_error(KREX_ERR_INVALID, "GEMM workspace of %zu bytes, need %zu", bytes, gemm_workspace_bytes());
    return KREX_OK;
}

static krex_status check_op_shapes(int32_t op, const krex_buf *in, int32_t n_in, const krex_buf &out,
                                   int32_t out_dtype, const char *out_name) {
    if (!in) return set_error(KREX_ERR_INVALID, "in is null");
    krex_status st;
    if (is_gemm(op)) {
        if (n_in != 2) return set_error(KREX_ERR_INVALID, "GEMM takes 2 inputs, got %d", n_in);
        if ((st = check_buf(in[0], "A")) || (st = check_buf(in[1], "B")) || (st = check_buf(out, out_name))) return st;
        if (in[0].dtype != op_dtype(op) || in[1].dtype != op_dtype(op))
            return set_error(KREX_ERR_INVALID, "GEMM inputs must be %s", op == KREX_OP_GEMM_F16 ? "fp16" : "bf16");
        if (out.dtype != out_dtype) return set_error(KREX_ERR_INVALID, "%s has the wrong dtype", out_name);
        if (in[0].cols != in[1].rows) return set_error(KREX_ERR_INVALID, "A.cols %lld != B.rows %lld",
                                                       (long long)in[0].cols, (long long)in[1].rows);
        if (out.rows != in[0].rows || out.cols != in[1].cols)
            return set_error(KREX_ERR_INVALID, "%s shape must be A.rows x B.cols", out_name);
        return KREX_OK;
    }
    if (op == KREX_OP_SOFTMAX_F32) {
        if (n_in != 1) return set_error(KREX_ERR_INVALID, "softmax takes 1 input, got %d", n_in);
        if ((st = check_buf(in[0], "X")) || (st = check_buf(out, out_name))) return st;
        if (in[0].dtype != KREX_F32 || out.dtype != KREX_F32)
            return set_error(KREX_ERR_INVALID, "softmax input and output must be fp32");
        if (out.rows != in[0].rows || out.cols != in[0].cols)
            return set_error(KREX_ERR_INVALID, "%s shape must equal X shape", out_name);
        return KREX_OK;
    }
    return set_error(KREX_ERR_INVALID, "unknown op %d", op);
}

// Candidate/reference dispatch after validation.
static krex_status do_candidate(int32_t op, const krex_buf *in, const krex_buf &out, cudaStream_t s,
                                void *ws = nullptr, size_t ws_bytes = 0) {
    if (is_gemm(op)) {
        const krex_buf &A = in[0], &B = in[1];
        const int64_t M = A.rows, K = A.cols, N = B.cols;
        if (M == 0 || N == 0) return ok();
        if (K > 0) {
            if ((K % 8) || (N % 8) || (A.ld % 8) || (B.ld % 8) || !aligned16(A.ptr) || !aligned16(B.ptr))
                return set_error(KREX_ERR_UNSUPPORTED,
                                 "tcgen05 GEMM needs K, N, lda, ldb multiples of 8 and 16-byte aligned A, B "
                                 "(TMA rows must start on 16 bytes)");
        }
        krex_status st = launch_gemm_tcgen05(static_cast<const uint16_t *>(A.ptr), A.ld,
                                             static_cast<const uint16_t *>(B.ptr), B.ld,
                                             static_cast<uint16_t *>(out.ptr), out.ld, M, N, K,
                                             op == KREX_OP_GEMM_F16, ws, ws_bytes, s);
        if (st != KREX_OK) return st;
        if (K > 0) count_launches(1);
        return ok();
    }
    const krex_buf &X = in[0];
    KREX_CUDA_TRY(launch_softmax(static_cast<const float *>(X.ptr), X.ld, static_cast<float *>(out.ptr), out.ld,
                                 X.rows, X.cols, s));
    if (X.rows * X.cols > 0) count_launches(1);
    return ok();
}

static krex_status do_reference(int32_t op, const krex_buf *in, const krex_buf &ref, cudaStream_t s) {
    if (is_gemm(op)) {
        const krex_buf &A = in[0], &B = in[1];
        KREX_CUDA_TRY(launch_gemm_ref(static_cast<const uint16_t *>(A.ptr), A.ld,
                                      static_cast<const uint16_t *>(B.ptr), B.ld, static_cast<float *>(ref.ptr),
                                      ref.ld, A.rows, B.cols, A.cols, op == KREX_OP_GEMM_F16, s));
        if (A.rows * B.cols > 0) count_launches(1);
        return ok();
    }
    const krex_buf &X = in[0];
    KREX_CUDA_TRY(launch_softmax_ref(static_cast<const float *>(X.ptr), X.ld, static_cast<float *>(ref.ptr),
                                     ref.ld, X.rows, X.cols, s));
    if (X.rows * X.cols > 0) count_launches(1);
    return ok();
}

static krex_status do_flush(void *scratch, size_t bytes, cudaStream_t s) {
    if (bytes == 0) return ok();
    if (!scratch) return set_error(KREX_ERR_INVALID, "flush scratch is null");
    if (!aligned16(scratch)) return set_error(KREX_ERR_UNSUPPORTED, "flush scratch must be 16-byte aligned");
    KREX_CUDA_TRY(launch_flush(scratch, bytes, g_flush_value.fetch_add(1u, std::memory_order_relaxed), s));
    count_launches(1);
    return ok();
}

// ----------------------------------------------------------------- region --

double percentile_sorted(const std::vector<double> &xs, double q) {
    const size_t n = xs.size();
    const double h = (double)(n - 1) * q;
    const double lo_f = std::floor(h);
    const size_t lo = (size_t)lo_f;
    if (lo >= n - 1) return xs[n - 1];
    return xs[lo] + (h - lo_f) * (xs[lo + 1] - xs[lo]);
}

namespace {

struct EventPool {
    std::mutex mu;
    std::vector<std::pair<int, cudaEvent_t>> free;  // (device, event)
    cudaError_t take(int dev, size_t n, std::vector<cudaEvent_t> &out) {
        std::lock_guard<std::mutex> lk(mu);
        for (size_t i = 0; i < free.size() && out.size() < n;) {
            if (free[i].first == dev) {
                out.push_back(free[i].second);
                free[i] = free.back();
                free.pop_back();
            } else {
                ++i;
            }
        }
        while (out.size() < n) {
            cudaEvent_t e;
            cudaError_t err = cudaEventCreate(&e);
            if (err != cudaSuccess) return err;
            out.push_back(e);
        }
        return cudaSuccess;
    }
    void give(int dev, std::vector<cudaEvent_t> &evs) {
        std::lock_guard<std::mutex> lk(mu);
        for (cudaEvent_t e : evs) free.emplace_back(dev, e);
        evs.clear();
    }
};
EventPool &event_pool() {
    static EventPool *p = new EventPool();  // intentionally never destroyed
    return *p;
}

std::mutex g_open_mu;
std::set<cudaStream_t> &open_streams() {
    static std::set<cudaStream_t> *s = new std::set<cudaStream_t>();
    return *s;
}

// Spin briefly, then park with growing sleeps (the spin-park policy of the
// paper's Section 4.3) until the stream is idle or the timeout passes.
krex_status drain_stream(cudaStream_t s, int64_t timeout_us) {
    using clk = std::chrono::steady_clock;
    if (timeout_us <= 0) timeout_us = 10 * 1000 * 1000;
    const auto t0 = clk::now();
    const auto spin_until = t0 + std::chrono::microseconds(50);
    const auto deadline = t0 + std::chrono::microseconds(timeout_us);
    long sleep_ns = 2000;
    for (;;) {
        cudaError_t e = cudaStreamQuery(s);
        if (e == cudaSuccess) return KREX_OK;
        if (e != cudaErrorNotReady) return cuda_error(e, "cudaStreamQuery (region drain)");
        const auto now = clk::now();
        if (now >= deadline)
            return set_error(KREX_ERR_TIMEOUT, "region entry: stream did not drain within %lld us",
                             (long long)timeout_us);
        if (now >= spin_until) {
            struct timespec ts = {0, sleep_ns};
            nanosleep(&ts, nullptr);
            sleep_ns = std::min(sleep_ns * 2, 1000000L);
        }
    }
}

}  // namespace
}  // namespace krex

struct krex_region {
    cudaStream_t stream;
    krex_gate *gate;
    int32_t tenant;
    uint64_t epoch;
    int device;
    int32_t max_iters;
    int32_t n_begun;
    int32_t n_ended;
    std::vector<cudaEvent_t> ev;  // start of iteration i = ev[2i], end = ev[2i+1]
    bool pinned;
    cpu_set_t old_mask;
};

using namespace krex;

static void region_release(krex_region *r) {
    if (r->gate) krex_gate_exit(r->gate, r->tenant, r->epoch);  // reopen the gate (step 8)
    if (r->pinned) pthread_setaffinity_np(pthread_self(), sizeof(cpu_set_t), &r->old_mask);
    event_pool().give(r->device, r->ev);
    {
        std::lock_guard<std::mutex> lk(g_open_mu);
        open_streams().erase(r->stream);
    }
    delete r;
}

extern "C" {

int32_t krex_version(void) { return 10000; }

const char *krex_status_string(krex_status s) {
    switch (s) {
    case KREX_OK: return "KREX_OK";
    case KREX_ERR_INVALID: return "KREX_ERR_INVALID";
    case KREX_ERR_UNSUPPORTED: return "KREX_ERR_UNSUPPORTED";
    case KREX_ERR_CUDA: return "KREX_ERR_CUDA";
    case KREX_ERR_STATE: return "KREX_ERR_STATE";
    case KREX_ERR_TIMEOUT: return "KREX_ERR_TIMEOUT";
    case KREX_ERR_DEVICE: return "KREX_ERR_DEVICE";
    }
    return "KREX_ERR_UNKNOWN";
}

const char *krex_last_error_string(void) { return t_err; }

uint64_t krex_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

krex_status krex_gen_inputs(uint64_t seed, uint32_t tensor_id, int32_t dist, float sigma, krex_buf out,
                            krex_stream_t stream) {
    krex_status st = check_buf(out, "out");
    if (st) return st;
    if (dist == KREX_DIST_UNIFORM_PM1) {
        if (out.dtype != KREX_BF16 && out.dtype != KREX_F16)
            return set_error(KREX_ERR_INVALID, "uniform inputs are bf16 or fp16");
    } else if (dist == KREX_DIST_NORMAL) {
        if (out.dtype != KREX_F32) return set_error(KREX_ERR_INVALID, "normal inputs are fp32");
        if (!std::isfinite(sigma)) return set_error(KREX_ERR_INVALID, "sigma must be finite");
    } else {
        return set_error(KREX_ERR_INVALID, "unknown distribution %d", dist);
    }
    if (out.rows * out.cols == 0) return ok();
    if (!aligned16(out.ptr)) return set_error(KREX_ERR_UNSUPPORTED, "out must be 16-byte aligned");
    const uint64_t key = stream_key(seed, tensor_id);
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (dist == KREX_DIST_UNIFORM_PM1)
        KREX_CUDA_TRY(launch_fill_uniform_16(key, out.dtype == KREX_F16, out.ptr, out.rows, out.cols, out.ld, s));
    else
        KREX_CUDA_TRY(launch_fill_normal_f32(key, sigma, static_cast<float *>(out.ptr), out.rows, out.cols, out.ld, s));
    count_launches(1);
    return ok();
}

krex_status krex_run_candidate(int32_t op, const krex_buf *in, int32_t n_in, krex_buf out, krex_stream_t stream) {
    krex_status st = check_op_shapes(op, in, n_in, out, op_dtype(op), "out");
    if (st) return st;
    return do_candidate(op, in, out, reinterpret_cast<cudaStream_t>(stream));
}

size_t krex_gemm_workspace_bytes(void) { return gemm_workspace_bytes(); }

krex_status krex_run_candidate_ws(int32_t op, const krex_buf *in, int32_t n_in, krex_buf out, void *workspace,
                                  size_t workspace_bytes, krex_stream_t stream) {
    krex_status st = check_op_shapes(op, in, n_in, out, op_dtype(op), "out");
    if (st) return st;
    if ((st = check_gemm_workspace(workspace, workspace_bytes))) return st;
    return do_candidate(op, in, out, reinterpret_cast<cudaStream_t>(stream), workspace, workspace_bytes);
}

krex_status krex_run_reference(int32_t op, const krex_buf *in, int32_t n_in, krex_buf ref, krex_stream_t stream) {
    krex_status st = check_op_shapes(op, in, n_in, ref, KREX_F32, "ref");
    if (st) return st;
    return do_reference(op, in, ref, reinterpret_cast<cudaStream_t>(stream));
}

krex_status krex_flush_l2(void *scratch, size_t bytes, krex_stream_t stream) {
    return do_flush(scratch, bytes, reinterpret_cast<cudaStream_t>(stream));
}

krex_status krex_l2_bytes(size_t *bytes) {
    if (!bytes) return set_error(KREX_ERR_INVALID, "bytes is null");
    int dev = 0;
    KREX_CUDA_TRY(cudaGetDevice(&dev));
    int a = 0;
    KREX_CUDA_TRY(cudaDeviceGetAttribute(&a, cudaDevAttrL2CacheSize, dev));
    *bytes = (size_t)a;
    return ok();
}

size_t krex_check_scratch_bytes(void) { return check_scratch_bytes(); }

krex_status krex_check_launch(krex_buf out, krex_buf ref, float atol, float rtol, void *dev_scratch,
                              size_t scratch_bytes, krex_stream_t stream) {
    krex_status st;
    if ((st = check_buf(out, "out")) || (st = check_buf(ref, "ref"))) return st;
    if (out.rows != ref.rows || out.cols != ref.cols) return set_error(KREX_ERR_INVALID, "out and ref shapes differ");
    if (!dev_scratch || scratch_bytes < check_scratch_bytes())
        return set_error(KREX_ERR_INVALID, "check scratch needs %zu bytes", check_scratch_bytes());
    if (!aligned16(dev_scratch)) return set_error(KREX_ERR_UNSUPPORTED, "check scratch must be 16-byte aligned");
    KREX_CUDA_TRY(launch_check(out.ptr, out.dtype, out.ld, ref.ptr, ref.dtype, ref.ld, out.rows, out.cols, atol, rtol,
                               dev_scratch, reinterpret_cast<cudaStream_t>(stream)));
    count_launches(1);
    return ok();
}

krex_status krex_check_fetch(const void *dev_scratch, krex_check_result *host_result, krex_stream_t stream) {
    if (!dev_scratch || !host_result) return set_error(KREX_ERR_INVALID, "check_fetch: null argument");
    krex_check_result r;
    krex_status st = read_check_header(dev_scratch, &r, reinterpret_cast<cudaStream_t>(stream));
    if (st) return st;
    *host_result = r;
    return ok();
}

krex_status krex_check_scratch_init(void *dev_scratch, size_t scratch_bytes, krex_stream_t stream) {
    if (!dev_scratch || scratch_bytes < check_scratch_bytes())
        return set_error(KREX_ERR_INVALID, "check scratch needs %zu bytes", check_scratch_bytes());
    if (!aligned16(dev_scratch)) return set_error(KREX_ERR_UNSUPPORTED, "check scratch must be 16-byte aligned");
    KREX_CUDA_TRY(init_check_scratch(dev_scratch, reinterpret_cast<cudaStream_t>(stream)));
    return ok();
}

krex_status krex_check(krex_buf out, krex_buf ref, float atol, float rtol, void *dev_scratch, size_t scratch_bytes,
                       krex_check_result *host_result, krex_stream_t stream) {
    if (!host_result) return set_error(KREX_ERR_INVALID, "host_result is null");
    krex_status st = krex_check_launch(out, ref, atol, rtol, dev_scratch, scratch_bytes, stream);
    if (st) return st;
    return krex_check_fetch(dev_scratch, host_result, stream);
}

krex_status krex_region_begin(krex_region **r, krex_stream_t stream, const krex_region_opts *opts) {
    if (!r || !opts) return set_error(KREX_ERR_INVALID, "region_begin: null argument");
    if (opts->max_iters < 1 || opts->max_iters > KREX_MAX_ITERS)
        return set_error(KREX_ERR_INVALID, "max_iters must be in [1, %d]", KREX_MAX_ITERS);
    if (opts->flush_on_entry && opts->flush_bytes > 0 && !opts->flush_scratch)
        return set_error(KREX_ERR_INVALID, "flush_on_entry needs flush_scratch");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    {
        std::lock_guard<std::mutex> lk(g_open_mu);
        if (open_streams().count(s)) return set_error(KREX_ERR_STATE, "a region is already open on this stream");
        open_streams().insert(s);
    }
    auto unmark = [&] {
        std::lock_guard<std::mutex> lk(g_open_mu);
        open_streams().erase(s);
    };
    // 0) optional gate: block and drain sibling tenants (Section 4.2 steps 1-3)
    uint64_t epoch = 0;
    if (opts->gate) {
        krex_status gst = krex_gate_enter(opts->gate, opts->tenant, opts->drain_timeout_us, &epoch);
        if (gst) {
            unmark();
            return gst;
        }
    }
    // 1) drain what is already queued: a failing entry starts nothing
    krex_status st = drain_stream(s, opts->drain_timeout_us);
    if (st) {
        if (opts->gate) krex_gate_exit(opts->gate, opts->tenant, epoch);
        unmark();
        return st;
    }
    krex_region *reg = new krex_region();
    reg->stream = s;
    reg->gate = opts->gate;
    reg->tenant = opts->tenant;
    reg->epoch = epoch;
    reg->max_iters = opts->max_iters;
    reg->n_begun = reg->n_ended = 0;
    reg->pinned = false;
    if (cudaGetDevice(&reg->device) != cudaSuccess) reg->device = 0;
    cudaError_t e = event_pool().take(reg->device, (size_t)2 * opts->max_iters, reg->ev);
    if (e != cudaSuccess) {
        region_release(reg);
        return cuda_error(e, "cudaEventCreate (region events)");
    }
    // 2) entry preparation: L2 flush, then pin the submitting thread
    if (opts->flush_on_entry && opts->flush_bytes > 0) {
        st = do_flush(opts->flush_scratch, opts->flush_bytes, s);
        if (st) {
            region_release(reg);
            return st;
        }
    }
    if (opts->pin_cpu) {
        int cpu = sched_getcpu();
        if (cpu >= 0 && pthread_getaffinity_np(pthread_self(), sizeof(cpu_set_t), &reg->old_mask) == 0) {
            cpu_set_t one;
            CPU_ZERO(&one);
            CPU_SET(cpu, &one);
            reg->pinned = pthread_setaffinity_np(pthread_self(), sizeof(cpu_set_t), &one) == 0;
        }
    }
    *r = reg;
    return ok();
}

krex_status krex_iter_begin(krex_region *r) {
    if (!r) return set_error(KREX_ERR_INVALID, "region is null");
    if (r->n_begun != r->n_ended) return set_error(KREX_ERR_STATE, "iter_begin twice without iter_end");
    if (r->n_begun >= r->max_iters) return set_error(KREX_ERR_INVALID, "more than max_iters=%d iterations", r->max_iters);
    KREX_CUDA_TRY(cudaEventRecord(r->ev[2 * r->n_begun], r->stream));
    ++r->n_begun;
    return ok();
}

krex_status krex_iter_end(krex_region *r) {
    if (!r) return set_error(KREX_ERR_INVALID, "region is null");
    if (r->n_ended + 1 != r->n_begun) return set_error(KREX_ERR_STATE, "iter_end without iter_begin");
    KREX_CUDA_TRY(cudaEventRecord(r->ev[2 * r->n_ended + 1], r->stream));
    ++r->n_ended;
    return ok();
}

krex_status krex_region_abort(krex_region *r) {
    if (!r) return set_error(KREX_ERR_INVALID, "region is null");
    cudaStreamSynchronize(r->stream);  // events may still be pending; drain before pooling them
    region_release(r);
    return ok();
}

krex_status krex_region_end(krex_region *r, float *durations_ms, int32_t cap, int32_t *n, double *p50_ms,
                            double *p95_ms) {
    if (!r) return set_error(KREX_ERR_INVALID, "region is null");
    if (n) *n = 0;
    if (p50_ms) *p50_ms = NAN;
    if (p95_ms) *p95_ms = NAN;
    if (r->n_begun != r->n_ended) {
        cudaStreamSynchronize(r->stream);
        region_release(r);
        return set_error(KREX_ERR_STATE, "region_end inside an iteration (iter_end missing)");
    }
    const int32_t iters = r->n_ended;
    std::vector<double> d;
    d.reserve(iters);
    krex_status st = KREX_OK;
    if (iters > 0) {
        cudaError_t e = cudaEventSynchronize(r->ev[2 * iters - 1]);
        if (e != cudaSuccess) st = cuda_error(e, "cudaEventSynchronize (region end)");
        for (int32_t i = 0; st == KREX_OK && i < iters; ++i) {
            float ms = 0.0f;
            e = cudaEventElapsedTime(&ms, r->ev[2 * i], r->ev[2 * i + 1]);
            if (e != cudaSuccess) {
                st = cuda_error(e, "cudaEventElapsedTime");
                break;
            }
            if (durations_ms && i < cap) durations_ms[i] = ms;
            d.push_back((double)ms);
        }
    }
    region_release(r);
    if (st) return st;
    if (n) *n = iters;
    if (!d.empty()) {
        std::sort(d.begin(), d.end());
        if (p50_ms) *p50_ms = percentile_sorted(d, 0.5);
        if (p95_ms) *p95_ms = percentile_sorted(d, 0.95);
    }
    return ok();
}

krex_status krex_bench_candidate(int32_t op, const krex_buf *in, int32_t n_in, krex_buf out,
                                 const krex_region_opts *opts, int32_t warmup, int32_t iters, float *durations_ms,
                                 double *p50_ms, double *p95_ms, void *workspace, size_t workspace_bytes,
                                 krex_stream_t stream) {
    if (!opts) return set_error(KREX_ERR_INVALID, "opts is null");
    if (warmup < 0 || iters < 0 || iters > opts->max_iters)
        return set_error(KREX_ERR_INVALID, "need 0 <= warmup and 0 <= iters <= max_iters");
    krex_status st = check_op_shapes(op, in, n_in, out, op_dtype(op), "out");
    if (st) return st;
    if ((st = check_gemm_workspace(workspace, workspace_bytes))) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    krex_region *r = nullptr;
    if ((st = krex_region_begin(&r, stream, opts))) return st;
    for (int32_t w = 0; w < warmup; ++w) {
        if ((st = do_flush(opts->flush_scratch, opts->flush_bytes, s)) ||
            (st = do_candidate(op, in, out, s, workspace, workspace_bytes))) {
            krex_region_abort(r);
            return st;
        }
    }
    for (int32_t i = 0; i < iters; ++i) {
        if ((st = do_flush(opts->flush_scratch, opts->flush_bytes, s)) || (st = krex_iter_begin(r)) ||
            (st = do_candidate(op, in, out, s, workspace, workspace_bytes)) || (st = krex_iter_end(r))) {
            krex_region_abort(r);
            return st;
        }
    }
    return krex_region_end(r, durations_ms, iters, nullptr, p50_ms, p95_ms);
}

// Host <-> device copy of `rows` rows of `width` bytes: one linear copy when
// the rows are packed on both sides, else a 2-D copy.
static cudaError_t copy_rows(void *dst, size_t dpitch, const void *src, size_t spitch, size_t width, size_t rows,
                             cudaMemcpyKind kind, cudaStream_t s) {
    if (dpitch == width && spitch == width) return cudaMemcpyAsync(dst, src, width * rows, kind, s);
    return cudaMemcpy2DAsync(dst, dpitch, src, spitch, width, rows, kind, s);
}

// The driver's cuPointerGetAttribute, through the runtime's entry-point query
// (the library links no driver library); nullptr if the driver lacks it.
typedef CUresult (*PointerAttrFn)(void *, CUpointer_attribute, CUdeviceptr);
static PointerAttrFn pointer_attr_fn() {
    static PointerAttrFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuPointerGetAttribute", &p, 4000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PointerAttrFn>(p);
    });
    return fn;
}

// True if the device can read all `bytes` at host address p directly, at the
// same address: page-locked memory mapped into the device's address space
// (cudaHostRegister / cudaHostAlloc) whose registered range covers the bytes.
// Anything else (pageable memory, a range that ends early, a device-side
// address that differs) is copied by the copy engine.
static bool device_reads_host(const void *p, size_t bytes) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (a.type != cudaMemoryTypeHost || a.devicePointer != p) return false;
    PointerAttrFn get = pointer_attr_fn();
    if (!get) return false;
    CUdeviceptr start = 0;
    size_t size = 0;
    const CUdeviceptr at = reinterpret_cast<CUdeviceptr>(p);
    if (get(&start, CU_POINTER_ATTRIBUTE_RANGE_START_ADDR, at) != CUDA_SUCCESS ||
        get(&size, CU_POINTER_ATTRIBUTE_RANGE_SIZE, at) != CUDA_SUCCESS)
        return false;
    return at >= start && bytes <= size && at - start <= size - bytes;
}

// Rows from a caller's host buffer into device memory: SM loads when the
// device reads the buffer directly (see host_copy.cu for why), else the copy
// engine.  *kernel counts the launches.
static cudaError_t copy_rows_in(void *dst, size_t dpitch, const void *src, size_t spitch, size_t width, size_t rows,
                                cudaStream_t s, int *kernel) {
    if (rows > 0 && width > 0 && device_reads_host(src, spitch * (rows - 1) + width)) {
        bool launched = false;
        cudaError_t e = launch_copy_rows_from_host(src, spitch, dst, dpitch, width, rows, s, &launched);
        if (e != cudaSuccess || launched) {
            *kernel += e == cudaSuccess;
            return e;
        }
    }
    return copy_rows(dst, dpitch, src, spitch, width, rows, cudaMemcpyHostToDevice, s);
}

krex_status krex_command_run(const krex_command *cmd, const krex_command_bufs *bufs, const void *const *host_in,
                             void *host_out, float *durations_ms, krex_command_result *result,
                             krex_stream_t stream) {
    using clk = std::chrono::steady_clock;
    if (!cmd || !bufs || !result) return set_error(KREX_ERR_INVALID, "command: null argument");
    if (cmd->iters < 1 || cmd->iters > KREX_MAX_ITERS || cmd->warmup < 0)
        return set_error(KREX_ERR_INVALID, "command: iters must be in [1, %d], warmup >= 0", KREX_MAX_ITERS);
    const int32_t op = cmd->op;
    const int n_in = is_gemm(op) ? 2 : 1;
    krex_status st = check_op_shapes(op, bufs->in, n_in, bufs->out, op_dtype(op), "out");
    if (st) return st;
    if ((st = check_op_shapes(op, bufs->in, n_in, bufs->ref, KREX_F32, "ref"))) return st;
    if (is_gemm(op)) {
        if (bufs->in[0].rows != cmd->M || bufs->in[0].cols != cmd->K || bufs->in[1].cols != cmd->N)
            return set_error(KREX_ERR_INVALID, "command: buffers do not match M, N, K");
    } else if (bufs->in[0].rows != cmd->M || bufs->in[0].cols != cmd->N) {
        return set_error(KREX_ERR_INVALID, "command: buffers do not match rows M, cols N");
    }
    if (cmd->flush_bytes > 0 && !bufs->flush_scratch) return set_error(KREX_ERR_INVALID, "command: flush scratch is null");
    if (krex_status st0 = check_gemm_workspace(bufs->gemm_workspace, bufs->gemm_workspace_bytes)) return st0;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    memset(result, 0, sizeof(*result));
    const uint64_t launches0 = g_launches.load();
    auto ms_since = [](clk::time_point t) {
        return std::chrono::duration<double, std::milli>(clk::now() - t).count();
    };

    // Phases 1-4 run back to back on the stream and are timed with events
    // between them (a host synchronisation per phase would add an idle gap to
    // each); the check ends by reading its verdict back to the host, and its
    // phase ends with an event recorded after that.  The timed loop is host
    // wall time.  The candidate's checked run comes before the reference, so
    // that with host_out its output (the command's result) is copied back on a
    // side stream while the reference runs; the copy is complete before the
    // timed region starts, so nothing overlaps the measurement.
    int dev = 0;
    KREX_CUDA_TRY(cudaGetDevice(&dev));
    std::vector<cudaEvent_t> pev;
    KREX_CUDA_TRY(event_pool().take(dev, 6, pev));
    struct Cleanup {
        int dev;
        std::vector<cudaEvent_t> &ev;
        cudaStream_t side = nullptr;
        ~Cleanup() {
            if (side) {
                cudaStreamSynchronize(side);  // a copy in flight finishes before anything is released
                cudaStreamDestroy(side);
            }
            event_pool().give(dev, ev);
        }
    } cleanup{dev, pev};
    KREX_CUDA_TRY(cudaEventRecord(pev[0], s));
    // 1) inputs: generated on the device, or copied from the caller's host buffers
    for (int i = 0; i < n_in; ++i) {
        const krex_buf &b = bufs->in[i];
        if (host_in && host_in[i]) {
            const size_t es = elem_size(b.dtype);
            int kernels = 0;
            KREX_CUDA_TRY(copy_rows_in(b.ptr, (size_t)b.ld * es, host_in[i], (size_t)b.cols * es,
                                       (size_t)b.cols * es, (size_t)b.rows, s, &kernels));
            count_launches(kernels);
        } else {
            st = is_gemm(op)
                     ? krex_gen_inputs(cmd->seed, (uint32_t)i, KREX_DIST_UNIFORM_PM1, 0.0f, b, stream)
                     : krex_gen_inputs(cmd->seed, 0u, KREX_DIST_NORMAL, cmd->sigma, b, stream);
            if (st) return st;
        }
    }
    KREX_CUDA_TRY(cudaEventRecord(pev[1], s));
    // 2) candidate once, for the check
    if ((st = do_candidate(op, bufs->in, bufs->out, s, bufs->gemm_workspace, bufs->gemm_workspace_bytes))) return st;
    KREX_CUDA_TRY(cudaEventRecord(pev[2], s));
    if (host_out) {
        // the result back to the host while the reference runs
        KREX_CUDA_TRY(cudaStreamCreateWithFlags(&cleanup.side, cudaStreamNonBlocking));
        KREX_CUDA_TRY(cudaStreamWaitEvent(cleanup.side, pev[2], 0));
        const krex_buf &b = bufs->out;
        const size_t es = elem_size(b.dtype);
        KREX_CUDA_TRY(copy_rows(host_out, (size_t)b.cols * es, b.ptr, (size_t)b.ld * es, (size_t)b.cols * es,
                                (size_t)b.rows, cudaMemcpyDeviceToHost, cleanup.side));
        KREX_CUDA_TRY(cudaEventRecord(pev[5], cleanup.side));
    }
    // 3) reference
    if ((st = do_reference(op, bufs->in, bufs->ref, s))) return st;
    KREX_CUDA_TRY(cudaEventRecord(pev[3], s));
    // 4) check (synchronous: every earlier phase on the stream has completed when it returns)
    if ((st = krex_check(bufs->out, bufs->ref, cmd->atol, cmd->rtol, bufs->check_scratch, bufs->check_scratch_bytes,
                         &result->check, stream)))
        return st;
    KREX_CUDA_TRY(cudaEventRecord(pev[4], s));
    KREX_CUDA_TRY(cudaEventSynchronize(pev[4]));
    {
        float ms = 0.0f;
        KREX_CUDA_TRY(cudaEventElapsedTime(&ms, pev[0], pev[1]));
        result->phase_ms[0] = ms;  // inputs
        KREX_CUDA_TRY(cudaEventElapsedTime(&ms, pev[2], pev[3]));
        result->phase_ms[1] = ms;  // reference
        KREX_CUDA_TRY(cudaEventElapsedTime(&ms, pev[1], pev[2]));
        result->phase_ms[2] = ms;  // candidate
        KREX_CUDA_TRY(cudaEventElapsedTime(&ms, pev[3], pev[4]));
        result->phase_ms[3] = ms;  // check
    }
    if (host_out) KREX_CUDA_TRY(cudaEventSynchronize(pev[5]));  // the copy back is done
    result->passed = result->check.n_violations == 0;
    // 5) timed loop inside a critical region (skipped when the check failed)
    const auto t = clk::now();
    result->p50_ms = result->p95_ms = NAN;
    if (result->passed) {
        krex_region_opts o;
        memset(&o, 0, sizeof(o));
        o.max_iters = cmd->iters;
        o.flush_on_entry = cmd->flush_bytes > 0;
        o.pin_cpu = cmd->pin_cpu;
        o.drain_timeout_us = cmd->drain_timeout_us;
        o.flush_scratch = bufs->flush_scratch;
        o.flush_bytes = cmd->flush_bytes;
        if ((st = krex_bench_candidate(op, bufs->in, n_in, bufs->out, &o, cmd->warmup, cmd->iters, durations_ms,
                                       &result->p50_ms, &result->p95_ms, bufs->gemm_workspace,
                                       bufs->gemm_workspace_bytes, stream)))
            return st;
        result->n_iters = cmd->iters;
    }
    result->phase_ms[4] = ms_since(t);
    result->launches = (int32_t)(g_launches.load() - launches0);
    return ok();
}

krex_status krex_percentile(const float *x, int32_t n, double q, double *out) {
    if (!x || !out || n < 1) return set_error(KREX_ERR_INVALID, "percentile: need x, out and n >= 1");
    if (!(q >= 0.0 && q <= 1.0)) return set_error(KREX_ERR_INVALID, "percentile: q must be in [0, 1]");
    std::vector<double> d(x, x + n);
    std::sort(d.begin(), d.end());
    *out = percentile_sorted(d, q);
    return ok();
}

krex_status krex_device_status(uint32_t *code) {
    if (!code) return set_error(KREX_ERR_INVALID, "code is null");
    KREX_CUDA_TRY(read_and_clear_device_status(code));
    if (*code) return set_error(KREX_ERR_DEVICE, "a kernel's bounded wait ran out (status 0x%x)", *code);
    return ok();
}

krex_status krex_device_status_detail(uint64_t *words) {
    if (!words) return set_error(KREX_ERR_INVALID, "words is null");
    unsigned long long w[8];
    KREX_CUDA_TRY(read_device_status_detail(w));
    for (int i = 0; i < 8; ++i) words[i] = (uint64_t)w[i];
    return ok();
}

struct HoldArg {
    volatile int32_t *gate;
    int32_t hold_ms;
};

static void CUDART_CB hold_fn(void *p) {
    HoldArg *a = static_cast<HoldArg *>(p);
    const auto t0 = std::chrono::steady_clock::now();
    while (*a->gate == 0) {
        if (std::chrono::steady_clock::now() - t0 > std::chrono::milliseconds(a->hold_ms)) break;
        struct timespec ts = {0, 100000};
        nanosleep(&ts, nullptr);
    }
    delete a;
}

// Host buffers: anonymous mappings aligned to the transparent huge-page size
// (read from the kernel, 2 MiB if it does not say), advised to use huge pages,
// zero-filled (which allocates the pages), then registered with CUDA.  The
// mapping is over-allocated by one alignment and trimmed, so krex_host_free
// unmaps exactly [ptr, ptr + rounded bytes).
static size_t host_huge_page_bytes() {
    static const size_t v = [] {
        size_t b = 0;
        if (FILE *f = fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
            unsigned long long x = 0;
            if (fscanf(f, "%llu", &x) == 1) b = (size_t)x;
            fclose(f);
        }
        if (b < ((size_t)2 << 20) || b > ((size_t)1 << 30) || (b & (b - 1))) b = (size_t)2 << 20;
        return b;
    }();
    return v;
}

static size_t host_rounded(size_t bytes) {
    const size_t a = host_huge_page_bytes();
    return (bytes + a - 1) / a * a;
}

krex_status krex_host_alloc(size_t bytes, void **ptr) {
    if (!ptr || bytes == 0 || bytes > ((size_t)1 << 46)) return set_error(KREX_ERR_INVALID, "host_alloc: bad arguments");
    *ptr = nullptr;
    const size_t align = host_huge_page_bytes(), len = host_rounded(bytes);
    void *raw = mmap(nullptr, len + align, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
    if (raw == MAP_FAILED) return set_error(KREX_ERR_INVALID, "host_alloc: mmap of %zu bytes failed", len + align);
    const uintptr_t r = reinterpret_cast<uintptr_t>(raw);
    const uintptr_t a = (r + align - 1) / align * align;
    if (a > r) munmap(raw, a - r);
    if (r + len + align > a + len) munmap(reinterpret_cast<void *>(a + len), r + len + align - (a + len));
    void *p = reinterpret_cast<void *>(a);
#ifdef MADV_HUGEPAGE
    madvise(p, len, MADV_HUGEPAGE);  // advice only: without it the buffer still works
#endif
    memset(p, 0, len);
    cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterDefault);
    if (e != cudaSuccess) {
        munmap(p, len);
        return cuda_error(e, "cudaHostRegister (host_alloc)");
    }
    *ptr = p;
    return ok();
}

krex_status krex_host_free(void *ptr, size_t bytes) {
    if (!ptr || bytes == 0) return set_error(KREX_ERR_INVALID, "host_free: bad arguments");
    const size_t len = host_rounded(bytes);
    cudaError_t e = cudaHostUnregister(ptr);
    munmap(ptr, len);
    if (e != cudaSuccess) return cuda_error(e, "cudaHostUnregister (host_free)");
    return ok();
}

krex_status krex_probe_generator(int32_t dist, uint64_t n_elements, int32_t blocks, float sigma, void *dev_sink,
                                 krex_stream_t stream) {
    if (dist != KREX_DIST_UNIFORM_PM1 && dist != KREX_DIST_NORMAL)
        return set_error(KREX_ERR_INVALID, "probe: bad distribution %d", dist);
    if (!dev_sink || blocks < 1 || n_elements == 0 || n_elements % 8 || n_elements > ((uint64_t)1 << 50))
        return set_error(KREX_ERR_INVALID, "probe: need a sink, blocks >= 1, n_elements a positive multiple of 8");
    KREX_CUDA_TRY(launch_generator_probe(dist, 0x243F6A8885A308D3ull, (int64_t)n_elements, sigma, blocks,
                                         static_cast<uint32_t *>(dev_sink), reinterpret_cast<cudaStream_t>(stream)));
    count_launches(1);
    return ok();
}

krex_status krex_probe_fma(int32_t iters, int32_t blocks, void *dev_sink, krex_stream_t stream) {
    if (!dev_sink || blocks < 1 || iters < 1)
        return set_error(KREX_ERR_INVALID, "probe_fma: need a sink, blocks >= 1, iters >= 1");
    KREX_CUDA_TRY(launch_fma_probe(iters, blocks, static_cast<float *>(dev_sink),
                                   reinterpret_cast<cudaStream_t>(stream)));
    count_launches(1);
    return ok();
}

void krex_tuning_defaults(krex_tuning *t) {
    if (t) *t = default_tuning();
}

krex_status krex_set_tuning(const krex_tuning *t) {
    const krex_tuning v = t ? *t : default_tuning();
    if (!tuning_valid(v)) return set_error(KREX_ERR_INVALID, "set_tuning: a field is out of its range");
    std::lock_guard<std::mutex> lk(g_tuning_mu);
    g_tuning = v;
    return ok();
}

krex_status krex_get_tuning(krex_tuning *t) {
    if (!t) return set_error(KREX_ERR_INVALID, "get_tuning: null argument");
    *t = tuning_snapshot();
    return ok();
}

krex_status krex_debug_stall_handover(int32_t on) {
    set_debug_stall_handover(on != 0);
    return ok();
}

krex_status krex_debug_hold_stream(krex_stream_t stream, volatile int32_t *gate, int32_t hold_ms) {
    if (!gate || hold_ms < 0 || hold_ms > 60000) return set_error(KREX_ERR_INVALID, "hold: bad gate or hold_ms");
    HoldArg *a = new HoldArg{gate, hold_ms};
    cudaError_t e = cudaLaunchHostFunc(reinterpret_cast<cudaStream_t>(stream), hold_fn, a);
    if (e != cudaSuccess) {
        delete a;
        return cuda_error(e, "cudaLaunchHostFunc");
    }
    return ok();
}

}  // extern "C"
