/*
 * krex.h — C ABI of the GB300 benchmarking-command data path.
 *
 * A kernel benchmarking command generates seeded inputs, runs a reference,
 * runs the candidate once and checks it against the reference, and finally
 * times the candidate in a loop of warm-up and timed launches, flushing L2
 * between iterations and summarising the durations (paper Section 2.1,
 * "Kernel agent" and "Benchmarking command"; Section 1).  Only the timed loop
 * needs the GPU to itself; the paper brackets it with a critical region
 * (Section 4.1, region.critical()) whose entry drains outstanding work,
 * flushes L2 and pins the submitting thread (Section 4.2, "Region entry and
 * exit", step 5).  This library is the data-parallel GPU work of one such
 * command on one GPU, plus the region's single-process form.
 *
 * Conventions (all entry points):
 *  - Every function returns a krex_status; nothing throws or aborts.  On
 *    failure krex_last_error_string() (thread-local) describes the cause.
 *  - Arguments are validated before any CUDA call; an invalid argument
 *    returns KREX_ERR_INVALID and launches nothing.
 *  - Device memory is owned by the caller (e.g. allocated with PyTorch).  The
 *    library allocates no device memory.  It owns only the CUDA events of a
 *    region, which krex_region_end / krex_region_abort release.
 *  - Work is enqueued on the given stream (a cudaStream_t; NULL means the
 *    legacy default stream) and is asynchronous, except where a function says
 *    it synchronises.
 *  - A sticky CUDA error is reported as KREX_ERR_CUDA and never hidden.
 *  - Matrices are row-major: element (r, c) is at ptr + (r*ld + c)*elem_size.
 */
#ifndef KREX_H
#define KREX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; declared here so callers need no CUDA headers. */
typedef struct CUstream_st *krex_stream_t;

typedef enum {
    KREX_OK = 0,
    KREX_ERR_INVALID = 1,      /* bad argument (null pointer, bad dtype/shape, size mismatch) */
    KREX_ERR_UNSUPPORTED = 2,  /* valid but not implemented (alignment, ld, shape class) */
    KREX_ERR_CUDA = 3,         /* a CUDA runtime/driver call failed */
    KREX_ERR_STATE = 4,        /* call out of order (region misuse) */
    KREX_ERR_TIMEOUT = 5,      /* a bounded wait ran out (region drain) */
    KREX_ERR_DEVICE = 6        /* a kernel reported an error through its status word */
} krex_status;

typedef enum { KREX_BF16 = 1, KREX_F32 = 2, KREX_F16 = 3 } krex_dtype;

typedef enum {
    KREX_DIST_UNIFORM_PM1 = 0, /* U[-1,1] rounded to bf16 or binary16 (out KREX_BF16 or KREX_F16) */
    KREX_DIST_NORMAL = 1       /* N(0, sigma^2) in fp32 (out must be KREX_F32)                     */
} krex_dist;

typedef enum {
    KREX_OP_GEMM_BF16 = 0,     /* C[MxN] = A[MxK] B[KxN]; bf16 in, fp32 accumulate, bf16 out */
    KREX_OP_SOFTMAX_F32 = 1,   /* Y = row softmax of X, fp32                                  */
    KREX_OP_GEMM_F16 = 2       /* the same GEMM with IEEE binary16 A, B and C                 */
} krex_op;

/* A caller-owned device matrix.  dtype is a krex_dtype; ld >= cols, in elements. */
typedef struct {
    void *ptr;
    int32_t dtype;
    int32_t reserved;
    int64_t rows, cols, ld;
} krex_buf;

/* Result of krex_check.  max_abs_err is the largest |out - ref| (compared by
 * IEEE bit pattern, so a NaN difference dominates; 0 for empty inputs). */
typedef struct {
    float max_abs_err;
    uint32_t reserved;
    uint64_t n_violations;
} krex_check_result;

/* Options of a critical region (paper Section 4.1 region.critical(); entry
 * preparation of Section 4.2 step 5).
 *   max_iters        capacity for timed iterations (1 .. KREX_MAX_ITERS)
 *   drain_timeout_us how long region_begin may wait for the stream to drain
 *                    (<= 0: 10 s)
 *   flush_on_entry   nonzero: write flush_bytes of flush_scratch after the
 *                    drain (the L2 flush of region entry)
 *   pin_cpu          nonzero: pin the calling thread to the core it runs on
 *                    for the region's lifetime, restored at region end
 *   flush_scratch    device buffer of >= flush_bytes (needed if flush_on_entry)
 *   gate, tenant     optional (gate may be NULL): region entry first enters the
 *                    gate as holder `tenant` (sibling tenants drained and
 *                    blocked, see krex_gate_enter); region end/abort exits it
 */
typedef struct krex_gate krex_gate; /* opaque; see the gate section below */

typedef struct {
    int32_t max_iters;
    int32_t flush_on_entry;
    int32_t pin_cpu;
    int32_t reserved;
    int64_t drain_timeout_us;
    void *flush_scratch;
    size_t flush_bytes;
    krex_gate *gate;           /* optional: enter this gate as `tenant` before the drain */
    int32_t tenant;
    int32_t reserved2;
} krex_region_opts;

#define KREX_MAX_ITERS 100000

typedef struct krex_region krex_region; /* opaque; created by begin, released by end/abort */

/* ----------------------------------------------------------- inputs ------ */

/* Seeded input generation (Section 2.1: a command generates its inputs before
 * the check and the timed loop).  Element e = r*cols + c of `out` (logical
 * row-major index) is element e of the counter-based stream
 *   key = mix64(seed + (tensor_id+1)*G), draw j = mix64(key + (j+1)*G),
 * G = 0x9E3779B97F4A7C15, mix64 = the SplitMix64 output mix.
 * KREX_DIST_UNIFORM_PM1: elements 2j, 2j+1 take bits 63..40 and 31..8 of draw
 * j; b -> (b - 2^23) 2^-23 rounded to bf16 (RNE; to IEEE binary16 with
 * subnormals, RNE, when out is KREX_F16).  KREX_DIST_NORMAL: pair j is
 * a Box-Muller pair from draw j (u1 = (hi24+1) 2^-24, u2 = lo24 2^-24) scaled by
 * sigma, in fp32.  Output is bit-identical for any launch shape.
 * Errors: INVALID for a null/empty-but-nonzero buffer, dtype/dist mismatch,
 * ld < cols, sigma not finite; UNSUPPORTED if ptr is not 16-byte aligned.
 * Asynchronous. */
krex_status krex_gen_inputs(uint64_t seed, uint32_t tensor_id, int32_t dist, float sigma,
                            krex_buf out, krex_stream_t stream);

/* ------------------------------------------------------- candidate ------- */

/* The timed candidate (Section 2.1, Figure 1a's GEMM benchmarking command).
 * KREX_OP_GEMM_BF16: in[0] = A (M x K, bf16), in[1] = B (K x N, bf16), out = C
 *   (M x N, bf16, RNE from the fp32 accumulator).  tcgen05 tensor cores with
 *   TMEM accumulators, TMA loads; pair tiles of 256 x 256, or 256 x 512 for
 *   long-K GEMMs (krex_tuning.gemm_pair_tile_n).  Needs K, N, lda, ldb
 *   multiples of 8 and 16-byte aligned A, B (TMA), else UNSUPPORTED.  K = 0
 *   gives C = 0.
 * KREX_OP_GEMM_F16: the same with IEEE binary16 A, B and C (RNE out).
 * KREX_OP_SOFTMAX_F32: in[0] = X (rows x cols, fp32), out = Y (same shape,
 *   fp32); y = exp(x - max) / sum exp(x - max) per row, one HBM pass.
 * Errors: INVALID for wrong n_in, dtypes or shapes; DEVICE if the kernel's
 * bounded waits ran out (reported by a later krex_device_status call).
 * Asynchronous. */
krex_status krex_run_candidate(int32_t op, const krex_buf *in, int32_t n_in, krex_buf out,
                               krex_stream_t stream);

/* Bytes of the optional GEMM workspace (16 MiB + 4 KiB). */
size_t krex_gemm_workspace_bytes(void);

/* krex_run_candidate with an optional GEMM workspace (device memory of >=
 * krex_gemm_workspace_bytes(), 16-byte aligned, zero-filled before its first
 * use; may be NULL).  With it, the 256-wide tiles of a GEMM that is one
 * partial wave are split into two K halves whose fp32 partial sums meet in
 * the workspace (the kernel leaves it ready for the next call); otherwise the
 * tiles of a final partial wave are split into column halves (256-wide tiles
 * only).  One workspace per GEMM in flight: calls that overlap on the
 * GPU must not share it.  After a KREX_ERR_DEVICE status, zero it again.
 * Other ops ignore the workspace.  Asynchronous. */
krex_status krex_run_candidate_ws(int32_t op, const krex_buf *in, int32_t n_in, krex_buf out,
                                  void *workspace, size_t workspace_bytes, krex_stream_t stream);

/* The reference the check compares against (Section 2.1: the command checks
 * its result against a reference implementation).  CUDA cores only, fp32
 * accumulation and fp32 output: GEMM ref = fp32 M x N; softmax ref = fp32,
 * computed in three passes (max, sum, write).  Same shapes and errors as
 * krex_run_candidate, except that ref must be KREX_F32. Asynchronous. */
krex_status krex_run_reference(int32_t op, const krex_buf *in, int32_t n_in, krex_buf ref,
                               krex_stream_t stream);

/* ---------------------------------------------------------- L2 flush ----- */

/* The L2 flush between timed iterations (Section 2.1: harnesses often flush
 * L2 between iterations; Section 4.2 step 5: region entry flushes L2 with a
 * write over an L2-sized buffer).  Writes `bytes` bytes of `scratch` (device,
 * 16-byte aligned); each call writes a different value so no write can be
 * elided.  bytes = 0 is a no-op.  Asynchronous. */
krex_status krex_flush_l2(void *scratch, size_t bytes, krex_stream_t stream);

/* Bytes of L2 on the current device (cudaDevAttrL2CacheSize). */
krex_status krex_l2_bytes(size_t *bytes);

/* ------------------------------------------------------------- check ----- */

/* Bytes of device scratch krex_check needs (at least 16-byte aligned). */
size_t krex_check_scratch_bytes(void);

/* Make a check scratch ready for its first use: zeroes its
 * krex_check_scratch_bytes() bytes on `stream` (asynchronous).  Equivalent to
 * allocating the scratch zero-filled.  Needed once per scratch buffer; every
 * check leaves the scratch ready for the next one (the next call's result slot
 * cleared, its ticket re-armed), so no per-call reset runs in front of the
 * check kernel.  Errors: INVALID for a null or small scratch, UNSUPPORTED if
 * it is not 16-byte aligned. */
krex_status krex_check_scratch_init(void *dev_scratch, size_t scratch_bytes, krex_stream_t stream);

/* The correctness check (Section 2.1: check against the reference, return a
 * verdict).  Per element, in IEEE fp32 without fused multiply-add:
 *   d = |out - ref|, violation iff !(d <= atol + rtol*|ref|)  (NaN counts).
 * out may be bf16 or fp32 (widened exactly); ref is fp32 or bf16.  Shapes must
 * match.  dev_scratch: caller-owned device memory of >= krex_check_scratch_bytes()
 * bytes that were zeroed once before its first check (zero-filled allocation
 * or krex_check_scratch_init) and have since been used only by checks; one
 * check at a time per scratch.  SYNCHRONISES `stream` and writes
 * *host_result.  The result is bit-identical for any launch shape (max and
 * count are exact).  Errors: INVALID for null pointers, shape/dtype mismatch,
 * small scratch; STATE if the scratch shows it was not ready (never
 * zeroed, or written by something else since): no result is returned then. */
krex_status krex_check(krex_buf out, krex_buf ref, float atol, float rtol, void *dev_scratch,
                       size_t scratch_bytes, krex_check_result *host_result,
                       krex_stream_t stream);

/* The check in two halves, for callers that overlap it with other work:
 * krex_check_launch enqueues the compare-and-reduce on `stream` and leaves the
 * result in dev_scratch (asynchronous; same arguments and errors as
 * krex_check); krex_check_fetch copies that result to *host_result and
 * SYNCHRONISES `stream`.  krex_check = launch + fetch. */
krex_status krex_check_launch(krex_buf out, krex_buf ref, float atol, float rtol, void *dev_scratch,
                              size_t scratch_bytes, krex_stream_t stream);
krex_status krex_check_fetch(const void *dev_scratch, krex_check_result *host_result,
                             krex_stream_t stream);

/* krex_check without caller scratch, for callers that cannot allocate device
 * memory: code whose device memory belongs to another allocator with nothing
 * to spare (a framework's caching pool, a fixed budget), and timing harnesses
 * that must not call cudaMalloc/cudaFree because those calls can synchronise
 * the device and disturb a measurement.  The paper has no counterpart; it is
 * an addition of this library.
 * Scratch: a static device array of 33,024 bytes inside libkrex.so, present on
 * every GPU that loads the library until the process exits.  The first call on
 * a device (and the first after that device's context was destroyed and
 * created again) does the set-up there: it resolves the array's address
 * (cudaGetSymbolAddress) and zeroes the check's scratch in it on `stream`;
 * make that first call before any stream capture.  It allocates nothing and
 * calls no allocating routine.  Every call shares the one array per device and
 * leaves the last result in it; the call clears what must start at zero, but
 * calls that overlap on the GPU (other streams, other threads) race on it, so
 * serialise them.  Same arguments, result and bit-exact semantics as
 * krex_check; UNSUPPORTED if the check ever needed more scratch than the
 * array holds.  SYNCHRONISES `stream`. */
krex_status krex_check_noalloc(krex_buf out, krex_buf ref, float atol, float rtol,
                               krex_check_result *host_result, krex_stream_t stream);

/* ------------------------------------------------------------ region ----- */

/* Enter a critical region on `stream` (Section 4.1; Section 4.2 step 5).
 * Drains the stream: polls cudaStreamQuery, spinning briefly and then
 * sleeping (the spin-park policy of Section 4.3), until it is idle or
 * drain_timeout_us passes (-> KREX_ERR_TIMEOUT; nothing is started and no
 * region is created: a failing entry never starts measurement, Section 4.2).
 * Then optionally flushes L2 and pins the thread.  The region owns 2*max_iters
 * CUDA events (pooled across regions).  One region per stream at a time:
 * begin on a stream that already has an open region returns KREX_ERR_STATE.
 * *r is set only on success. */
krex_status krex_region_begin(krex_region **r, krex_stream_t stream, const krex_region_opts *opts);

/* Record the start / end event of the next timed iteration on the region's
 * stream.  Must alternate begin, end; STATE on misuse; INVALID past max_iters. */
krex_status krex_iter_begin(krex_region *r);
krex_status krex_iter_end(krex_region *r);

/* Leave the region: synchronise the last event, read each iteration's
 * duration (cudaEventElapsedTime, ms), sort a copy and report p50 and p95 by
 * linear interpolation between order statistics; unpin the thread; release
 * the region.  durations_ms (may be NULL) receives min(n, cap) durations in
 * iteration order; *n (may be NULL) the number of timed iterations; p50/p95
 * (may be NULL) are NaN if there were none.  The region is released even when
 * an error is returned. */
krex_status krex_region_end(krex_region *r, float *durations_ms, int32_t cap, int32_t *n,
                            double *p50_ms, double *p95_ms);

/* Release a region without reading its timings (error paths). */
krex_status krex_region_abort(krex_region *r);

/* -------------------------------------------------- in-region gate ----- */

/* The in-process form of the paper's in-region GPU exclusivity (Section 4.2,
 * "GPU exclusivity", steps 1-3 and 8).  Tenants are submitting threads, each
 * with the stream its GPU work goes to.  Host-side only: a tenant brackets
 * every submission with submit_begin/submit_end; a holder's gate_enter blocks
 * new sibling submissions and drains the outstanding ones before returning.
 * Timeouts are in microseconds (<= 0: 10 s).  Thread-safe. */

/* Create / destroy a gate with up to max_tenants tenants (1..4096).  Destroy
 * fails with STATE while a holder is inside. */
krex_status krex_gate_create(krex_gate **gate, int32_t max_tenants);
krex_status krex_gate_destroy(krex_gate *gate);

/* Register a tenant whose work goes to `stream` (NULL: nothing to synchronise
 * in the drain).  Registration is serialised with gate closure: while a holder
 * is inside, it waits for the gate to reopen (TIMEOUT after timeout_us). */
krex_status krex_gate_register(krex_gate *gate, krex_stream_t stream, int64_t timeout_us,
                               int32_t *tenant);
/* STATE if the tenant holds the gate or has a submission open. */
krex_status krex_gate_unregister(krex_gate *gate, int32_t tenant);

/* Counter-and-gate (Section 4.2): increment the tenant's in-flight counter,
 * then check the gate; if another tenant holds it, retract the increment and
 * park until it reopens (TIMEOUT after timeout_us).  On OK the caller issues
 * its GPU work, then calls submit_end, also when the work failed. */
krex_status krex_gate_submit_begin(krex_gate *gate, int32_t tenant, int64_t timeout_us);
krex_status krex_gate_submit_end(krex_gate *gate, int32_t tenant);

/* Enter as holder (steps 1-3): take the region lock, claim the gate with a new
 * epoch (*epoch), then for every sibling wait for its in-flight counter to
 * reach zero, synchronise its stream and acknowledge the epoch.  Returns only
 * when every sibling shows this epoch's acknowledgement and a zero counter
 * (polled: a submission bouncing off the closed gate raises a counter for a
 * moment).  On TIMEOUT
 * or a CUDA error the gate is reopened and the lock released: a failing entry
 * never starts measurement.  STATE if the caller already holds the gate. */
krex_status krex_gate_enter(krex_gate *gate, int32_t holder, int64_t timeout_us, uint64_t *epoch);

/* Exit (step 8), bound to the holder and the epoch of its entry: wait for the
 * holder's own submissions to finish host-side, reopen the gate (parked
 * tenants resume), release the region lock.  STATE for a stale holder/epoch. */
krex_status krex_gate_exit(krex_gate *gate, int32_t holder, uint64_t epoch);

/* Current holder (-1 = open), last epoch, and number of parked submitters. */
krex_status krex_gate_state(krex_gate *gate, int32_t *holder, uint64_t *epoch, int32_t *parked);

/* ------------------------------------------- cross-process gate -------- */

/* The same gate with its state in shared memory, so that tenants in several
 * processes take part (Section 4.2: region lock, gate with holder and epoch,
 * per-tenant in-flight counters, registration serialised with closure,
 * drainer threads that acknowledge the epoch; Section 4.2 "Region entry and
 * exit": a participant's death fails the entry, a dead holder's gate is
 * reclaimed bound to holder and epoch).  Host-side only.
 *
 * `mem` is caller-owned shared memory (for example a POSIX shared-memory
 * object or a file mapped MAP_SHARED by every participant), 64-byte aligned,
 * of at least krex_gate_shared_bytes(max_tenants) bytes; it holds only
 * address-free atomics, so each process may map it anywhere.  One process
 * formats it with krex_gate_shared_init before any process attaches. */
size_t krex_gate_shared_bytes(int32_t max_tenants);
krex_status krex_gate_shared_init(void *mem, size_t bytes, int32_t max_tenants);

/* Attach this process to a formatted gate.  The returned handle works with
 * every krex_gate_* call above and as krex_region_opts.gate; tenants it
 * registers belong to this process (their streams are drained by this
 * process's drainer thread, started here).  krex_gate_destroy detaches: the
 * drainer stops, this process's tenants finish their stream work and leave
 * (STATE while one of them holds the gate); the shared memory is untouched.
 * In this form: unregister is refused (STATE) while another tenant holds the
 * gate, so drained entries stay until the region ends; registration and
 * entry free the slots of tenants whose process no longer exists; an entry
 * fails with STATE when a sibling's process dies while it is being drained,
 * and with CUDA when a sibling's stream synchronisation fails. */
krex_status krex_gate_shared_attach(void *mem, size_t bytes, krex_gate **gate);

/* Reclaim a gate whose holder died inside (the dispatcher's recovery of
 * Section 4.2): if `holder` still holds it with `epoch` and the holder's
 * process no longer exists, free the holder's slot, reopen the gate and
 * release the region lock.  Bound to holder and epoch, so a delayed recovery
 * never reopens a later entry.  STATE if the holder is alive or the gate has
 * moved on; INVALID for an in-process gate. */
krex_status krex_gate_recover(krex_gate *gate, int32_t holder, uint64_t epoch);

/* ------------------------------------------------ shared-memory ring ---- */

/* Single-producer single-consumer ring in caller-owned shared memory, the
 * transport between a client and its context process (Section 4.3, "minimal
 * shared-memory transport": fixed-layout entries, one producer and one
 * consumer per ring; a request/reply pair is two rings).  Waiting follows the
 * spin-park policy of Section 4.3: a side that finds the ring empty (pop) or
 * full (push) spins for the ring's spin interval (default 20 us), then parks
 * on a futex until the other side's wake or the timeout; the other side
 * issues a wake only when a peer has announced that it parks.
 * `mem`: 64-byte aligned, krex_ring_bytes(capacity, entry_bytes) bytes;
 * capacity a power of two in [2, 2^24], entry_bytes a multiple of 8 in
 * [8, 4096].  Timeouts in microseconds (<= 0: 10 s); TIMEOUT when the ring
 * stayed full / empty.  At most one thread (in any process) pushes and one
 * pops. */
size_t krex_ring_bytes(uint32_t capacity, uint32_t entry_bytes);
krex_status krex_ring_init(void *mem, size_t bytes, uint32_t capacity, uint32_t entry_bytes);
krex_status krex_ring_push(void *ring, const void *entry, int64_t timeout_us);
krex_status krex_ring_pop(void *ring, void *entry, int64_t timeout_us);
/* Entries currently queued. */
krex_status krex_ring_count(void *ring, uint64_t *n);
/* The spinning interval of the spin-park policy (0: park at once). */
krex_status krex_ring_set_spin(void *ring, int64_t spin_us);
/* Counters: pushes, pops, consumer parks, producer parks, wakes sent. */
krex_status krex_ring_stats(void *ring, uint64_t *out5);

/* ------------------------------------------------ timing loop (native) --- */

/* The whole timed loop of a benchmarking command in native code: region
 * entry (drain, flush, pin), `warmup` untimed iterations and `iters` timed
 * iterations, each = L2 flush (opts->flush_bytes of opts->flush_scratch,
 * outside the event pair) then the candidate between a start and an end event
 * (Section 2.1; warm-up belongs inside the region, Section 4.1), then region
 * end.  durations_ms needs room for `iters` values.  workspace / workspace_bytes:
 * the optional GEMM workspace of krex_run_candidate_ws (may be NULL). */
krex_status krex_bench_candidate(int32_t op, const krex_buf *in, int32_t n_in, krex_buf out,
                                 const krex_region_opts *opts, int32_t warmup, int32_t iters,
                                 float *durations_ms, double *p50_ms, double *p95_ms,
                                 void *workspace, size_t workspace_bytes, krex_stream_t stream);

/* ------------------------------------------------------- one command ----- */

/* One benchmarking command (Section 2.1): inputs -> reference -> candidate
 * once -> check -> timed loop.  */
typedef struct {
    int32_t op;                /* krex_op */
    int32_t warmup;            /* untimed iterations inside the region */
    int32_t iters;             /* timed iterations (1 .. KREX_MAX_ITERS) */
    int32_t pin_cpu;           /* pin the thread inside the region */
    int64_t M, N, K;           /* GEMM: A MxK, B KxN, C MxN.  softmax: rows M, cols N */
    uint64_t seed;             /* input seed; A = tensor 0, B = tensor 1 (softmax X = 0) */
    float sigma;               /* softmax inputs: N(0, sigma^2) */
    float atol, rtol;          /* check tolerances */
    int32_t reserved;
    int64_t drain_timeout_us;
    size_t flush_bytes;        /* L2 flush size per iteration (and at region entry) */
} krex_command;

/* Device buffers of a command, all caller-owned.  in[0], in[1] (GEMM A, B) or
 * in[0] (softmax X); out = candidate output; ref = fp32 reference output;
 * flush_scratch >= flush_bytes; check_scratch >= krex_check_scratch_bytes(). */
typedef struct {
    krex_buf in[2];
    krex_buf out;
    krex_buf ref;
    void *flush_scratch;
    void *check_scratch;
    size_t check_scratch_bytes;
    void *gemm_workspace;      /* optional (may be NULL), see krex_run_candidate_ws */
    size_t gemm_workspace_bytes;
} krex_command_bufs;

typedef struct {
    krex_check_result check;
    int32_t passed;            /* 1 iff check.n_violations == 0 */
    int32_t n_iters;           /* timed iterations run (0 if the check failed) */
    double p50_ms, p95_ms;     /* of the timed iterations */
    int32_t launches;          /* kernels this command launched */
    int32_t reserved;
    double phase_ms[5];        /* inputs, reference, candidate, check: device time between CUDA
                                  events (they run back to back in the order inputs, candidate,
                                  reference, check; the check's ends when its verdict is on the
                                  host); timed loop: host wall time */
} krex_command_result;

/* Run one command (Section 2.1): inputs, the candidate once, the reference,
 * the check, then (if it passed) the timed loop in a critical region.
 * host_in (may be NULL): if given, host_in[i] (host memory, e.g. from
 * krex_host_alloc; rows*cols contiguous elements of in[i]) is copied to the
 * device instead of generating the inputs: by a copy kernel (SM loads over
 * the host link, one launch per operand) when the device reads the buffer
 * directly at the same address (page-locked, mapped, registered over the
 * whole copy) and the buffer, in[i] and their row pitches are multiples of 16
 * bytes; otherwise by the copy engine (pageable memory included, no launch).
 * On GB300 the kernel reads as fast as the copy engine from huge pages and
 * stays at that rate from 64 KiB pages, where a copy-engine read after a
 * pause slowed to 12-14 GB/s (see krex_host_alloc).  host_out (may be NULL): if
 * given, the output of the candidate's checked run (rows*cols contiguous
 * elements; the timed runs write the same values) is copied back to it on a
 * side stream while the reference runs, and the copy is complete before the
 * timed region starts.  durations_ms (may be NULL) receives the `iters` timed
 * durations.  A failing check skips the timed loop (passed = 0, n_iters = 0)
 * and still returns KREX_OK: the verdict is the result.  SYNCHRONISES. */
krex_status krex_command_run(const krex_command *cmd, const krex_command_bufs *bufs,
                             const void *const *host_in, void *host_out, float *durations_ms,
                             krex_command_result *result, krex_stream_t stream);

/* ------------------------------------------------------- host memory ----- */

/* Page-locked host memory for a command's host-side inputs and outputs
 * (krex_command_run's host_in / host_out).  Not part of the paper's method.
 * The buffer is an anonymous mapping advised to use transparent huge pages,
 * aligned to the huge-page size, then registered with CUDA (page-locked, so
 * copies run asynchronously at the host link's rate).  On hosts whose kernel
 * gives huge pages only on request (transparent hugepage mode "madvise"), a
 * buffer without them keeps its copies at full rate only while they run back
 * to back: measured on GB300 (64 KiB base pages), a 512 MiB host-to-device
 * copy took 2.6 ms back to back but 15-90 ms after a pause of a quarter
 * second, every other time, with memory pinned by cudaHostAlloc or by
 * registering an unadvised mapping; with huge pages it took 2.6 ms every
 * time.  (krex_command_run now reads page-locked inputs with SM loads, which
 * showed no such slowdown; huge pages still help the copy engine's reads.)
 * The host grants a huge page only where it finds that much contiguous free
 * memory (512 MiB on a 64 KiB-page kernel); a buffer without them works the
 * same, at those rates.  bytes > 0; *ptr receives the buffer (zero-filled).
 * Free it with krex_host_free(ptr, bytes).  Errors: INVALID for a null ptr or zero bytes,
 * CUDA if registration fails (nothing stays allocated then). */
krex_status krex_host_alloc(size_t bytes, void **ptr);
krex_status krex_host_free(void *ptr, size_t bytes);

/* ------------------------------------------------------ measurement ----- */

/* Measurement probe, not part of the paper's method: the fill kernel of a
 * seeded generator (dist as in krex_gen_inputs; the uniform one in its bf16
 * form) walking a contiguous buffer of n_elements elements on `blocks` blocks
 * of 256 threads (the fills use 8 per SM), with each 16-byte group folded into
 * a per-thread word instead of stored.  Timing it gives the rate at which the
 * GPU computes the generator: the compute ceiling the fills are measured
 * against (their outputs are 2 bf16 (uniform) or 2 fp32 (normal) per draw).
 * dev_sink: device memory of at least blocks * 256 * 4 bytes (its contents
 * afterwards are unspecified).  Asynchronous.  Errors: INVALID for a bad dist,
 * a null sink, blocks < 1 or n_elements not a positive multiple of 8. */
krex_status krex_probe_generator(int32_t dist, uint64_t n_elements, int32_t blocks, float sigma, void *dev_sink,
                                 krex_stream_t stream);

/* Measurement probe, not part of the paper's method: the FP32 fused
 * multiply-add pipe's rate, for the CUDA-core reference GEMM's roofline.
 * `blocks` blocks of 256 threads each run `iters` rounds of 16 independent
 * fp32 FMAs (2 * 16 * iters flops per thread) and store nothing but what keeps
 * the chains live.  dev_sink: device memory of at least blocks * 256 * 4 bytes
 * (contents afterwards unspecified).  Asynchronous.  Errors: INVALID for a
 * null sink, blocks < 1 or iters < 1. */
krex_status krex_probe_fma(int32_t iters, int32_t blocks, void *dev_sink, krex_stream_t stream);

/* ------------------------------------------------------------ tuning ----- */

/* The kernels' launch configuration, process-wide.  The library never reads
 * its environment: every choice is a field here, and a field left at its
 * default (0, or -1 where stated) takes the measured choice.  Not part of the
 * paper: the knobs of this implementation's kernels.  Changing it affects
 * launches issued after the call (it is read once per launch). */
typedef struct {
    int32_t gemm_pair_tile_n;  /* columns of a 2-SM pair tile: 0 = by shape (512 for long-K GEMMs whose wide
                                  tiles fill their waves, else 256); else 128, 192, 256 or 512 (two MMAs
                                  of N = 256 per K step into one 512-column accumulator) */
    int32_t gemm_stage_k;      /* K depth of a shared-memory ring stage: 0 = 128; else 64 or 128 */
    int32_t gemm_ring_stages;  /* stages of the ring in use: 0 = all that fit (3 of K 128, 6 of K 64); else
                                  2 .. that number */
    int32_t gemm_raster_group; /* pair-tile rows per raster group: 0 = 4 for GEMMs of 1.5 to 5 waves of pair
                                  tiles, else 8; else 1..64 */
    int32_t gemm_tail_split;   /* split a final partial wave: -1 = yes (default), 0 = no, 1 = yes */
    int32_t gemm_split_k;      /* split a single partial wave into K halves (needs the workspace of
                                  krex_run_candidate_ws): -1 = when K >= 4096 (default), 0 = never,
                                  1 = whenever the shape allows */
    int32_t gemm_k_alternate;  /* walk K backwards on every other wave of pair tiles, so a wave starts on
                                  the K blocks the previous one left in L2: -1 = yes (default), 0 = no,
                                  1 = yes */
    int32_t reference_tiling;  /* the CUDA-core reference GEMM's tiling: -1 = by size (default); 0..5 as
                                  documented in gemm_ref.cu (all give identical bits) */
    int32_t wait_timeout_ms;   /* bound on every wait inside a kernel: 0 = 2000 ms; else 1..600000 */
} krex_tuning;

/* The defaults (what every measurement of this library uses). */
void krex_tuning_defaults(krex_tuning *t);
/* Replace the process-wide tuning (NULL: back to the defaults).  INVALID for
 * a field out of its range (nothing changes then). */
krex_status krex_set_tuning(const krex_tuning *t);
krex_status krex_get_tuning(krex_tuning *t);

/* Test hook for failure detection: while on (non-zero), the second K half of a
 * split GEMM tile waits for a tag that no launch publishes, so its bounded
 * wait runs out (status 0x1052; see krex_device_status) without faulting or
 * hanging the GPU.  Off by default. */
krex_status krex_debug_stall_handover(int32_t on);

/* ------------------------------------------------------ host helpers ----- */

/* Linear-interpolated percentile of n host floats (q in [0,1]); host only. */
krex_status krex_percentile(const float *x, int32_t n, double q, double *out);

/* Read and clear the device-side status word written by kernels whose
 * bounded waits ran out (0 = none).  Synchronises the device. */
krex_status krex_device_status(uint32_t *code);

/* Where the first time-out since the status word was last cleared happened
 * (all zero if none), as 8 words: 0 status code | wait parity << 32;
 * 1 CTA index | grid size << 32; 2 SM id | rank in the cluster << 32;
 * 3 nanoseconds waited; then that CTA's progress: 4 producer work item |
 * K stage << 32; 5 MMA issuer work item | K stage << 32 (0xFFFFFFFF: waiting
 * for an accumulator); 6 first epilogue warp's work item | step << 32
 * (1 waiting for an accumulator, 2 draining it, 3 released); work items
 * count within the CTA pair's own sequence; 7 M | N << 21 |
 * K << 42 (each mod 2^21).  Read it before krex_device_status, which clears
 * both.  Synchronises the device. */
krex_status krex_device_status_detail(uint64_t *words);

/* Kernels this library has launched in this process, over all entry points
 * (host-side counter; the bench reports its change over the timed region). */
uint64_t krex_launch_count(void);

const char *krex_status_string(krex_status s);
const char *krex_last_error_string(void);
int32_t krex_version(void);

/* Test hook: enqueue on `stream` a host callback that waits until *gate != 0
 * (polled every 100 us, at most hold_ms milliseconds), so tests can make a
 * stream busy from the host and exercise the region drain timeout without
 * stalling the GPU. */
krex_status krex_debug_hold_stream(krex_stream_t stream, volatile int32_t *gate, int32_t hold_ms);

#ifdef __cplusplus
}
#endif
#endif /* KREX_H */
