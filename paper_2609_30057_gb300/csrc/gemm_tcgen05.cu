// K4: the timed GEMM candidate, C = A B with bf16 (or IEEE binary16)
// operands, fp32 accumulation in tensor memory and a 16-bit output rounded to
// nearest even (paper Section 2.1 and Figure 1a: the GEMM benchmarking
// command whose timed loop is 8.5% of the command).
//
// Default form, gemm_tcgen05_2sm: a cluster of two CTAs (a TPC) computes a
// 256 x bn pair tile with tcgen05.mma.cta_group::2 (M = 256, K = 16); a
// persistent grid holds one cluster per co-resident SM pair.  Pair tiles are
// up to 256 wide (one MMA of N = bn per K step) or 256 x 512 (two MMAs of
// N = 256 per K step sharing the A operand; picked for long K, where the
// SM's load rate rather than the tail decides).  Per CTA:
//   warp 0      TMA producer: A (K-major) and its half of B (N-major) tiles,
//               128-byte swizzle, into a ring of 64- or 128-deep K stages;
//               both CTAs' loads complete on the leader's full barrier, on
//               which the peer producer also arrives.
//   warp 1      (leader only) MMA issuer: one thread, 4 or 8 MMAs per stage,
//               each stage released to both producers by a multicast commit.
//   warp 2      allocates / frees 512 TMEM columns: two 256-column
//               accumulators, so the epilogue of one tile overlaps the MMAs
//               of the next, or one 512-column accumulator for 256 x 512
//               tiles, handed back in halves so that the next tile's first
//               MMAs start while its second half is still read.
//   warps 4-7   epilogue: tcgen05.ld of 32 rows each, 16-bit RNE, TMA store
//               from 128B-swizzled staging (direct stores when C's rows are
//               not 16-byte aligned).
// Pair tiles run in raster groups of rows so concurrently running pairs share
// A and B panels in L2; a final partial wave is split in two (column halves,
// or K halves whose fp32 partials meet in a caller-provided workspace).  The
// launch configuration (pair-tile width, stage depth, ring depth, raster
// group, tail split, split-K policy, wait bound) comes from the library's
// tuning record (krex_set_tuning); its defaults are the measured choices.
//
// Every mbarrier and flag wait is bounded (globaltimer); a wait that runs out
// sets a shared abort flag, the device status word and a record of where each
// role was, every role drains what it has in flight (bounded), TMEM is freed
// and the kernel returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <unordered_map>

#include "common.cuh"

namespace krex {

__device__ uint32_t g_gemm_status;  // 0 = ok; else 0x1000 | role << 4 | site
// Where the first time-out happened (written by the thread whose CAS set
// g_gemm_status): see record_timeout.
__device__ unsigned long long g_gemm_diag[8];

namespace {

// TMA boxes shared by the host-side tensor maps: A boxes of BK x BM (K-major),
// B boxes of B_BOX_N x BK (N-major); 256 threads per CTA.
constexpr int BM = 128, BK = 64;
constexpr int B_BOX_N = 64;                         // 64 bf16 = 128-byte swizzle span
constexpr int THREADS = 256;

// Shared-memory matrix descriptor: start >> 4 (bits 0-13), leading byte
// offset >> 4 (16-29), stride byte offset >> 4 (32-45), version 1 (46-47),
// base offset 0, swizzle mode 2 = 128B (61-63).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t globaltimer() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Elapsed time of a bounded wait, summed over the steps between successive
// checks.  A step that goes backwards or forward by more than 50 ms is a
// timer adjustment, not waiting, and is not counted: an unsigned difference
// against the start would turn a timer that steps back into an immediate
// time-out.
struct WaitClock {
    uint64_t last, elapsed;
    __device__ __forceinline__ WaitClock() : last(globaltimer()), elapsed(0) {}
    __device__ __forceinline__ bool expired(uint64_t limit_ns) {
        const uint64_t now = globaltimer();
        const int64_t d = (int64_t)(now - last);
        last = now;
        if (d > 0 && d < 50000000ll) elapsed += (uint64_t)d;
        return elapsed > limit_ns;
    }
};

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Non-blocking probe of a phase (no suspend): the fast path of every wait.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Per-CTA progress words that follow the abort flag in shared memory
// (prog[0] is the abort flag): 1-2 producer item / K stage, 3-4 MMA item / K
// stage, 5-6 first epilogue warp's item / step, 7-9 M, N, K.  Plain stores by
// one thread per role; read only when a wait runs out.
constexpr int PROG_WORDS = 10;

__device__ __forceinline__ uint32_t smid() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
    return r;
}

// First time-out of the device: set the status word and, if this thread set
// it, record where every role of this CTA was.
__device__ __noinline__ void record_timeout(uint32_t code, volatile uint32_t *prog, uint64_t elapsed_ns,
                                            uint32_t parity) {
    prog[0] = 1u;  // abort
    if (atomicCAS(&g_gemm_status, 0u, code) != 0u) return;
    uint32_t rank;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
    g_gemm_diag[0] = code | ((unsigned long long)parity << 32);
    g_gemm_diag[1] = blockIdx.x | ((unsigned long long)gridDim.x << 32);
    g_gemm_diag[2] = smid() | ((unsigned long long)rank << 32);
    g_gemm_diag[3] = elapsed_ns;
    g_gemm_diag[4] = prog[1] | ((unsigned long long)prog[2] << 32);
    g_gemm_diag[5] = prog[3] | ((unsigned long long)prog[4] << 32);
    g_gemm_diag[6] = prog[5] | ((unsigned long long)prog[6] << 32);
    g_gemm_diag[7] = prog[7] | ((unsigned long long)prog[8] << 21) | ((unsigned long long)prog[9] << 42);
    __threadfence();
}

// Slow path of mbar_wait: bounded polling with try_wait.
__device__ __noinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity, volatile uint32_t *abort_flag,
                                            uint64_t timeout_ns, uint32_t site, bool drain) {
    WaitClock clk;
    for (uint32_t spin = 1;; ++spin) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((spin & 63u) == 0) {
            if (!drain && *abort_flag) return false;
            if (clk.expired(timeout_ns)) {
                record_timeout(0x1000u | site, abort_flag, clk.elapsed, parity);
                return false;
            }
        }
    }
}

// Wait for the phase with parity `parity` of `bar` to complete.  Returns false
// if the CTA is aborting (unless `drain`) or `timeout_ns` passed (then it
// starts the abort).  Drain waits ignore the abort flag: they let work that is
// already in flight finish before shared memory or TMEM is released.  The
// common case (phase already complete) costs one inlined test_wait: the MMA
// issuer's waits sit on the tensor pipe's critical path.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile uint32_t *abort_flag,
                                          uint64_t timeout_ns, uint32_t site, bool drain = false) {
    if (mbar_test_wait(bar, parity)) return true;
    return mbar_wait_slow(bar, parity, abort_flag, timeout_ns, site, drain);
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, uint32_t bar,
                                            int32_t c0, int32_t c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1)
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes, without waiting
// for them (tmem_wait_ld makes them usable).
__device__ __forceinline__ void tmem_ld32_async(uint32_t taddr, uint32_t *v) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
          "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
          "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
          "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (thread t <-> lane base+t).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
          "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
          "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
          "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}


// ===================================================== 2-SM (cta_group::2) form
//
// A cluster of two CTAs on a TPC computes a 256 x 256 tile with
// tcgen05.mma.cta_group::2 (M = 256): CTA r holds rows [128r, 128r+128) of the
// A tile and columns [128r, 128r+128) of the B tile in its own shared memory,
// and its own TMEM holds its 128 rows of the 256-column accumulator.  Per SM
// a stage is 32 KiB (A 128x64 + half of B 64x128), so six stages fit and the
// L2 -> SM traffic per flop is two thirds of a one-SM 128 x 256 tile's.  A
// 256 x 512 tile is two such column chunks side by side: each CTA holds the
// 128-column halves of both chunks of B (48 KiB per 64-deep stage with A),
// the MMA thread issues one MMA per chunk and K step into columns
// [256c, 256c + 256) of one 512-column accumulator, and each SM loads 48
// bytes per MMA cycle instead of 64.
//   - both CTAs' TMA loads complete on the leader CTA's (rank 0) full barrier
//     (.cta_group::2 lets the barrier live in the peer CTA);
//   - the leader's MMA thread releases a stage in both CTAs and publishes an
//     accumulator to both epilogues with multicast tcgen05.commit;
//   - each epilogue warp of either CTA tells the leader its accumulator half
//     is drained with a remote mbarrier arrive.

namespace v2 {
constexpr int BM = 128;                          // rows per CTA (256 per pair)
constexpr int BN = 256;                          // widest pair tile (the kernel takes bn <= BN)
constexpr int BK = 64;                           // K per TMA box / swizzle atom ("sub-block")
constexpr int A_SUB_BYTES = BM * BK * 2;         // 16 KiB
constexpr int B_HALF = BN / 2;                   // 128 columns per CTA
constexpr int B_BOX_N = 64;
constexpr int B_BOX_BYTES = BK * B_BOX_N * 2;    // 8 KiB
constexpr int B_SUB_BYTES = BK * B_HALF * 2;     // 16 KiB
constexpr int RING_BYTES = 6 * (A_SUB_BYTES + B_SUB_BYTES);  // 192 KiB of stages per CTA
constexpr int EPI_BOX_COLS = 64;                 // TMA-store box: 64 columns x 32 rows (4 KiB)
constexpr int EPI_BUF_BYTES = 32 * EPI_BOX_COLS * 2;
constexpr int EPI_BYTES = 4 * 2 * EPI_BUF_BYTES; // 4 epilogue warps x 2 buffers
constexpr int TMEM_COLS = 2 * BN;                // two 256-column accumulators, or one of 512
constexpr int GROUP_M = 8;                       // pair-tile rows per raster group (see raster_group)
constexpr int EPI_WARPS = 4;
// A stage holds KSUB K sub-blocks (KSUB x 64 of K) of A and of NCH 256-column
// chunks of B: 6 stages of 32 KiB or 3 of 64 KiB for pair tiles up to 256
// wide (NCH 1), 4 stages of 48 KiB for pair tiles of 256 x 512 (NCH 2).
// Fewer, deeper stages issue 8 MMAs per barrier wait and commit instead of 4
// (each commit costs the tensor pipe a few percent).
template <int KSUB, int NCH = 1>
struct Cfg {
    static constexpr int A_STAGE_BYTES = KSUB * A_SUB_BYTES;
    static constexpr int B_STAGE_BYTES = KSUB * NCH * B_SUB_BYTES;
    static constexpr int STAGES = RING_BYTES / (A_STAGE_BYTES + B_STAGE_BYTES);
    static constexpr int NUM_BARS = 2 * STAGES + 4 + 1;
    static constexpr size_t SMEM_BYTES = 1024 + (size_t)RING_BYTES + EPI_BYTES + NUM_BARS * 8 + 48;
};
static_assert(Cfg<1>::STAGES == 6 && Cfg<2>::STAGES == 3 && Cfg<1, 2>::STAGES == 4, "ring layout");
// kind::f16, D fp32, A/B bf16, A K-major, B MN-major, M = 256 (pair); N is
// added at run time in bits 17-22
constexpr uint32_t IDESC_NO_N = (1u << 4) | (1u << 7) | (1u << 10) | (0u << 15) | (1u << 16) |
                                ((uint32_t)(256 >> 4) << 24);
}  // namespace v2

__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// shared::cluster address of the same shared variable in CTA `rank`
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
                 : "memory");
}

// Arrive without ordering: a count only (publishes no data).  The release
// form costs a cluster-scope fence, which on the producer's per-stage path
// took a third off the GEMM's throughput (measured on GB300).
__device__ __forceinline__ void mbar_arrive_remote_relaxed(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
                 : "memory");
}

// TMA load into this CTA's shared memory, completing on an mbarrier that may
// live in the peer CTA of the pair (the leader's full barrier).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar_cluster,
                                                 int32_t c0, int32_t c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1)
        : "memory");
}

// TMA store of one box from this CTA's shared memory (bulk-group completion).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, uint32_t src, int32_t c0, int32_t c1) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(src), "r"(c0), "r"(c1)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit_group() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// wait until at most N committed bulk groups still read shared memory
template <int N>
__device__ __forceinline__ void bulk_wait_group_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_group_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive on the barrier at this shared offset in both CTAs of the pair once
// all MMAs issued so far by this thread have completed.
__device__ __forceinline__ void mma_commit_pair(uint32_t bar) {
    const uint16_t mask = 0x3;
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
        " [%0], %1;" ::"r"(bar), "h"(mask)
        : "memory");
}

__device__ __forceinline__ void mma_commit_local_pair(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

__device__ __forceinline__ void tile_coords_pair(int tile, int tiles_m, int tiles_n, int group_m, int &mb,
                                                 int &nb) {
    const int per_group = group_m * tiles_n;
    const int g = tile / per_group;
    const int first_m = g * group_m;
    const int gsize = min(tiles_m - first_m, group_m);
    const int in_g = tile - g * per_group;
    mb = first_m + in_g % gsize;
    nb = in_g / gsize;
}

// Work item w of the 2-SM kernel.  Items below full_items are whole pair
// tiles: width bn, all K stages.  The rest split the tiles of a final partial
// wave in two, so that wave keeps twice as many SM pairs busy: into K halves
// (split_k: stages [0, mid) and [mid, num_kb), partial sums combined through
// the workspace; slot = tile - full_items) or, without a workspace, into
// column halves of width bn/2.
struct WorkItem {
    int mb, nb, col0, width, kb0, kb1, slot;
};

__device__ __forceinline__ WorkItem work_item(int w, int full_items, int tiles_m, int tiles_n, int group_m, int bn,
                                              int num_kb, int split_k) {
    WorkItem it;
    int tile = w, half = -1;
    if (w >= full_items) {
        const int u = w - full_items;
        tile = full_items + (u >> 1);
        half = u & 1;
    }
    tile_coords_pair(tile, tiles_m, tiles_n, group_m, it.mb, it.nb);
    it.col0 = it.nb * bn;
    it.width = bn;
    it.kb0 = 0;
    it.kb1 = num_kb;
    it.slot = -1;
    if (half >= 0) {
        if (split_k) {
            const int mid = num_kb >> 1;
            it.kb0 = half ? mid : 0;
            it.kb1 = half ? num_kb : mid;
            it.slot = tile - full_items;
        } else {
            it.width = bn >> 1;
            it.col0 += half * it.width;
        }
    }
    return it;
}

// Whether whole pair tile w walks K from its end: every other wave of the
// persistent grid (w / nclusters odd) when k_alternate is set.  All pairs of a
// wave run at about the same time and step through K together, and the
// previous wave's last K blocks are the ones still in L2, A's rows of them
// shared with this wave; so a wave that starts where the previous one ended
// reads them from L2 instead of HBM.  The accumulation order of a tile changes
// with it (each output stays within the tolerance of the exact product).
// Split tiles (the final partial wave's halves) keep the forward order.
__device__ __forceinline__ bool k_reversed(int w, int nclusters, int full_items, int k_alternate) {
    return k_alternate && w < full_items && ((w / nclusters) & 1);
}

// Two fp32 values rounded (RNE) to bf16 or binary16, packed low | high << 16.
template <bool F16>
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    if constexpr (F16) {
        __half2 h = __floats2half2_rn(lo, hi);
        return *reinterpret_cast<uint32_t *>(&h);
    } else {
        __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
        return *reinterpret_cast<uint32_t *>(&h);
    }
}

__device__ __forceinline__ void flag_store_release(uint32_t *p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t flag_load_acquire(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
// Bounded wait until *p == v (a peer CTA that is already running publishes it).
__device__ __noinline__ uint32_t flag_wait_acquire(const uint32_t *p, uint32_t v, volatile uint32_t *abort_flag,
                                                   uint64_t timeout_ns, uint32_t site) {
    WaitClock clk;
    for (uint32_t spin = 1;; ++spin) {
        if (flag_load_acquire(p) == v) return 1u;
        if ((spin & 63u) == 0) {
            if (*abort_flag) return 0u;
            if (clk.expired(timeout_ns)) {
                record_timeout(0x1000u | site, abort_flag, clk.elapsed, v);
                return 0u;
            }
        }
    }
}

__device__ __forceinline__ void spin_ns(uint64_t ns) {
    WaitClock clk;
    while (!clk.expired(ns)) {
    }
}

// Pair tiles are 256 x bn (NCH 1: bn a multiple of 64, 128 <= bn <= 256;
// NCH 2: bn = 512, two MMAs of N = 256 per K step into the two halves of one
// 512-column accumulator); tiles_m, tiles_n count them.  The host picks bn so
// the tiles fill whole waves.  F16: IEEE binary16 A, B and C
// (instruction-descriptor formats 0); else bf16.
template <int KSUB, bool F16, int NCH>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_tcgen05_2sm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmC, uint16_t *__restrict__ C, int64_t ldc, int M,
                      int N, int K, int bn, int tiles_m, int tiles_n, int full_items, int num_items,
                      int group_m, int c_vec, int c_tma, int stages, uint64_t timeout_ns, int split_k,
                      float *ws_partial, uint32_t *ws_count, uint32_t *ws_flag, uint32_t launch_id,
                      uint32_t wait_tag, int k_alternate) {
    // the pair kernel's tile constants (the file-level BM, BK serve the host's tensor maps)
    using CF = v2::Cfg<KSUB, NCH>;
    static_assert(NCH == 1 || (NCH == 2 && KSUB == 1), "wide pair tiles use 64-deep stages");
    constexpr int BM = v2::BM, BN = v2::BN, BK = v2::BK, STAGES = CF::STAGES;
    constexpr int A_STAGE_BYTES = CF::A_STAGE_BYTES, B_STAGE_BYTES = CF::B_STAGE_BYTES;
    constexpr int A_SUB_BYTES = v2::A_SUB_BYTES, B_SUB_BYTES = v2::B_SUB_BYTES;
    constexpr int B_BOX_N = v2::B_BOX_N, B_BOX_BYTES = v2::B_BOX_BYTES;
    constexpr int TMEM_COLS = v2::TMEM_COLS, NUM_BARS = CF::NUM_BARS, EPI_WARPS = v2::EPI_WARPS;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~uintptr_t(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + STAGES * A_STAGE_BYTES;
    uint8_t *sEpi = sB + STAGES * B_STAGE_BYTES;  // 1024-aligned staging buffers
    uint64_t *bars = reinterpret_cast<uint64_t *>(sEpi + v2::EPI_BYTES);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + NUM_BARS);
    volatile uint32_t *abort_flag = tmem_slot + 1;

    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
    auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
    const uint32_t mma_done_bar = bar0 + 8u * (2 * STAGES + 4);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int cluster_id = blockIdx.x >> 1, nclusters = gridDim.x >> 1;
    const int num_ksub = (K + BK - 1) / BK;               // 64-deep K sub-blocks
    const int num_kb = (num_ksub + KSUB - 1) / KSUB;      // ring stages per tile

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full_bar(s), 2);  // leader's expect_tx + the peer producer's arrive
            mbar_init(empty_bar(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull_bar(a), 1);
            mbar_init(tempty_bar(a), 2 * EPI_WARPS);  // one arrive per epilogue warp of both CTAs
        }
        mbar_init(mma_done_bar, 1);
        for (int i = 0; i < PROG_WORDS; ++i) abort_flag[i] = 0u;
        abort_flag[7] = (uint32_t)M;
        abort_flag[8] = (uint32_t)N;
        abort_flag[9] = (uint32_t)K;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    }
    if (warp == 2) {
        // one warp of each CTA of the pair allocates collectively
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncwarp();    // .aligned cluster barrier: every warp converged
    cluster_sync();  // barriers of both CTAs initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ------------------------------------------------------ TMA producer
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int w = cluster_id; ok && w < num_items; w += nclusters) {
            const WorkItem it = work_item(w, full_items, tiles_m, tiles_n, group_m, bn, num_kb, split_k);
            const int mb = it.mb, nb = it.nb, col0 = it.col0, width = it.width;
            (void)nb;
            const int cw = width / NCH;                               // columns of one MMA (a chunk)
            const int b_half = cw >> 1;                               // B columns per CTA and chunk
            const int b_boxes = (b_half + B_BOX_N - 1) / B_BOX_N;     // TMA boxes per CTA, chunk and stage
            // what each CTA of the pair loads (boxes wholly outside the matrix are skipped)
            int a_ok[2], nbox[2][NCH], nbox_all = 0;
            for (int r = 0; r < 2; ++r) {
                a_ok[r] = (mb * 2 * BM + r * BM) < M;
                for (int ch = 0; ch < NCH; ++ch) {
                    const int n0r = col0 + ch * cw + r * b_half;
                    nbox[r][ch] = n0r < N ? min(b_boxes, (N - n0r + B_BOX_N - 1) / B_BOX_N) : 0;
                    nbox_all += nbox[r][ch];
                }
            }
            const uint32_t sub_bytes = (uint32_t)((a_ok[0] + a_ok[1]) * A_SUB_BYTES +
                                                  nbox_all * B_BOX_BYTES);  // per K sub-block
            const int m0 = mb * 2 * BM + (int)rank * BM;
            const int n0 = col0 + (int)rank * b_half;                 // this CTA's columns of chunk 0
            abort_flag[1] = (uint32_t)w;
            const bool rev = k_reversed(w, nclusters, full_items, k_alternate);
            for (int i = it.kb0; i < it.kb1; ++i) {
                const int kb = rev ? it.kb0 + it.kb1 - 1 - i : i;
                abort_flag[2] = (uint32_t)kb;
                if (!mbar_wait(empty_bar(stage), phase ^ 1u, abort_flag, timeout_ns, 0x31)) {
                    ok = false;
                    break;
                }
                const int nsub = min(KSUB, num_ksub - kb * KSUB);  // sub-blocks inside K
                const uint32_t fb = mapa_shared(full_bar(stage), 0);
                // Both producers arrive on the leader's full barrier, so the MMA
                // never consumes a stage the peer producer has not reached.  A
                // peer whose rows and columns of this item all lie outside the
                // matrix loads nothing; without its arrive it could fall two
                // phases behind its empty barrier and wait on an aliased parity.
                if (leader) mbar_expect_tx(full_bar(stage), sub_bytes * (uint32_t)nsub);
                else mbar_arrive_remote_relaxed(fb);
                for (int h = 0; h < nsub; ++h) {
                    const int k0 = (kb * KSUB + h) * BK;
                    if (a_ok[rank])
                        tma_load_2d_pair(smem_u32(sA + stage * A_STAGE_BYTES + h * A_SUB_BYTES), &tmA, fb, k0, m0);
#pragma unroll
                    for (int ch = 0; ch < NCH; ++ch)
                        for (int j = 0; j < nbox[rank][ch]; ++j)
                            tma_load_2d_pair(smem_u32(sB + stage * B_STAGE_BYTES + (h * NCH + ch) * B_SUB_BYTES +
                                                      j * B_BOX_BYTES),
                                             &tmB, fb, n0 + ch * cw + j * B_BOX_N, k0);
                }
                if (++stage == stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
        if (!ok) spin_ns(200000);  // let loads already issued land before shared memory is released
    } else if (warp == 1 && lane == 0 && leader) {
        // ------------------------------------------------ MMA issuer (leader)
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        int local = 0;
        for (int w = cluster_id; ok && w < num_items; w += nclusters, ++local) {
            const WorkItem it = work_item(w, full_items, tiles_m, tiles_n, group_m, bn, num_kb, split_k);
            constexpr uint32_t idesc_ab = F16 ? (v2::IDESC_NO_N & ~((7u << 7) | (7u << 10))) : v2::IDESC_NO_N;
            const uint32_t idesc = idesc_ab | ((uint32_t)((it.width / NCH) >> 3) << 17);
            // NCH 1: two accumulators used in turn; NCH 2: one of 512 columns
            const int acc = NCH == 1 ? (local & 1) : 0;
            const uint32_t acc_phase = (uint32_t)(NCH == 1 ? ((local >> 1) & 1) : (local & 1));
            abort_flag[3] = (uint32_t)w;
            abort_flag[4] = 0xFFFFFFFFu;  // waiting for the accumulator
            const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
            const bool rev = k_reversed(w, nclusters, full_items, k_alternate);
            // the MMAs of chunks [c0, c1) of ring stage st, which holds K stage kb (item step i)
            auto issue = [&](int st, int kb, int i, int c0, int c1) {
                const int nsub = min(KSUB, num_ksub - kb * KSUB);
#pragma unroll
                for (int h = 0; h < KSUB; ++h) {
                    if (h < nsub) {
                        const uint64_t adesc =
                            sdesc_sw128(smem_u32(sA + st * A_STAGE_BYTES + h * A_SUB_BYTES), 16, 1024);
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k) {
#pragma unroll
                            for (int ch = 0; ch < NCH; ++ch) {
                                if (ch < c0 || ch >= c1) continue;
                                const uint64_t bdesc = sdesc_sw128(
                                    smem_u32(sB + st * B_STAGE_BYTES + (h * NCH + ch) * B_SUB_BYTES),
                                    B_BOX_BYTES, 1024);
                                mma_bf16_pair(d_tmem + (uint32_t)(ch * BN), adesc + (uint64_t)(2 * k),
                                              bdesc + (uint64_t)(128 * k), idesc,
                                              ((i - it.kb0) | h | k) != 0 ? 1u : 0u);
                            }
                        }
                    }
                }
            };
            int i = it.kb0;
            if constexpr (NCH == 2) {
                // One accumulator whose halves the epilogue releases in turn: the
                // chunk-0 MMAs of the first ring's worth of stages run as soon as
                // half 0 is drained, while the epilogue still drains half 1; then
                // their chunk-1 MMAs, and the stages are released.
                if (!mbar_wait(tempty_bar(0), acc_phase ^ 1u, abort_flag, timeout_ns, 0x41)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int pre = min(stages, it.kb1 - it.kb0);
                int st = stage;
                uint32_t ph = phase;
                for (int q = 0; q < pre && ok; ++q) {
                    const int kb = rev ? it.kb0 + it.kb1 - 1 - (i + q) : i + q;
                    abort_flag[4] = (uint32_t)kb;
                    if (!mbar_wait(full_bar(st), ph, abort_flag, timeout_ns, 0x42)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    issue(st, kb, i + q, 0, 1);
                    if (++st == stages) {
                        st = 0;
                        ph ^= 1u;
                    }
                }
                if (ok && !mbar_wait(tempty_bar(1), acc_phase ^ 1u, abort_flag, timeout_ns, 0x45)) ok = false;
                if (!ok) break;
                tc_fence_after();
                for (int q = 0; q < pre; ++q) {
                    const int kb = rev ? it.kb0 + it.kb1 - 1 - (i + q) : i + q;
                    issue(stage, kb, i + q, 1, 2);
                    mma_commit_pair(empty_bar(stage));
                    if (++stage == stages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                i += pre;
            } else {
                if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, abort_flag, timeout_ns, 0x41)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
            }
            for (; i < it.kb1; ++i) {
                const int kb = rev ? it.kb0 + it.kb1 - 1 - i : i;  // the stage the producer loaded
                abort_flag[4] = (uint32_t)kb;
                if (!mbar_wait(full_bar(stage), phase, abort_flag, timeout_ns, 0x42)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                issue(stage, kb, i, 0, NCH);
                mma_commit_pair(empty_bar(stage));
                if (++stage == stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (ok) mma_commit_pair(tfull_bar(acc));
        }
        mma_commit_local_pair(mma_done_bar);
        mbar_wait(mma_done_bar, 0u, abort_flag, 10000000ull, 0x43, true);
    } else if (warp >= 4) {
        // ------------------------------------------------ epilogue (both CTAs)
        const int ew = warp - 4;
        const uint32_t tempty_leader0 = mapa_shared(tempty_bar(0), 0);
        const uint32_t tempty_leader1 = mapa_shared(tempty_bar(1), 0);
        uint32_t epi_buf = 0;  // staging buffers used so far by this warp
        int local = 0;
        for (int w = cluster_id; w < num_items; w += nclusters, ++local) {
            const WorkItem it = work_item(w, full_items, tiles_m, tiles_n, group_m, bn, num_kb, split_k);
            const int mb = it.mb, nb = it.nb, col0 = it.col0, width = it.width;
            (void)nb;
            const int acc = NCH == 1 ? (local & 1) : 0;
            const uint32_t acc_phase = (uint32_t)(NCH == 1 ? ((local >> 1) & 1) : (local & 1));
            if (ew == 0 && lane == 0) {
                abort_flag[5] = (uint32_t)w;
                abort_flag[6] = 1u;  // waiting for the accumulator
            }
            const bool waited = mbar_wait(tfull_bar(acc), acc_phase, abort_flag, timeout_ns, 0x51);
            if (ew == 0 && lane == 0) abort_flag[6] = 2u;  // draining it
            if (!__all_sync(0xffffffffu, waited)) break;
            tc_fence_after();
            const int row0 = mb * 2 * BM + (int)rank * BM + ew * 32;  // this warp's 32 rows
            const int row = row0 + lane;
            const int n0 = col0;
            const uint32_t tbase = tmem_base + ((uint32_t)(ew * 32) << 16) + (uint32_t)(acc * BN);
            // Split-K half: of the two halves of a tile, the first to get here
            // parks its fp32 partial for these 32 rows in the workspace
            // ([column][row], coalesced) and publishes it with a flag tagged by
            // this launch; the second waits for the flag, adds the partial and
            // stores C.  The arrival counter resets itself (atomicInc wraps).
            // Partials are written and read at L2 (st.cg / ld.cg): they cross SMs
            // inside one launch.
            bool store_c = true;
            const float *add = nullptr;
            if (it.slot >= 0) {
                const int sidx = (it.slot * 2 + (int)rank) * EPI_WARPS + ew;
                float *part = ws_partial + (size_t)sidx * (32 * BN);
                uint32_t first = 0;
                if (lane == 0) first = atomicInc(&ws_count[sidx], 1u) == 0u ? 1u : 0u;
                first = __shfl_sync(0xffffffffu, first, 0);
                if (first) {
#pragma unroll 1
                    for (int c = 0; c < width / 32; ++c) {
                        uint32_t v[32];
                        tmem_ld32(tbase + (uint32_t)(c * 32), v);
#pragma unroll
                        for (int i = 0; i < 32; ++i) __stcg(part + (c * 32 + i) * 32 + lane, __uint_as_float(v[i]));
                    }
                    __threadfence();
                    __syncwarp();
                    if (lane == 0) flag_store_release(ws_flag + sidx, launch_id);
                    store_c = false;
                } else {
                    uint32_t ok = 1u;
                    if (lane == 0) ok = flag_wait_acquire(ws_flag + sidx, wait_tag, abort_flag, timeout_ns, 0x52);
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (ok) {
                        (void)flag_load_acquire(ws_flag + sidx);  // every lane acquires the partial
                        add = part;
                    } else {
                        store_c = false;
                    }
                }
            }
            // NCH 2: the first half of the accumulator goes back to the MMA
            // issuer as soon as it is read, the second at the end
            bool half0_released = false;
            auto release_half0 = [&]() {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_remote(tempty_leader0);
                half0_released = true;
            };
            if (!store_c) {
                // nothing to store for this item
            } else if (c_tma) {
                // 64-column chunks: TMEM -> registers -> bf16 -> 128B-swizzled staging
                // buffer (row = lane, 16-byte chunk j at j ^ (lane % 8)) -> one TMA store of
                // the 32 x 64 box; two buffers per warp alternate.
                // one 64-column chunk from registers to its staging buffer and the TMA store
                auto store_chunk = [&](int c, const uint32_t *v) {
                    uint8_t *buf = sEpi + (ew * 2 + (epi_buf & 1)) * v2::EPI_BUF_BYTES;
                    if (lane == 0) bulk_wait_group_read<1>();  // the store that used `buf` has read it
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < 8; ++j) {  // 16-byte chunk j of the 128-byte row
                        uint32_t w[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            w[i] = pack2<F16>(__uint_as_float(v[8 * j + 2 * i]), __uint_as_float(v[8 * j + 2 * i + 1]));
                        *reinterpret_cast<uint4 *>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                            make_uint4(w[0], w[1], w[2], w[3]);
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(&tmC, smem_u32(buf), n0 + c * v2::EPI_BOX_COLS, row0);
                        bulk_commit_group();
                    }
                    ++epi_buf;
                };
                if (row0 < M && !add) {
                    // No partial to add: both 32-column loads of a chunk in flight
                    // at once, one wait per chunk.
                    const int nc = min(width, N - n0) <= 0 ? 0
                                   : (min(width, N - n0) + v2::EPI_BOX_COLS - 1) / v2::EPI_BOX_COLS;
#pragma unroll 1
                    for (int c = 0; c < nc; ++c) {
                        if constexpr (NCH == 2) {
                            if (c == width / (2 * v2::EPI_BOX_COLS)) release_half0();
                        }
                        uint32_t va[64];
                        tmem_ld32_async(tbase + (uint32_t)(c * v2::EPI_BOX_COLS), va);
                        tmem_ld32_async(tbase + (uint32_t)(c * v2::EPI_BOX_COLS + 32), va + 32);
                        tmem_wait_ld();
                        store_chunk(c, va);
                    }
                } else if (row0 < M) {
                    // The other K half's partials (split-K) are read one 64-column
                    // chunk ahead, so their L2 round trips overlap this chunk's work
                    // instead of adding one per 32 columns.
                    constexpr int PC = v2::EPI_BOX_COLS;
                    float pnext[PC];
                    if (add) {
#pragma unroll
                        for (int i = 0; i < PC; ++i) pnext[i] = __ldcg(add + i * 32 + lane);
                    }
#pragma unroll 1
                    for (int c = 0; c < width / v2::EPI_BOX_COLS; ++c) {
                        if constexpr (NCH == 2) {
                            if (c == width / (2 * v2::EPI_BOX_COLS)) release_half0();
                        }
                        const int col0 = n0 + c * v2::EPI_BOX_COLS;
                        if (col0 >= N) break;  // warp-uniform
                        float pcur[PC];
#pragma unroll
                        for (int i = 0; i < PC; ++i) pcur[i] = pnext[i];
                        if (add && c + 1 < width / v2::EPI_BOX_COLS) {
#pragma unroll
                            for (int i = 0; i < PC; ++i) pnext[i] = __ldcg(add + ((c + 1) * PC + i) * 32 + lane);
                        }
                        uint8_t *buf = sEpi + (ew * 2 + (epi_buf & 1)) * v2::EPI_BUF_BYTES;
                        if (lane == 0) bulk_wait_group_read<1>();  // the store that used `buf` has read it
                        __syncwarp();
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            uint32_t v[32];
                            tmem_ld32(tbase + (uint32_t)(c * v2::EPI_BOX_COLS + h * 32), v);
                            if (add) {
#pragma unroll
                                for (int i = 0; i < 32; ++i)
                                    v[i] = __float_as_uint(__uint_as_float(v[i]) + pcur[h * 32 + i]);
                            }
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                uint32_t w[4];
#pragma unroll
                                for (int i = 0; i < 4; ++i) {
                                    w[i] = pack2<F16>(__uint_as_float(v[8 * q + 2 * i]),
                                                      __uint_as_float(v[8 * q + 2 * i + 1]));
                                }
                                const int j = h * 4 + q;  // 16-byte chunk of the 128-byte row
                                *reinterpret_cast<uint4 *>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                                    make_uint4(w[0], w[1], w[2], w[3]);
                            }
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&tmC, smem_u32(buf), col0, row0);
                            bulk_commit_group();
                        }
                        ++epi_buf;
                    }
                }
            } else {
                uint16_t *crow = C + (int64_t)row * ldc;
#pragma unroll 1
                for (int c = 0; c < width / 32; ++c) {
                    if constexpr (NCH == 2) {
                        if (c == width / 64) release_half0();
                    }
                    const int col0 = n0 + c * 32;
                    if (col0 >= N) break;  // warp-uniform
                    uint32_t v[32];
                    tmem_ld32(tbase + (uint32_t)(c * 32), v);
                    if (add) {
                        const float *pc = add + (c * 32) * 32 + lane;
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) + __ldcg(pc + i * 32));
                    }
                    if (row < M) {
                        uint32_t p[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i)
                            p[i] = pack2<F16>(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
                        if (c_vec && col0 + 32 <= N) {
                            uint4 *dst = reinterpret_cast<uint4 *>(crow + col0);
                            dst[0] = make_uint4(p[0], p[1], p[2], p[3]);
                            dst[1] = make_uint4(p[4], p[5], p[6], p[7]);
                            dst[2] = make_uint4(p[8], p[9], p[10], p[11]);
                            dst[3] = make_uint4(p[12], p[13], p[14], p[15]);
                        } else {
                            for (int i = 0; i < 32 && col0 + i < N; ++i)
                                crow[col0 + i] = (uint16_t)((i & 1) ? (p[i >> 1] >> 16) : (p[i >> 1] & 0xFFFFu));
                        }
                    }
                }
            }
            if constexpr (NCH == 2) {
                if (!half0_released) release_half0();
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote((NCH == 2 || acc) ? tempty_leader1 : tempty_leader0);
            if (ew == 0 && lane == 0) abort_flag[6] = 3u;  // released
        }
        if (lane == 0) bulk_wait_group_all();  // stores complete before shared memory goes away
        __syncwarp();
    }

    // ---------------------------------------------------------------- teardown
    tc_fence_before();
    __syncwarp();
    cluster_sync();  // the leader's MMAs into both CTAs' TMEM are complete
    if (warp == 2) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(TMEM_COLS)
                     : "memory");
    }
}

// ---------------------------------------------------------------- host side

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

struct MapKey {
    const void *ptr;
    uint64_t inner, outer, stride_bytes;
    uint32_t box_inner, box_outer;
    bool f16;
    bool operator==(const MapKey &o) const {
        return ptr == o.ptr && inner == o.inner && outer == o.outer && stride_bytes == o.stride_bytes &&
               box_inner == o.box_inner && box_outer == o.box_outer && f16 == o.f16;
    }
};
struct MapKeyHash {
    size_t operator()(const MapKey &k) const {
        size_t h = std::hash<const void *>()(k.ptr);
        h ^= std::hash<uint64_t>()(k.inner * 0x9E3779B97F4A7C15ull + k.outer) + (h << 6) + (h >> 2);
        h ^= std::hash<uint64_t>()(k.stride_bytes ^ ((uint64_t)k.box_inner << 32 | k.box_outer)) + (h << 6);
        h ^= (size_t)k.f16;
        return h;
    }
};

// 2-D bf16 (f16: binary16) tensor map: inner dimension contiguous, 128-byte
// swizzle, OOB -> 0.  Encoded maps are cached (a map is a pure function of
// its key).
krex_status make_map(const void *ptr, uint64_t inner, uint64_t outer, uint64_t ld_elems,
                     uint32_t box_inner, uint32_t box_outer, bool f16, CUtensorMap *out) {
    static std::mutex mu;
    static std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
    MapKey key{ptr, inner, outer, ld_elems * 2, box_inner, box_outer, f16};
    {
        std::lock_guard<std::mutex> lk(mu);
        auto it = cache.find(key);
        if (it != cache.end()) {
            *out = it->second;
            return KREX_OK;
        }
    }
    auto enc = get_encode_fn();
    if (!enc) return set_error(KREX_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {ld_elems * 2};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(out, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                     const_cast<void *>(ptr), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return set_error(KREX_ERR_CUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", (int)r);
    std::lock_guard<std::mutex> lk(mu);
    if (cache.size() > 4096) cache.clear();
    cache.emplace(key, *out);
    return KREX_OK;
}

// Launch configuration of the 2-SM kernel, from the library's tuning record
// (krex_get_tuning_internal); a field at its default takes the measured
// choice documented beside it.
//
// Pair-tile width.  Measured on GB300, a tcgen05.mma of N = 224 or 192 costs
// about as much time as N = 256, so narrower tiles only add waves.  Wide pair
// tiles of 256 x 512 (two MMAs of N = 256 per K step into one 512-column
// accumulator) load a quarter fewer bytes per flop into each SM, whose load
// rate (about 100 GB/s per SM) holds 256-wide tiles near 87 % of the tensor
// pipe (wide ones: 96 %); but with one accumulator the epilogue overlaps the
// next tile's MMAs only in part, and the tail split into column halves does
// not apply.  So the choice weighs how well each width fills its waves (a
// split tail's half-width items cost about 0.8 of a whole tile) against the
// wide tiles' per-tile gain, measured (L2 flushed, 256 vs 512, ratio of
// times): 1.01 at K = 2048 (8192^2), 0.95-0.97 at K = 4096 (8192^2, 16384^2;
// a tie at 4096^3, whose wide tiles fill 1.7 waves), 0.92-0.96 from K = 6144
// on (6144^3 to 16384^3), and 1.05 for 4096 x 8192 x 16384, where the wide
// tiles fill 3.4 waves against the 256-wide tiles' 6.7.  The tuning record
// fixes the width (128, 192, 256 or 512: the epilogue stores 64-column boxes).
constexpr int64_t kWideMinK = 4096;

int pick_pair_tile_n(const krex_tuning &t, int64_t M, int64_t N, int64_t K, int max_clusters) {
    if (t.gemm_pair_tile_n) return t.gemm_pair_tile_n;
    if (K < kWideMinK || max_clusters <= 0) return 256;
    const double gain = K < 6144 ? 1.04 : 1.08;  // the wide tiles' per-tile gain at this K
    const int64_t tm = (M + 2 * v2::BM - 1) / (2 * v2::BM);
    const int64_t t512 = tm * ((N + 511) / 512), t256 = tm * ((N + 255) / 256);
    const double c = (double)max_clusters;
    const double eff512 = (double)t512 / (c * (double)((t512 + max_clusters - 1) / max_clusters));
    const int64_t rem = t256 % max_clusters;
    const double waves256 = (double)(t256 / max_clusters) + (rem == 0 ? 0.0 : (2 * rem <= max_clusters ? 0.8 : 1.0));
    const double eff256 = (double)t256 / (c * waves256);
    return eff512 * gain >= eff256 ? 512 : 256;
}

// Pair-tile rows per raster group.  Measured on GB300 (TFLOP/s, group 4 vs
// 8, L2 flushed): 3072^3 1381 vs 1325, 4096^3 1561 vs 1525, 4608^3 1579 vs
// 1557, but 2064^3 578 vs 592, 5120^3 1616 vs 1638, 7168^3 1739 vs 1794,
// 8192^3 1799 vs 1851: 4 for GEMMs of 1.5 to 5 waves of pair tiles, else 8.
int raster_group(const krex_tuning &t, int64_t tiles, int max_clusters) {
    if (t.gemm_raster_group) return t.gemm_raster_group;
    return (2 * tiles >= 3 * (int64_t)max_clusters && tiles < 5 * (int64_t)max_clusters) ? 4 : v2::GROUP_M;
}

// K halves for a single partial wave (when a workspace is given): by default
// when K >= kSplitKMinK; the tuning record can force them whenever the shape
// allows (the tests use that to exercise the hand-over on small shapes) or
// switch them off.  Measured on GB300 (L2 flushed): the hand-over of the fp32
// partials costs about 4-6 us, so below K = 4096 column halves win (256^3:
// 10.2 against 16.4 us; 1024^3: 14.3 against 18.5 us), while 1024 x 2048 x
// 8192 gains 8 %.
constexpr int64_t kSplitKMinK = 4096;

// Stages of the shared-memory ring in use (at most `max_stages`).
int ring_stages(const krex_tuning &t, int max_stages) {
    return t.gemm_ring_stages ? t.gemm_ring_stages : max_stages;
}

// K sub-blocks (of 64) per ring stage: 2 = three 64 KiB stages (default),
// 1 = six 32 KiB stages.
int stage_ksub(const krex_tuning &t) { return t.gemm_stage_k == 64 ? 1 : 2; }

// The second K half of a split tile waits for a tag that no launch publishes
// while this is set (krex_debug_stall_handover; the failure-detection test
// only), so its bounded wait runs out: the kernel then sets the status word
// (0x1052), drains and returns, and the context stays usable.
std::atomic<int> g_debug_stall_handover{0};

uint64_t wait_timeout_ns(const krex_tuning &t) {
    return (uint64_t)(t.wait_timeout_ms > 0 ? t.wait_timeout_ms : 2000) * 1000000ull;
}

}  // namespace

// Split-K workspace: fp32 partials of up to WS_SLOTS split tiles (2 CTAs x 4
// epilogue warps x 32 rows x 256 columns each), then one arrival counter and
// one flag per 32-row slab.
constexpr int WS_SLOTS = 64;
constexpr size_t WS_SLABS = (size_t)WS_SLOTS * 2 * 4;
constexpr size_t WS_PARTIAL_BYTES = WS_SLABS * 32 * 256 * sizeof(float);
constexpr size_t WS_BYTES = WS_PARTIAL_BYTES + 2 * WS_SLABS * sizeof(uint32_t);

size_t gemm_workspace_bytes() { return WS_BYTES; }

krex_status launch_gemm_tcgen05(const uint16_t *a, int64_t lda, const uint16_t *b, int64_t ldb,
                                uint16_t *c, int64_t ldc, int64_t M, int64_t N, int64_t K, bool f16,
                                void *workspace, size_t workspace_bytes, cudaStream_t s) {
    if (M == 0 || N == 0) return KREX_OK;
    if (K == 0) {
        KREX_CUDA_TRY(cudaMemset2DAsync(c, (size_t)ldc * 2, 0, (size_t)N * 2, (size_t)M, s));
        return KREX_OK;
    }
    if (M > (1ll << 31) - 2 * v2::BM || N > (1ll << 31) - v2::BN || K > (1ll << 31) - BK)
        return set_error(KREX_ERR_UNSUPPORTED, "GEMM dimension too large for the tcgen05 path");
    // Tensor-map encoding is a driver call and needs a current context on this
    // thread; a thread whose first CUDA work is this GEMM has none yet, so bind
    // the runtime's current device (its primary context) once per thread.
    static thread_local int bound_dev = -1;
    {
        int d = 0;
        KREX_CUDA_TRY(cudaGetDevice(&d));
        if (bound_dev != d) {
            KREX_CUDA_TRY(cudaSetDevice(d));
            bound_dev = d;
        }
    }
    const krex_tuning tun = tuning_snapshot();
    CUtensorMap ma, mb;
    krex_status st = make_map(a, (uint64_t)K, (uint64_t)M, (uint64_t)lda, BK, BM, f16, &ma);
    if (st != KREX_OK) return st;
    st = make_map(b, (uint64_t)N, (uint64_t)K, (uint64_t)ldb, B_BOX_N, BK, f16, &mb);
    if (st != KREX_OK) return st;

    static thread_local int attr_dev = -1;
    static thread_local int max_clusters = 0;
    int dev = 0;
    KREX_CUDA_TRY(cudaGetDevice(&dev));
    if (attr_dev != dev) {
        KREX_CUDA_TRY(cudaFuncSetAttribute(gemm_tcgen05_2sm<1, false, 1>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)v2::Cfg<1>::SMEM_BYTES));
        KREX_CUDA_TRY(cudaFuncSetAttribute(gemm_tcgen05_2sm<2, false, 1>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)v2::Cfg<2>::SMEM_BYTES));
        KREX_CUDA_TRY(cudaFuncSetAttribute(gemm_tcgen05_2sm<1, true, 1>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)v2::Cfg<1>::SMEM_BYTES));
        KREX_CUDA_TRY(cudaFuncSetAttribute(gemm_tcgen05_2sm<2, true, 1>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)v2::Cfg<2>::SMEM_BYTES));
        KREX_CUDA_TRY(cudaFuncSetAttribute(gemm_tcgen05_2sm<1, false, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)v2::Cfg<1, 2>::SMEM_BYTES));
        KREX_CUDA_TRY(cudaFuncSetAttribute(gemm_tcgen05_2sm<1, true, 2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)v2::Cfg<1, 2>::SMEM_BYTES));
        // co-resident CTA pairs; a persistent grid larger than this would only queue
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * (unsigned)(sm_count() / 2), 1, 1);
        cfg.blockDim = dim3(THREADS, 1, 1);
        cfg.dynamicSmemBytes = v2::Cfg<2>::SMEM_BYTES;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, gemm_tcgen05_2sm<2, false, 1>, &cfg) != cudaSuccess || n <= 0) {
            cudaGetLastError();
            n = sm_count() / 2;
        }
        max_clusters = n;
        attr_dev = dev;
    }
    const int c_vec = ((reinterpret_cast<uintptr_t>(c) & 15u) == 0) && (ldc % 8 == 0);
    {
        // TMA-store epilogue when C rows start on 16 bytes; else direct stores
        CUtensorMap mc;
        int c_tma = c_vec;
        if (c_tma) {
            st = make_map(c, (uint64_t)N, (uint64_t)M, (uint64_t)ldc, v2::EPI_BOX_COLS, 32, f16, &mc);
            if (st != KREX_OK) return st;
        } else {
            mc = ma;  // unused
        }
        const int tiles_m = (int)((M + 2 * v2::BM - 1) / (2 * v2::BM));
        const int bn = pick_pair_tile_n(tun, M, N, K, max_clusters);
        const int tiles_n = (int)((N + bn - 1) / bn);
        const int64_t tiles = (int64_t)tiles_m * tiles_n;
        // Split the tiles of a final partial wave into column halves when that
        // at most fills the co-resident pairs (4096^2: 256 tiles on 76 pairs ->
        // 228 whole tiles + 56 halves instead of a last wave of 28 tiles).
        const int64_t rem = tiles % max_clusters;
        const bool split = bn == 256 && rem > 0 && 2 * rem <= max_clusters && tun.gemm_tail_split != 0;
        const int64_t full_items = split ? tiles - rem : tiles;
        const int64_t items = split ? tiles + rem : tiles;
        const int clusters = (int)(items < max_clusters ? items : max_clusters);
        // K halves (full-width MMAs) when a zero-initialised workspace is given,
        // K has at least two ring stages and is long enough (the tuning's split_k), and
        // the split tiles are the whole GEMM (one partial wave); else column
        // halves.  Measured on GB300: K
        // halves load a third less than column halves (1024 x 2048 x 8192:
        // 49 -> 44 us), but the hand-over of the fp32 partials (128 KiB per CTA
        // written, then read) sits on the last wave's critical path: at 4096^3
        // the K halves end their MMAs 6.8 us earlier and spend about as long
        // exchanging partials, so the multi-wave case gains nothing.
        const int ksub = bn == 512 ? 1 : stage_ksub(tun);
        const int64_t num_kb = (((K + 63) / 64) + ksub - 1) / ksub;
        const int sk_mode = tun.gemm_split_k;
        const bool k_worth_it = sk_mode == 1 || (sk_mode < 0 && K >= kSplitKMinK);
        const int split_k = split && full_items == 0 && workspace && workspace_bytes >= WS_BYTES &&
                            rem <= WS_SLOTS && num_kb >= 2 && clusters >= 2 && k_worth_it;
        static std::atomic<uint32_t> launch_counter{0};
        uint32_t launch_id = launch_counter.fetch_add(1) + 1;
        if (launch_id == 0) launch_id = launch_counter.fetch_add(1) + 1;  // 0 never tags a published partial
        // the tag the second K half waits for: this launch's, or (the failure-
        // detection test's switch) one that no launch publishes
        const uint32_t wait_tag = g_debug_stall_handover.load() ? (launch_id ^ 0x80000000u) : launch_id;
        float *ws_partial = split_k ? static_cast<float *>(workspace) : nullptr;
        uint32_t *ws_count =
            split_k ? reinterpret_cast<uint32_t *>(static_cast<uint8_t *>(workspace) + WS_PARTIAL_BYTES) : nullptr;
        uint32_t *ws_flag = split_k ? ws_count + WS_SLABS : nullptr;
        auto go = [&](auto kernel, size_t smem, int stages) {
            kernel<<<2 * clusters, THREADS, smem, s>>>(ma, mb, mc, c, ldc, (int)M, (int)N, (int)K, bn, tiles_m,
                                                       tiles_n, (int)full_items, (int)items,
                                                       raster_group(tun, tiles, max_clusters), c_vec,
                                                       c_tma, stages, wait_timeout_ns(tun), split_k, ws_partial,
                                                       ws_count, ws_flag, launch_id, wait_tag,
                                                       tun.gemm_k_alternate == 0 ? 0 : 1);
        };
        const int st2 = ring_stages(tun, v2::Cfg<2>::STAGES), st1 = ring_stages(tun, v2::Cfg<1>::STAGES);
        const int stw = std::min(ring_stages(tun, v2::Cfg<1, 2>::STAGES), v2::Cfg<1, 2>::STAGES);
        if (bn == 512 && f16)
            go(gemm_tcgen05_2sm<1, true, 2>, v2::Cfg<1, 2>::SMEM_BYTES, stw);
        else if (bn == 512)
            go(gemm_tcgen05_2sm<1, false, 2>, v2::Cfg<1, 2>::SMEM_BYTES, stw);
        else if (ksub == 2 && f16)
            go(gemm_tcgen05_2sm<2, true, 1>, v2::Cfg<2>::SMEM_BYTES, st2);
        else if (ksub == 2)
            go(gemm_tcgen05_2sm<2, false, 1>, v2::Cfg<2>::SMEM_BYTES, st2);
        else if (f16)
            go(gemm_tcgen05_2sm<1, true, 1>, v2::Cfg<1>::SMEM_BYTES, st1);
        else
            go(gemm_tcgen05_2sm<1, false, 1>, v2::Cfg<1>::SMEM_BYTES, st1);
    }
    KREX_CUDA_TRY(cudaGetLastError());
    return KREX_OK;
}

void set_debug_stall_handover(bool on) { g_debug_stall_handover.store(on ? 1 : 0); }

cudaError_t read_device_status_detail(unsigned long long *words) {
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return e;
    return cudaMemcpyFromSymbol(words, g_gemm_diag, sizeof(g_gemm_diag));
}

cudaError_t read_and_clear_device_status(uint32_t *code) {
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbol(code, g_gemm_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    const uint32_t zero = 0;
    e = cudaMemcpyToSymbol(g_gemm_status, &zero, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    const unsigned long long zeros[8] = {};
    return cudaMemcpyToSymbol(g_gemm_diag, zeros, sizeof(zeros));
}

}  // namespace krex
