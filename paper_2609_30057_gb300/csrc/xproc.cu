// Cross-process pieces of the paper's runtime, host-only:
//
//  - The in-region gate of Section 4.2 ("GPU exclusivity") with its state in
//    shared memory, so tenants in different processes take part: region lock,
//    gate (holder, epoch), per-tenant in-flight counters and acknowledgements.
//    Each attached process runs a drainer thread that, when the gate closes,
//    waits for its own tenants' counters to reach zero, synchronises their
//    streams and publishes the epoch as acknowledged; the holder polls the
//    acknowledgements and counters.  A sibling process that dies during entry
//    fails the entry; a holder that dies leaves the gate to
//    krex_gate_recover, bound to that holder and epoch.
//  - The single-producer single-consumer shared-memory ring of Section 4.3
//    ("minimal shared-memory transport") with the spin-park waiting policy:
//    spin for a short interval, then park on a futex; the other side wakes a
//    parked peer only when the peer has announced that it parks.
//
// Everything in shared memory is a lock-free std::atomic (address-free), so
// each process may map the memory at a different address.  Futexes are the
// shared (not process-private) kind.
#include <errno.h>
#include <linux/futex.h>
#include <signal.h>
#include <string.h>
#include <sys/syscall.h>
#include <time.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <climits>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "common.cuh"
#include "xproc.h"

namespace krex {
namespace {

using clk = std::chrono::steady_clock;

static_assert(std::atomic<uint32_t>::is_always_lock_free && std::atomic<int32_t>::is_always_lock_free &&
                  std::atomic<uint64_t>::is_always_lock_free && std::atomic<int64_t>::is_always_lock_free,
              "shared-memory state needs lock-free (address-free) atomics");

long futex_wait(std::atomic<uint32_t> *w, uint32_t expected, int64_t timeout_ns) {
    if (timeout_ns < 0) timeout_ns = 0;
    struct timespec ts;
    ts.tv_sec = (time_t)(timeout_ns / 1000000000);
    ts.tv_nsec = (long)(timeout_ns % 1000000000);
    return syscall(SYS_futex, reinterpret_cast<uint32_t *>(w), FUTEX_WAIT, expected, &ts, nullptr, 0);
}

void futex_wake_all(std::atomic<uint32_t> *w) {
    syscall(SYS_futex, reinterpret_cast<uint32_t *>(w), FUTEX_WAKE, INT_MAX, nullptr, nullptr, 0);
}

bool pid_alive(int32_t pid) {
    if (pid <= 0) return false;
    return kill(pid, 0) == 0 || errno == EPERM;
}

clk::time_point deadline_from(int64_t timeout_us) {
    if (timeout_us <= 0) timeout_us = 10 * 1000 * 1000;
    return clk::now() + std::chrono::microseconds(timeout_us);
}

int64_t ns_left(clk::time_point deadline) {
    return std::chrono::duration_cast<std::chrono::nanoseconds>(deadline - clk::now()).count();
}

// Spin-park (Section 4.3): poll ready() for spin_ns, then park on the futex
// word `seq`, announcing it through `parked`, until ready() or the deadline.
// A waker publishes its change, then reads `parked` and, if set, bumps `seq`
// and wakes: with sequentially consistent accesses on both sides either the
// waiter sees the change or the waker sees the announcement, and a bump
// between the waiter's read of `seq` and its futex call makes the call
// return at once.
template <class Ready>
bool spin_park_futex(Ready ready, std::atomic<uint32_t> &seq, std::atomic<uint32_t> &parked, int64_t spin_ns,
                     clk::time_point deadline, std::atomic<uint64_t> *park_count) {
    if (ready()) return true;
    const auto spin_until = clk::now() + std::chrono::nanoseconds(spin_ns);
    while (clk::now() < spin_until)
        if (ready()) return true;
    for (;;) {
        const uint32_t s = seq.load(std::memory_order_seq_cst);
        parked.fetch_add(1, std::memory_order_seq_cst);
        if (ready()) {
            parked.fetch_sub(1, std::memory_order_seq_cst);
            return true;
        }
        const int64_t left = ns_left(deadline);
        if (left <= 0) {
            parked.fetch_sub(1, std::memory_order_seq_cst);
            return ready();
        }
        if (park_count) park_count->fetch_add(1, std::memory_order_relaxed);
        futex_wait(&seq, s, std::min<int64_t>(left, 100000000));
        parked.fetch_sub(1, std::memory_order_seq_cst);
        if (ready()) return true;
    }
}

// ------------------------------------------------------------------- ring --

constexpr uint64_t kRingMagic = 0x474E4952584552ull;  // "REXRING"
constexpr uint32_t kVersion = 1;

struct alignas(64) RingHdr {
    uint64_t magic;
    uint32_t version, capacity, entry_bytes, pad0;
    std::atomic<int64_t> spin_ns;
    alignas(64) std::atomic<uint64_t> head;  // next entry the producer writes (producer-owned)
    alignas(64) std::atomic<uint64_t> tail;  // next entry the consumer reads (consumer-owned)
    alignas(64) std::atomic<uint32_t> data_seq;  // the consumer parks on it
    std::atomic<uint32_t> consumer_parked;
    alignas(64) std::atomic<uint32_t> space_seq;  // the producer parks on it
    std::atomic<uint32_t> producer_parked;
    // pushes, pops, consumer parks, producer parks, wakes sent
    alignas(64) std::atomic<uint64_t> stats[5];
};
static_assert(sizeof(RingHdr) % 64 == 0, "ring entries start on a cache line");

RingHdr *ring_of(void *mem) {
    RingHdr *r = static_cast<RingHdr *>(mem);
    if (!r || (reinterpret_cast<uintptr_t>(mem) & 63u) || r->magic != kRingMagic || r->version != kVersion)
        return nullptr;
    return r;
}

uint8_t *ring_slot(RingHdr *r, uint64_t i) {
    return reinterpret_cast<uint8_t *>(r + 1) + (size_t)(i & (r->capacity - 1)) * r->entry_bytes;
}

// ---------------------------------------------------------------- gate -----

constexpr uint64_t kGateMagic = 0x4554414758455252ull;  // "RREXGATE"

struct alignas(64) XTenant {
    std::atomic<int32_t> state;       // 0 free, 1 registered
    std::atomic<int32_t> pid;         // owning process
    std::atomic<int64_t> inflight;    // submissions in the host submission path
    std::atomic<uint64_t> acked_epoch;
    std::atomic<int32_t> ack_status;  // krex_status of the drain that acknowledged acked_epoch
};

struct alignas(64) XGateHdr {
    uint64_t magic;
    uint32_t version;
    int32_t max_tenants;
    alignas(64) std::atomic<int32_t> reg_lock;  // pid of the owner, 0 = free (registration vs closure)
    std::atomic<int32_t> region_owner;          // holder tenant of the region lock, -1 = free
    std::atomic<int32_t> holder;                // -1 = gate open
    std::atomic<int32_t> holder_pid;
    std::atomic<uint64_t> epoch;
    alignas(64) std::atomic<uint32_t> gate_seq;  // futex word, bumped on every change of the gate
    std::atomic<uint32_t> gate_waiters;
    std::atomic<int32_t> parked;
};
static_assert(sizeof(XGateHdr) % 64 == 0 && sizeof(XTenant) == 64, "shared gate layout");

}  // namespace

struct XGate {
    XGateHdr *h = nullptr;
    XTenant *t = nullptr;
    std::mutex mu;                       // guards the local tables
    std::vector<char> local;             // tenant slots registered by this process
    std::vector<cudaStream_t> stream;    // their streams (drained by this process)
    std::vector<int> device;             // the device current when each registered
    std::thread drainer;
    std::atomic<bool> stop{false};
};

namespace {

bool reg_lock(XGateHdr *h, clk::time_point deadline) {
    const int32_t me = (int32_t)getpid();
    for (uint64_t spin = 0;; ++spin) {
        int32_t expected = 0;
        if (h->reg_lock.compare_exchange_weak(expected, me, std::memory_order_seq_cst)) return true;
        if ((spin & 1023u) == 1023u) {
            // an owner that died inside the (short) critical section is taken over
            if (expected != 0 && expected != me && !pid_alive(expected))
                h->reg_lock.compare_exchange_strong(expected, 0, std::memory_order_seq_cst);
            if (clk::now() >= deadline) return false;
            std::this_thread::yield();
        }
    }
}

void reg_unlock(XGateHdr *h) { h->reg_lock.store(0, std::memory_order_seq_cst); }

void gate_changed(XGateHdr *h) {
    h->gate_seq.fetch_add(1, std::memory_order_seq_cst);
    futex_wake_all(&h->gate_seq);
}

// Wait for pred() or the deadline: spin ~20 us, then sleep on gate changes
// (bounded naps, so a predicate that changes without a bump is still seen).
template <class Pred>
bool wait_gate(XGateHdr *h, Pred pred, clk::time_point deadline, int64_t nap_ns = 2000000) {
    const auto spin_until = clk::now() + std::chrono::microseconds(20);
    while (clk::now() < spin_until)
        if (pred()) return true;
    for (;;) {
        const uint32_t s = h->gate_seq.load(std::memory_order_seq_cst);
        if (pred()) return true;
        const int64_t left = ns_left(deadline);
        if (left <= 0) return pred();
        h->gate_waiters.fetch_add(1, std::memory_order_relaxed);
        futex_wait(&h->gate_seq, s, std::min(left, nap_ns));
        h->gate_waiters.fetch_sub(1, std::memory_order_relaxed);
    }
}

// Free the slots of tenants whose process no longer exists (reg_lock held,
// gate open).
void reap_dead(XGate *x) {
    for (int32_t i = 0; i < x->h->max_tenants; ++i) {
        XTenant &t = x->t[i];
        if (t.state.load() == 1 && !pid_alive(t.pid.load())) {
            t.inflight.store(0);
            t.state.store(0, std::memory_order_seq_cst);
        }
    }
}

bool local_tenant(XGate *x, int32_t i) {
    if (i < 0 || i >= x->h->max_tenants) return false;
    std::lock_guard<std::mutex> lk(x->mu);
    return x->local[(size_t)i] && x->t[i].state.load() == 1;
}

// This process's part of an entry (Section 4.2 step 3): for every local
// tenant other than the holder, wait for its counter to reach zero,
// synchronise its stream and acknowledge the epoch.  Abandoned if the gate
// moves on (the entry failed or ended).
void drain_local(XGate *x, int32_t holder, uint64_t e) {
    XGateHdr *h = x->h;
    std::vector<int32_t> mine;
    std::vector<cudaStream_t> streams;
    std::vector<int> devs;
    {
        std::lock_guard<std::mutex> lk(x->mu);
        for (int32_t i = 0; i < h->max_tenants; ++i)
            if (x->local[(size_t)i] && i != holder) {
                mine.push_back(i);
                streams.push_back(x->stream[(size_t)i]);
                devs.push_back(x->device[(size_t)i]);
            }
    }
    auto same_entry = [&] { return h->holder.load() == holder && h->epoch.load() == e; };
    for (size_t k = 0; k < mine.size(); ++k) {
        XTenant &t = x->t[mine[k]];
        if (t.state.load() != 1) continue;
        const auto deadline = clk::now() + std::chrono::seconds(60);
        const bool idle = wait_gate(h, [&] { return t.inflight.load() == 0 || !same_entry(); }, deadline, 200000);
        if (!same_entry()) return;
        krex_status st = KREX_OK;
        if (!idle) {
            st = KREX_ERR_TIMEOUT;
        } else if (streams[k]) {
            cudaError_t err = cudaSetDevice(devs[k]);
            if (err == cudaSuccess) err = cudaStreamSynchronize(streams[k]);
            if (err != cudaSuccess) st = KREX_ERR_CUDA;
        }
        t.ack_status.store(st, std::memory_order_seq_cst);
        t.acked_epoch.store(e, std::memory_order_seq_cst);
    }
}

void drainer_main(XGate *x) {
    XGateHdr *h = x->h;
    uint64_t drained = 0;
    for (;;) {
        const uint32_t s = h->gate_seq.load(std::memory_order_seq_cst);
        if (x->stop.load()) return;
        const int32_t hold = h->holder.load(std::memory_order_seq_cst);
        const uint64_t e = h->epoch.load(std::memory_order_seq_cst);
        if (hold >= 0 && e != drained) {
            drain_local(x, hold, e);
            drained = e;
            continue;
        }
        futex_wait(&h->gate_seq, s, 20000000);
    }
}

}  // namespace

// ------------------------------------------------------------ gate (API) ---

krex_status xgate_attach(void *mem, size_t bytes, XGate **out) {
    XGateHdr *h = static_cast<XGateHdr *>(mem);
    if (!h || !out || (reinterpret_cast<uintptr_t>(mem) & 63u))
        return set_error(KREX_ERR_INVALID, "gate_shared_attach: need 64-byte aligned memory and out");
    if (bytes < sizeof(XGateHdr) || h->magic != kGateMagic || h->version != kVersion)
        return set_error(KREX_ERR_INVALID, "gate_shared_attach: memory does not hold a formatted gate");
    if (bytes < sizeof(XGateHdr) + (size_t)h->max_tenants * sizeof(XTenant))
        return set_error(KREX_ERR_INVALID, "gate_shared_attach: %zu bytes is too small", bytes);
    XGate *x = new XGate();
    x->h = h;
    x->t = reinterpret_cast<XTenant *>(h + 1);
    x->local.assign((size_t)h->max_tenants, 0);
    x->stream.assign((size_t)h->max_tenants, nullptr);
    x->device.assign((size_t)h->max_tenants, 0);
    x->drainer = std::thread(drainer_main, x);
    *out = x;
    return KREX_OK;
}

krex_status xgate_detach(XGate *x) {
    XGateHdr *h = x->h;
    std::vector<int32_t> mine;
    {
        std::lock_guard<std::mutex> lk(x->mu);
        for (int32_t i = 0; i < h->max_tenants; ++i)
            if (x->local[(size_t)i]) mine.push_back(i);
    }
    for (int32_t i : mine)
        if (h->holder.load() == i) return set_error(KREX_ERR_STATE, "gate detach: tenant %d holds the gate", i);
    x->stop.store(true);
    futex_wake_all(&h->gate_seq);
    if (x->drainer.joinable()) x->drainer.join();
    // this process's tenants leave: their work first finishes, then the slots free
    for (int32_t i : mine) {
        if (x->stream[(size_t)i] && cudaSetDevice(x->device[(size_t)i]) == cudaSuccess)
            cudaStreamSynchronize(x->stream[(size_t)i]);
        if (x->t[i].pid.load() == (int32_t)getpid()) x->t[i].state.store(0, std::memory_order_seq_cst);
    }
    delete x;
    return KREX_OK;
}

krex_status xgate_register(XGate *x, krex_stream_t stream, int64_t timeout_us, int32_t *tenant) {
    if (!tenant) return set_error(KREX_ERR_INVALID, "gate_register: null tenant");
    XGateHdr *h = x->h;
    const auto deadline = deadline_from(timeout_us);
    int dev = 0;
    if (stream && cudaGetDevice(&dev) != cudaSuccess) dev = 0;
    for (;;) {
        if (!reg_lock(h, deadline)) return set_error(KREX_ERR_TIMEOUT, "gate_register: registration lock");
        if (h->holder.load() == -1) {  // serialised with closure: only while the gate is open
            reap_dead(x);
            for (int32_t i = 0; i < h->max_tenants; ++i) {
                XTenant &t = x->t[i];
                if (t.state.load() == 0) {
                    t.pid.store((int32_t)getpid());
                    t.inflight.store(0);
                    t.acked_epoch.store(0);
                    t.ack_status.store(KREX_OK);
                    t.state.store(1, std::memory_order_seq_cst);
                    {
                        std::lock_guard<std::mutex> lk(x->mu);
                        x->local[(size_t)i] = 1;
                        x->stream[(size_t)i] = reinterpret_cast<cudaStream_t>(stream);
                        x->device[(size_t)i] = dev;
                    }
                    reg_unlock(h);
                    *tenant = i;
                    return KREX_OK;
                }
            }
            reg_unlock(h);
            return set_error(KREX_ERR_INVALID, "gate_register: all %d tenant slots taken", h->max_tenants);
        }
        reg_unlock(h);
        if (!wait_gate(h, [&] { return h->holder.load() == -1; }, deadline))
            return set_error(KREX_ERR_TIMEOUT, "gate_register: gate stayed closed");
    }
}

krex_status xgate_unregister(XGate *x, int32_t i) {
    if (!local_tenant(x, i)) return set_error(KREX_ERR_INVALID, "gate_unregister: not a tenant of this process");
    XGateHdr *h = x->h;
    if (!reg_lock(h, deadline_from(0))) return set_error(KREX_ERR_TIMEOUT, "gate_unregister: registration lock");
    krex_status st = KREX_OK;
    const int32_t hold = h->holder.load();
    if (hold == i)
        st = set_error(KREX_ERR_STATE, "gate_unregister: tenant holds the gate");
    else if (hold != -1)
        st = set_error(KREX_ERR_STATE, "gate_unregister: gate closed (drained entries stay until the region ends)");
    else if (x->t[i].inflight.load() != 0)
        st = set_error(KREX_ERR_STATE, "gate_unregister: submission open");
    else
        x->t[i].state.store(0, std::memory_order_seq_cst);
    reg_unlock(h);
    if (st == KREX_OK) {
        std::lock_guard<std::mutex> lk(x->mu);
        x->local[(size_t)i] = 0;
        x->stream[(size_t)i] = nullptr;
    }
    return st;
}

krex_status xgate_submit_begin(XGate *x, int32_t i, int64_t timeout_us) {
    if (!local_tenant(x, i)) return set_error(KREX_ERR_INVALID, "gate_submit_begin: not a tenant of this process");
    XGateHdr *h = x->h;
    XTenant &t = x->t[i];
    const auto deadline = deadline_from(timeout_us);
    for (;;) {
        t.inflight.fetch_add(1, std::memory_order_seq_cst);            // increment first ...
        const int32_t hold = h->holder.load(std::memory_order_seq_cst);  // ... then check the gate
        if (hold == -1 || hold == i) return KREX_OK;
        t.inflight.fetch_sub(1, std::memory_order_seq_cst);            // retract and park
        h->parked.fetch_add(1);
        const bool reopened = wait_gate(h, [&] {
            const int32_t cur = h->holder.load();
            return cur == -1 || cur == i;
        }, deadline, 50000000);
        h->parked.fetch_sub(1);
        if (!reopened) return set_error(KREX_ERR_TIMEOUT, "gate_submit_begin: gate held past the timeout");
    }
}

krex_status xgate_submit_end(XGate *x, int32_t i) {
    if (!local_tenant(x, i)) return set_error(KREX_ERR_INVALID, "gate_submit_end: not a tenant of this process");
    XTenant &t = x->t[i];
    if (t.inflight.fetch_sub(1, std::memory_order_seq_cst) <= 0) {
        t.inflight.fetch_add(1);
        return set_error(KREX_ERR_STATE, "gate_submit_end without submit_begin");
    }
    return KREX_OK;
}

krex_status xgate_enter(XGate *x, int32_t holder, int64_t timeout_us, uint64_t *epoch) {
    if (!epoch || !local_tenant(x, holder))
        return set_error(KREX_ERR_INVALID, "gate_enter: holder must be a tenant of this process");
    XGateHdr *h = x->h;
    if (h->holder.load() == holder) return set_error(KREX_ERR_STATE, "gate_enter: already holding the gate");
    const auto deadline = deadline_from(timeout_us);
    // 1) region lock: one holder at a time, across processes
    auto try_lock = [&] {
        int32_t expected = -1;
        return h->region_owner.compare_exchange_strong(expected, holder, std::memory_order_seq_cst);
    };
    if (!wait_gate(h, try_lock, deadline)) return set_error(KREX_ERR_TIMEOUT, "gate_enter: region lock not acquired in time");
    // 2) claim the gate with a fresh epoch, serialised with registration
    if (!reg_lock(h, deadline)) {
        h->region_owner.store(-1, std::memory_order_seq_cst);
        gate_changed(h);
        return set_error(KREX_ERR_TIMEOUT, "gate_enter: registration lock");
    }
    reap_dead(x);
    const uint64_t e = h->epoch.load() + 1;
    h->epoch.store(e, std::memory_order_seq_cst);
    h->holder_pid.store((int32_t)getpid(), std::memory_order_seq_cst);
    h->holder.store(holder, std::memory_order_seq_cst);
    reg_unlock(h);
    gate_changed(h);  // wakes every process's drainer and parks new submissions
    auto fail = [&](krex_status st) {
        h->holder.store(-1, std::memory_order_seq_cst);  // a failing entry never starts measurement
        h->holder_pid.store(0);
        h->region_owner.store(-1, std::memory_order_seq_cst);
        gate_changed(h);
        return st;
    };
    // 3) poll every sibling: this epoch acknowledged by its process's drainer
    //    and a zero counter; a sibling whose process died fails the entry
    for (int32_t i = 0; i < h->max_tenants; ++i) {
        if (i == holder) continue;
        XTenant &t = x->t[i];
        uint32_t polls = 0;
        for (;;) {
            if (t.state.load(std::memory_order_seq_cst) != 1) break;  // left
            if (t.acked_epoch.load(std::memory_order_seq_cst) == e) {
                const int32_t ast = t.ack_status.load();
                if (ast != KREX_OK)
                    return fail(set_error((krex_status)ast, "gate_enter: tenant %d's drain failed", i));
                if (t.inflight.load(std::memory_order_seq_cst) == 0) break;
            }
            if ((++polls & 15u) == 0 && !pid_alive(t.pid.load()))
                return fail(set_error(KREX_ERR_STATE, "gate_enter: the process of tenant %d died during entry", i));
            if (clk::now() >= deadline)
                return fail(set_error(KREX_ERR_TIMEOUT, "gate_enter: tenant %d did not drain in time", i));
            if (polls < 256) continue;                       // spin first ...
            std::this_thread::sleep_for(std::chrono::microseconds(20));  // ... then short naps
        }
    }
    *epoch = e;
    return KREX_OK;
}

krex_status xgate_exit(XGate *x, int32_t holder, uint64_t epoch) {
    if (!local_tenant(x, holder)) return set_error(KREX_ERR_INVALID, "gate_exit: not a tenant of this process");
    XGateHdr *h = x->h;
    if (h->holder.load() != holder || h->epoch.load() != epoch)
        return set_error(KREX_ERR_STATE, "gate_exit: not the holder of epoch %llu", (unsigned long long)epoch);
    XTenant &t = x->t[holder];
    wait_gate(h, [&] { return t.inflight.load() == 0; }, deadline_from(0), 200000);
    h->holder.store(-1, std::memory_order_seq_cst);  // reopen the gate ...
    h->holder_pid.store(0);
    h->region_owner.store(-1, std::memory_order_seq_cst);  // ... release the lock
    gate_changed(h);
    return KREX_OK;
}

krex_status xgate_state(XGate *x, int32_t *holder, uint64_t *epoch, int32_t *parked) {
    if (holder) *holder = x->h->holder.load();
    if (epoch) *epoch = x->h->epoch.load();
    if (parked) *parked = x->h->parked.load();
    return KREX_OK;
}

krex_status xgate_recover(XGate *x, int32_t holder, uint64_t epoch) {
    XGateHdr *h = x->h;
    if (!reg_lock(h, deadline_from(0))) return set_error(KREX_ERR_TIMEOUT, "gate_recover: registration lock");
    krex_status st = KREX_OK;
    if (h->holder.load() != holder || h->epoch.load() != epoch) {
        st = set_error(KREX_ERR_STATE, "gate_recover: the gate is not held by %d with epoch %llu", holder,
                       (unsigned long long)epoch);
    } else if (pid_alive(h->holder_pid.load())) {
        st = set_error(KREX_ERR_STATE, "gate_recover: the holder's process is alive");
    } else {
        if (holder >= 0 && holder < h->max_tenants) {
            x->t[holder].inflight.store(0);
            x->t[holder].state.store(0, std::memory_order_seq_cst);
        }
        h->holder.store(-1, std::memory_order_seq_cst);
        h->holder_pid.store(0);
        int32_t owner = holder;
        h->region_owner.compare_exchange_strong(owner, -1, std::memory_order_seq_cst);
    }
    reg_unlock(h);
    if (st == KREX_OK) gate_changed(h);
    return st;
}

}  // namespace krex

using krex::set_error;

extern "C" {

// ---------------------------------------------------------------- ring -----

size_t krex_ring_bytes(uint32_t capacity, uint32_t entry_bytes) {
    return sizeof(krex::RingHdr) + (size_t)capacity * entry_bytes;
}

krex_status krex_ring_init(void *mem, size_t bytes, uint32_t capacity, uint32_t entry_bytes) {
    if (!mem || (reinterpret_cast<uintptr_t>(mem) & 63u))
        return set_error(KREX_ERR_INVALID, "ring_init: need 64-byte aligned memory");
    if (capacity < 2 || (capacity & (capacity - 1)) || capacity > (1u << 24))
        return set_error(KREX_ERR_INVALID, "ring_init: capacity must be a power of two in [2, 2^24]");
    if (entry_bytes < 8 || entry_bytes > 4096 || (entry_bytes & 7u))
        return set_error(KREX_ERR_INVALID, "ring_init: entry_bytes must be a multiple of 8 in [8, 4096]");
    if (bytes < krex_ring_bytes(capacity, entry_bytes))
        return set_error(KREX_ERR_INVALID, "ring_init: %zu bytes, need %zu", bytes, krex_ring_bytes(capacity, entry_bytes));
    memset(mem, 0, sizeof(krex::RingHdr));
    krex::RingHdr *r = new (mem) krex::RingHdr();
    r->version = krex::kVersion;
    r->capacity = capacity;
    r->entry_bytes = entry_bytes;
    r->spin_ns.store(20000);
    r->head.store(0);
    r->tail.store(0);
    r->data_seq.store(0);
    r->consumer_parked.store(0);
    r->space_seq.store(0);
    r->producer_parked.store(0);
    for (auto &c : r->stats) c.store(0);
    std::atomic_thread_fence(std::memory_order_seq_cst);
    r->magic = krex::kRingMagic;
    std::atomic_thread_fence(std::memory_order_seq_cst);
    return KREX_OK;
}

krex_status krex_ring_set_spin(void *ring, int64_t spin_us) {
    krex::RingHdr *r = krex::ring_of(ring);
    if (!r || spin_us < 0) return set_error(KREX_ERR_INVALID, "ring_set_spin: not a ring, or negative spin");
    r->spin_ns.store(spin_us * 1000);
    return KREX_OK;
}

krex_status krex_ring_push(void *ring, const void *entry, int64_t timeout_us) {
    krex::RingHdr *r = krex::ring_of(ring);
    if (!r || !entry) return set_error(KREX_ERR_INVALID, "ring_push: not a ring, or null entry");
    const uint64_t head = r->head.load(std::memory_order_relaxed);  // only the producer writes head
    auto space = [&] { return head - r->tail.load(std::memory_order_seq_cst) < r->capacity; };
    if (!krex::spin_park_futex(space, r->space_seq, r->producer_parked, r->spin_ns.load(),
                               krex::deadline_from(timeout_us), &r->stats[3]))
        return set_error(KREX_ERR_TIMEOUT, "ring_push: ring stayed full");
    memcpy(krex::ring_slot(r, head), entry, r->entry_bytes);
    r->head.store(head + 1, std::memory_order_seq_cst);
    r->stats[0].fetch_add(1, std::memory_order_relaxed);
    if (r->consumer_parked.load(std::memory_order_seq_cst)) {
        r->data_seq.fetch_add(1, std::memory_order_seq_cst);
        krex::futex_wake_all(&r->data_seq);
        r->stats[4].fetch_add(1, std::memory_order_relaxed);
    }
    return KREX_OK;
}

krex_status krex_ring_pop(void *ring, void *entry, int64_t timeout_us) {
    krex::RingHdr *r = krex::ring_of(ring);
    if (!r || !entry) return set_error(KREX_ERR_INVALID, "ring_pop: not a ring, or null entry");
    const uint64_t tail = r->tail.load(std::memory_order_relaxed);  // only the consumer writes tail
    auto data = [&] { return r->head.load(std::memory_order_seq_cst) != tail; };
    if (!krex::spin_park_futex(data, r->data_seq, r->consumer_parked, r->spin_ns.load(),
                               krex::deadline_from(timeout_us), &r->stats[2]))
        return set_error(KREX_ERR_TIMEOUT, "ring_pop: ring stayed empty");
    memcpy(entry, krex::ring_slot(r, tail), r->entry_bytes);
    r->tail.store(tail + 1, std::memory_order_seq_cst);
    r->stats[1].fetch_add(1, std::memory_order_relaxed);
    if (r->producer_parked.load(std::memory_order_seq_cst)) {
        r->space_seq.fetch_add(1, std::memory_order_seq_cst);
        krex::futex_wake_all(&r->space_seq);
        r->stats[4].fetch_add(1, std::memory_order_relaxed);
    }
    return KREX_OK;
}

krex_status krex_ring_count(void *ring, uint64_t *n) {
    krex::RingHdr *r = krex::ring_of(ring);
    if (!r || !n) return set_error(KREX_ERR_INVALID, "ring_count: not a ring, or null n");
    *n = r->head.load(std::memory_order_seq_cst) - r->tail.load(std::memory_order_seq_cst);
    return KREX_OK;
}

krex_status krex_ring_stats(void *ring, uint64_t *out5) {
    krex::RingHdr *r = krex::ring_of(ring);
    if (!r || !out5) return set_error(KREX_ERR_INVALID, "ring_stats: not a ring, or null out");
    for (int i = 0; i < 5; ++i) out5[i] = r->stats[i].load();
    return KREX_OK;
}

// ---------------------------------------------------------------- gate -----

size_t krex_gate_shared_bytes(int32_t max_tenants) {
    if (max_tenants < 1) max_tenants = 1;
    return sizeof(krex::XGateHdr) + (size_t)max_tenants * sizeof(krex::XTenant);
}

krex_status krex_gate_shared_init(void *mem, size_t bytes, int32_t max_tenants) {
    if (!mem || (reinterpret_cast<uintptr_t>(mem) & 63u))
        return set_error(KREX_ERR_INVALID, "gate_shared_init: need 64-byte aligned memory");
    if (max_tenants < 1 || max_tenants > 4096)
        return set_error(KREX_ERR_INVALID, "gate_shared_init: need 1 <= max_tenants <= 4096");
    if (bytes < krex_gate_shared_bytes(max_tenants))
        return set_error(KREX_ERR_INVALID, "gate_shared_init: %zu bytes, need %zu", bytes,
                         krex_gate_shared_bytes(max_tenants));
    memset(mem, 0, krex_gate_shared_bytes(max_tenants));
    krex::XGateHdr *h = new (mem) krex::XGateHdr();
    h->version = krex::kVersion;
    h->max_tenants = max_tenants;
    h->reg_lock.store(0);
    h->region_owner.store(-1);
    h->holder.store(-1);
    h->holder_pid.store(0);
    h->epoch.store(0);
    h->gate_seq.store(0);
    h->gate_waiters.store(0);
    h->parked.store(0);
    krex::XTenant *t = reinterpret_cast<krex::XTenant *>(h + 1);
    for (int32_t i = 0; i < max_tenants; ++i) {
        new (&t[i]) krex::XTenant();
        t[i].state.store(0);
        t[i].pid.store(0);
        t[i].inflight.store(0);
        t[i].acked_epoch.store(0);
        t[i].ack_status.store(0);
    }
    std::atomic_thread_fence(std::memory_order_seq_cst);
    h->magic = krex::kGateMagic;
    std::atomic_thread_fence(std::memory_order_seq_cst);
    return KREX_OK;
}

}  // extern "C"
