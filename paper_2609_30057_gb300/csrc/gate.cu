// In-process form of the paper's in-region GPU exclusivity (Section 4.2,
// "GPU exclusivity", steps 1-3 and 8): a region lock admits one holder; the
// holder claims the gate with a fresh epoch; every other tenant's submissions
// are either covered by the drain or blocked before they reach CUDA.
//
//  - Submission (counter-and-gate): a tenant increments its in-flight counter,
//    then reads the gate.  If another tenant holds it, the tenant retracts the
//    increment and parks (spin briefly, then sleep on a condition variable)
//    until the gate changes; otherwise it submits and decrements afterwards,
//    on errors too.  All counter and gate accesses are sequentially consistent,
//    so a racing submission is either seen by the holder's drain (counter > 0)
//    or sees the closed gate (Dekker-style ordering).
//  - Entry: lock, claim the gate (holder, epoch), then for each sibling wait
//    for its counter to reach zero, synchronise its stream and record the
//    epoch as acknowledged.  The holder then polls until every sibling shows
//    this epoch's acknowledgement and a zero counter; a previous epoch's
//    acknowledgement never counts.  (A counter may rise for a moment after the
//    drain: the increment of a submission that then sees the closed gate and
//    retracts.)  A drain that runs out of time releases the
//    gate and the lock and fails the entry: measurement never starts.
//  - Registration is serialised with gate closure: a tenant registering while
//    the gate is closed waits for it to reopen.
//  - Exit is bound to the holder and the epoch of its entry: the holder's own
//    submissions finish, the gate reopens (parked tenants wake), the lock is
//    released.  A stale exit (wrong holder or epoch) is rejected.
// Host code only: no kernel is involved, so the protocol is testable with CPU
// threads (tenant streams may be NULL, which makes the stream drain a no-op).
#include <algorithm>
#include <atomic>
#include <chrono>
#include <condition_variable>
#include <memory>
#include <mutex>
#include <thread>
#include <vector>

#include "common.cuh"
#include "xproc.h"

namespace {

using clk = std::chrono::steady_clock;

struct Tenant {
    std::atomic<int64_t> inflight{0};
    std::atomic<uint64_t> acked_epoch{0};
    cudaStream_t stream = nullptr;
    bool registered = false;
};

}  // namespace

struct krex_gate {
    krex::XGate *x = nullptr;             // non-null: the gate lives in shared memory (xproc.cu)
    int32_t max_tenants = 0;
    std::unique_ptr<Tenant[]> tenants;
    std::atomic<int32_t> holder{-1};      // -1: gate open
    std::atomic<uint64_t> epoch{0};       // epoch of the current / last entry
    std::atomic<int32_t> parked{0};       // tenants waiting for the gate
    std::atomic<bool> region_locked{false};  // admits one holder at a time (any thread may release)
    std::mutex reg_mu;                    // registration vs. gate closure
    std::mutex park_mu;
    std::condition_variable park_cv;
};

namespace {

// Spin for ~20 us, then sleep with growing naps (the spin-park policy of
// Section 4.3) until pred() or the deadline.
template <class Pred>
bool spin_park(Pred pred, clk::time_point deadline) {
    const auto spin_until = clk::now() + std::chrono::microseconds(20);
    while (clk::now() < spin_until)
        if (pred()) return true;
    long nap_us = 5;
    while (!pred()) {
        if (clk::now() >= deadline) return false;
        std::this_thread::sleep_for(std::chrono::microseconds(nap_us));
        nap_us = std::min(nap_us * 2, 1000L);
    }
    return true;
}

clk::time_point deadline_from(int64_t timeout_us) {
    if (timeout_us <= 0) timeout_us = 10 * 1000 * 1000;
    return clk::now() + std::chrono::microseconds(timeout_us);
}

bool valid_tenant(const krex_gate *g, int32_t t) {
    return g && t >= 0 && t < g->max_tenants && g->tenants[t].registered;
}

void wake_parked(krex_gate *g) {
    std::lock_guard<std::mutex> lk(g->park_mu);
    g->park_cv.notify_all();
}

}  // namespace

using krex::set_error;

extern "C" {

krex_status krex_gate_create(krex_gate **g, int32_t max_tenants) {
    if (!g || max_tenants < 1 || max_tenants > 4096)
        return set_error(KREX_ERR_INVALID, "gate_create: need g and 1 <= max_tenants <= 4096");
    krex_gate *x = new krex_gate();
    x->max_tenants = max_tenants;
    x->tenants.reset(new Tenant[max_tenants]);
    *g = x;
    return KREX_OK;
}

krex_status krex_gate_destroy(krex_gate *g) {
    if (!g) return set_error(KREX_ERR_INVALID, "gate is null");
    if (g->x) {
        krex_status st = krex::xgate_detach(g->x);
        if (st == KREX_OK) delete g;
        return st;
    }
    if (g->holder.load() != -1) return set_error(KREX_ERR_STATE, "gate_destroy while a holder is inside");
    delete g;
    return KREX_OK;
}

krex_status krex_gate_register(krex_gate *g, krex_stream_t stream, int64_t timeout_us, int32_t *tenant) {
    if (!g || !tenant) return set_error(KREX_ERR_INVALID, "gate_register: null argument");
    if (g->x) return krex::xgate_register(g->x, stream, timeout_us, tenant);
    const auto deadline = deadline_from(timeout_us);
    for (;;) {
        {
            std::lock_guard<std::mutex> lk(g->reg_mu);
            if (g->holder.load() == -1) {  // serialised with closure: only while the gate is open
                for (int32_t t = 0; t < g->max_tenants; ++t) {
                    Tenant &x = g->tenants[t];
                    if (!x.registered) {
                        x.registered = true;
                        x.stream = reinterpret_cast<cudaStream_t>(stream);
                        x.inflight.store(0);
                        x.acked_epoch.store(0);
                        *tenant = t;
                        return KREX_OK;
                    }
                }
                return set_error(KREX_ERR_INVALID, "gate_register: all %d tenant slots taken", g->max_tenants);
            }
        }
        if (!spin_park([&] { return g->holder.load() == -1; }, deadline))
            return set_error(KREX_ERR_TIMEOUT, "gate_register: gate stayed closed");
    }
}

krex_status krex_gate_unregister(krex_gate *g, int32_t tenant) {
    if (g && g->x) return krex::xgate_unregister(g->x, tenant);
    if (!valid_tenant(g, tenant)) return set_error(KREX_ERR_INVALID, "gate_unregister: bad tenant");
    std::lock_guard<std::mutex> lk(g->reg_mu);
    if (g->holder.load() == tenant) return set_error(KREX_ERR_STATE, "gate_unregister: tenant holds the gate");
    if (g->tenants[tenant].inflight.load() != 0) return set_error(KREX_ERR_STATE, "gate_unregister: submission open");
    g->tenants[tenant].registered = false;
    return KREX_OK;
}

krex_status krex_gate_submit_begin(krex_gate *g, int32_t tenant, int64_t timeout_us) {
    if (g && g->x) return krex::xgate_submit_begin(g->x, tenant, timeout_us);
    if (!valid_tenant(g, tenant)) return set_error(KREX_ERR_INVALID, "gate_submit_begin: bad tenant");
    Tenant &x = g->tenants[tenant];
    const auto deadline = deadline_from(timeout_us);
    for (;;) {
        x.inflight.fetch_add(1, std::memory_order_seq_cst);        // increment first ...
        const int32_t h = g->holder.load(std::memory_order_seq_cst); // ... then check the gate
        if (h == -1 || h == tenant) return KREX_OK;
        x.inflight.fetch_sub(1, std::memory_order_seq_cst);        // retract and park
        g->parked.fetch_add(1);
        bool reopened;
        {
            std::unique_lock<std::mutex> lk(g->park_mu);
            reopened = g->park_cv.wait_until(lk, deadline, [&] {
                const int32_t cur = g->holder.load();
                return cur == -1 || cur == tenant;
            });
        }
        g->parked.fetch_sub(1);
        if (!reopened) return set_error(KREX_ERR_TIMEOUT, "gate_submit_begin: gate held past the timeout");
    }
}

krex_status krex_gate_submit_end(krex_gate *g, int32_t tenant) {
    if (g && g->x) return krex::xgate_submit_end(g->x, tenant);
    if (!valid_tenant(g, tenant)) return set_error(KREX_ERR_INVALID, "gate_submit_end: bad tenant");
    Tenant &x = g->tenants[tenant];
    if (x.inflight.fetch_sub(1, std::memory_order_seq_cst) <= 0) {
        x.inflight.fetch_add(1);
        return set_error(KREX_ERR_STATE, "gate_submit_end without submit_begin");
    }
    return KREX_OK;
}

krex_status krex_gate_enter(krex_gate *g, int32_t holder, int64_t timeout_us, uint64_t *epoch) {
    if (g && g->x) return krex::xgate_enter(g->x, holder, timeout_us, epoch);
    if (!valid_tenant(g, holder) || !epoch) return set_error(KREX_ERR_INVALID, "gate_enter: bad holder or epoch");
    if (g->holder.load() == holder) return set_error(KREX_ERR_STATE, "gate_enter: already holding the gate");
    const auto deadline = deadline_from(timeout_us);
    // 1) region lock: one holder at a time
    auto try_lock = [&] {
        bool expected = false;
        return g->region_locked.compare_exchange_strong(expected, true, std::memory_order_seq_cst);
    };
    if (!spin_park(try_lock, deadline)) return set_error(KREX_ERR_TIMEOUT, "gate_enter: region lock not acquired in time");
    // 2) claim the gate with a fresh epoch (serialised with registration)
    uint64_t e;
    {
        std::lock_guard<std::mutex> lk(g->reg_mu);
        e = g->epoch.load() + 1;
        g->epoch.store(e, std::memory_order_seq_cst);
        g->holder.store(holder, std::memory_order_seq_cst);
    }
    // 3) drain every sibling: counter -> 0, stream synchronised, epoch acknowledged
    for (int32_t t = 0; t < g->max_tenants; ++t) {
        Tenant &x = g->tenants[t];
        if (!x.registered || t == holder) continue;
        const bool idle = spin_park([&] { return x.inflight.load(std::memory_order_seq_cst) == 0; }, deadline);
        cudaError_t err = cudaSuccess;
        if (idle && x.stream) err = cudaStreamSynchronize(x.stream);
        if (!idle || err != cudaSuccess) {
            // a failing entry never starts measurement: reopen and release
            g->holder.store(-1, std::memory_order_seq_cst);
            wake_parked(g);
            g->region_locked.store(false, std::memory_order_seq_cst);
            if (!idle) return set_error(KREX_ERR_TIMEOUT, "gate_enter: tenant %d did not drain in time", t);
            return krex::cuda_error(err, "cudaStreamSynchronize (gate drain)");
        }
        x.acked_epoch.store(e, std::memory_order_seq_cst);
    }
    // The holder polls until every sibling shows this epoch's acknowledgement
    // and a zero counter.  A counter can rise for a moment after the drain:
    // the increment of a submission that then sees the closed gate and
    // retracts, so the counters are polled (within the entry deadline), not
    // read once.
    for (int32_t t = 0; t < g->max_tenants; ++t) {
        Tenant &x = g->tenants[t];
        if (!x.registered || t == holder) continue;
        if (x.acked_epoch.load() != e) {
            g->holder.store(-1, std::memory_order_seq_cst);
            wake_parked(g);
            g->region_locked.store(false, std::memory_order_seq_cst);
            return set_error(KREX_ERR_STATE, "gate_enter: tenant %d acknowledgement does not match epoch", t);
        }
        if (!spin_park([&] { return x.inflight.load(std::memory_order_seq_cst) == 0; }, deadline)) {
            g->holder.store(-1, std::memory_order_seq_cst);
            wake_parked(g);
            g->region_locked.store(false, std::memory_order_seq_cst);
            return set_error(KREX_ERR_TIMEOUT, "gate_enter: tenant %d counter stayed non-zero", t);
        }
    }
    *epoch = e;
    return KREX_OK;
}

krex_status krex_gate_exit(krex_gate *g, int32_t holder, uint64_t epoch) {
    if (g && g->x) return krex::xgate_exit(g->x, holder, epoch);
    if (!valid_tenant(g, holder)) return set_error(KREX_ERR_INVALID, "gate_exit: bad holder");
    if (g->holder.load() != holder || g->epoch.load() != epoch)
        return set_error(KREX_ERR_STATE, "gate_exit: not the holder of epoch %llu", (unsigned long long)epoch);
    // the holder's own submissions finish host-side first
    Tenant &x = g->tenants[holder];
    spin_park([&] { return x.inflight.load() == 0; }, deadline_from(0));
    g->holder.store(-1, std::memory_order_seq_cst);  // reopen the gate ...
    wake_parked(g);
    g->region_locked.store(false, std::memory_order_seq_cst);                          // ... then release the lock
    return KREX_OK;
}

krex_status krex_gate_state(krex_gate *g, int32_t *holder, uint64_t *epoch, int32_t *parked) {
    if (!g) return set_error(KREX_ERR_INVALID, "gate is null");
    if (g->x) return krex::xgate_state(g->x, holder, epoch, parked);
    if (holder) *holder = g->holder.load();
    if (epoch) *epoch = g->epoch.load();
    if (parked) *parked = g->parked.load();
    return KREX_OK;
}

krex_status krex_gate_shared_attach(void *mem, size_t bytes, krex_gate **g) {
    if (!g) return set_error(KREX_ERR_INVALID, "gate_shared_attach: null out");
    krex::XGate *x = nullptr;
    krex_status st = krex::xgate_attach(mem, bytes, &x);
    if (st) return st;
    krex_gate *h = new krex_gate();
    h->x = x;
    *g = h;
    return KREX_OK;
}

krex_status krex_gate_recover(krex_gate *g, int32_t holder, uint64_t epoch) {
    if (!g || !g->x) return set_error(KREX_ERR_INVALID, "gate_recover: needs a shared gate");
    return krex::xgate_recover(g->x, holder, epoch);
}

}  // extern "C"
