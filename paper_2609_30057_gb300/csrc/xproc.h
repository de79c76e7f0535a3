// Internal: the cross-process form of the in-region gate and the
// shared-memory SPSC ring (xproc.cu), used by gate.cu's dispatch.
#pragma once

#include <stdint.h>

#include "krex.h"

namespace krex {

struct XGate;  // process-local view of a gate in shared memory

krex_status xgate_attach(void *mem, size_t bytes, XGate **out);
krex_status xgate_detach(XGate *x);
krex_status xgate_register(XGate *x, krex_stream_t stream, int64_t timeout_us, int32_t *tenant);
krex_status xgate_unregister(XGate *x, int32_t tenant);
krex_status xgate_submit_begin(XGate *x, int32_t tenant, int64_t timeout_us);
krex_status xgate_submit_end(XGate *x, int32_t tenant);
krex_status xgate_enter(XGate *x, int32_t holder, int64_t timeout_us, uint64_t *epoch);
krex_status xgate_exit(XGate *x, int32_t holder, uint64_t epoch);
krex_status xgate_state(XGate *x, int32_t *holder, uint64_t *epoch, int32_t *parked);
krex_status xgate_recover(XGate *x, int32_t holder, uint64_t epoch);

}  // namespace krex
