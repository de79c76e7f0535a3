"""Child-process bodies for the cross-process gate and ring tests (run under
the multiprocessing 'spawn' start method; CPU only)."""
import ctypes
import os
import time

import paper_2609_30057_gb300 as krex

# control words after the gate / rings in the shared file (int64 each)
CTRL_STOP, CTRL_READY, CTRL_INSIDE, CTRL_SUBMITS, CTRL_PARKS, CTRL_A, CTRL_B, CTRL_C = range(8)


def ctrl(m: "krex.SharedMap", off: int):
    return (ctypes.c_int64 * 8).from_address(m.addr + off)


def ring_producer(path, nbytes, ring_off, n, spin_us):
    m = krex.SharedMap(path, nbytes)
    r = krex.Ring(m.addr + ring_off)
    e = (ctypes.c_uint64 * 4)()
    for i in range(n):
        e[0], e[1] = i, i * 3 + 1
        r.push(e, timeout_us=5_000_000)


def ring_echo(path, nbytes, req_off, rep_off, n, spin_us):
    m = krex.SharedMap(path, nbytes)
    req, rep = krex.Ring(m.addr + req_off), krex.Ring(m.addr + rep_off)
    req.set_spin(spin_us)
    e = (ctypes.c_uint64 * 2)()
    for _ in range(n):
        req.pop_into(e, timeout_us=5_000_000)
        e[1] = e[0] + 1
        rep.push(e, timeout_us=5_000_000)


def gate_sibling(path, nbytes, ctrl_off):
    """Registers a tenant and submits in a loop until told to stop; counts
    itself 'inside' between submit_begin and submit_end."""
    m = krex.SharedMap(path, nbytes)
    c = ctrl(m, ctrl_off)
    g = krex.Gate.attach(m.addr, ctrl_off)
    t = g.register()
    c[CTRL_READY] = 1
    while not c[CTRL_STOP]:
        g.submit_begin(t, timeout_us=5_000_000)
        c[CTRL_INSIDE] += 1
        c[CTRL_SUBMITS] += 1
        c[CTRL_INSIDE] -= 1
        g.submit_end(t)
    g.unregister(t)
    g.close()


def gate_open_submission_then_sleep(path, nbytes, ctrl_off):
    """Registers, opens a submission and never closes it (until killed)."""
    m = krex.SharedMap(path, nbytes)
    c = ctrl(m, ctrl_off)
    g = krex.Gate.attach(m.addr, ctrl_off)
    t = g.register()
    g.submit_begin(t)
    c[CTRL_A] = t
    c[CTRL_READY] = 1
    time.sleep(60)


def gate_holder_dies(path, nbytes, ctrl_off):
    """Enters the gate as holder and exits the process without gate_exit."""
    m = krex.SharedMap(path, nbytes)
    c = ctrl(m, ctrl_off)
    g = krex.Gate.attach(m.addr, ctrl_off)
    t = g.register()
    e = g.enter(t, timeout_us=5_000_000)
    c[CTRL_A], c[CTRL_B] = t, e
    c[CTRL_READY] = 1
    os._exit(0)


def gate_register_timed(path, nbytes, ctrl_off):
    """Registers (waiting while the gate is closed) and reports how long it took."""
    m = krex.SharedMap(path, nbytes)
    c = ctrl(m, ctrl_off)
    g = krex.Gate.attach(m.addr, ctrl_off)
    c[CTRL_READY] = 1
    t0 = time.monotonic()
    t = g.register(timeout_us=5_000_000)
    c[CTRL_A] = int((time.monotonic() - t0) * 1e6)
    c[CTRL_B] = t
    g.unregister(t)
    g.close()
