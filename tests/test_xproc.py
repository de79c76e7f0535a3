"""The cross-process gate and the shared-memory SPSC ring (paper Sections 4.2
and 4.3), host-only: spawned processes on the CPU, no GPU, no stream (tenant
streams are NULL, so the drain's synchronisation is a no-op)."""
import ctypes
import multiprocessing as mp
import os
import statistics
import threading
import time

import pytest

import paper_2609_30057_gb300 as krex
import xproc_workers as W


@pytest.fixture(scope="module", autouse=True)
def built():
    krex.build()


@pytest.fixture
def shm(tmp_path):
    """A shared file (under /dev/shm when it exists) mapped by every process."""
    base = "/dev/shm" if os.path.isdir("/dev/shm") else str(tmp_path)
    path = os.path.join(base, f"krex_test_{os.getpid()}_{time.monotonic_ns()}")
    maps = []

    def make(nbytes):
        m = krex.SharedMap(path, nbytes, create=True)
        maps.append(m)
        return m

    yield path, make
    if os.path.exists(path):
        os.unlink(path)


def _spawn(target, *args):
    p = mp.get_context("spawn").Process(target=target, args=args, daemon=True)
    p.start()
    return p


def _wait(pred, timeout=20.0):
    t0 = time.monotonic()
    while not pred():
        if time.monotonic() - t0 > timeout:
            raise TimeoutError
        time.sleep(0.005)


# ------------------------------------------------------------------ ring ----

def test_ring_order_wraparound_full_and_empty(shm):
    path, make = shm
    nb = krex.Ring.nbytes(8, 16)
    m = make(nb)
    r = krex.Ring.init(m.addr, nb, 8, 16)
    e = (ctypes.c_uint64 * 2)()
    for i in range(8):
        e[0], e[1] = i, ~i & 0xFFFF
        r.push(e)
    assert r.count() == 8
    t0 = time.monotonic()
    with pytest.raises(krex.KrexError, match="TIMEOUT"):
        r.push(e, timeout_us=30_000)              # full
    assert 0.02 < time.monotonic() - t0 < 2.0
    out = (ctypes.c_uint64 * 2)()
    for i in range(8):
        r.pop_into(out)
        assert (out[0], out[1]) == (i, ~i & 0xFFFF)
    with pytest.raises(krex.KrexError, match="TIMEOUT"):
        r.pop_into(out, timeout_us=30_000)        # empty
    for i in range(1000):                         # many laps of the 8 slots
        e[0] = 100 + i
        r.push(e)
        r.pop_into(out)
        assert out[0] == 100 + i
    s = r.stats()
    assert s["pushes"] == s["pops"] == 1008


def test_ring_rejects_bad_layouts(shm):
    path, make = shm
    m = make(1 << 16)
    lib = krex.lib()
    assert lib.krex_ring_init(m.addr, 1 << 16, 6, 16) == krex.KREX_ERR_INVALID       # not a power of two
    assert lib.krex_ring_init(m.addr, 1 << 16, 8, 12) == krex.KREX_ERR_INVALID       # entry not a multiple of 8
    assert lib.krex_ring_init(m.addr, 64, 8, 16) == krex.KREX_ERR_INVALID            # too small
    assert lib.krex_ring_init(m.addr + 8, 1 << 15, 8, 16) == krex.KREX_ERR_INVALID   # not 64-byte aligned
    with pytest.raises(krex.KrexError, match="INVALID"):
        krex.Ring(m.addr)                                                             # never formatted


@pytest.mark.parametrize("spin_us", [0, 20])
def test_ring_between_processes_keeps_order(shm, spin_us):
    path, make = shm
    nb = krex.Ring.nbytes(64, 32)
    m = make(nb)
    r = krex.Ring.init(m.addr, nb, 64, 32)
    r.set_spin(spin_us)
    n = 20000
    p = _spawn(W.ring_producer, path, nb, 0, n, spin_us)
    e = (ctypes.c_uint64 * 4)()
    for i in range(n):
        r.pop_into(e, timeout_us=10_000_000)
        assert (e[0], e[1]) == (i, i * 3 + 1)
    p.join(20)
    assert p.exitcode == 0
    s = r.stats()
    assert s["pushes"] == s["pops"] == n


def _ping_pong(shm, spin_us, n=3000):
    path, make = shm
    nb1 = krex.Ring.nbytes(16, 16)
    m = make(2 * nb1)
    req = krex.Ring.init(m.addr, nb1, 16, 16)
    rep = krex.Ring.init(m.addr + nb1, nb1, 16, 16)
    rep.set_spin(spin_us)
    p = _spawn(W.ring_echo, path, 2 * nb1, 0, nb1, n, spin_us)
    e, out = (ctypes.c_uint64 * 2)(), (ctypes.c_uint64 * 2)()
    rtt = []
    for i in range(n):
        e[0] = i
        t0 = time.perf_counter_ns()
        req.push(e, timeout_us=5_000_000)
        rep.pop_into(out, timeout_us=5_000_000)
        rtt.append(time.perf_counter_ns() - t0)
        assert out[1] == i + 1
    p.join(20)
    assert p.exitcode == 0
    parks = req.stats()["consumer_parks"] + rep.stats()["consumer_parks"]
    return statistics.median(rtt[100:]), parks


def test_spin_park_avoids_most_parks_in_a_ping_pong(shm):
    # Section 4.3: a reply that arrives within the spinning interval is taken
    # without a futex park and wake-up; parking at once parks on every wait
    rtt_spin, parks_spin = _ping_pong(shm, 200)
    rtt_park, parks_park = _ping_pong(shm, 0)
    assert parks_park > 1000
    assert parks_spin < parks_park / 4, (parks_spin, parks_park, rtt_spin, rtt_park)


# ------------------------------------------------------------------ gate ----

def _gate_map(make, tenants=8):
    gb = (krex.gate_shared_bytes(tenants) + 63) // 64 * 64
    m = make(gb + 64)
    krex.gate_shared_init(m.addr, gb, tenants)
    return m, gb


def test_shared_gate_protocol_in_one_process(shm):
    # two attachments in one process behave like two processes' views
    path, make = shm
    m, gb = _gate_map(make)
    a, b = krex.Gate.attach(m.addr, gb), krex.Gate.attach(m.addr, gb)
    holder, sib = a.register(), b.register()
    e = a.enter(holder)
    assert a.state()[:2] == b.state()[:2] == (holder, e)
    done = threading.Event()

    def sibling():
        with b.submission(sib, timeout_us=5_000_000):
            done.set()

    th = threading.Thread(target=sibling)
    th.start()
    time.sleep(0.2)
    assert not done.is_set()                      # parked while the gate is held
    with pytest.raises(krex.KrexError, match="STATE"):
        b.unregister(sib)                         # drained entries stay until the region ends
    with pytest.raises(krex.KrexError, match="STATE"):
        a.exit(holder, e + 1)                     # stale epoch
    a.exit(holder, e)
    th.join(2)
    assert done.is_set()
    with pytest.raises(krex.KrexError, match="INVALID"):
        a.submit_begin(sib)                       # a tenant of the other attachment
    with pytest.raises(krex.KrexError, match="STATE"):
        a.recover(holder, e)                      # not held
    b.unregister(sib)
    a.unregister(holder)
    a.close()
    b.close()


def test_no_sibling_submission_inside_a_region_across_processes(shm):
    path, make = shm
    m, gb = _gate_map(make)
    c = W.ctrl(m, gb)
    g = krex.Gate.attach(m.addr, gb)
    holder = g.register()
    p = _spawn(W.gate_sibling, path, gb + 64, gb)
    _wait(lambda: c[W.CTRL_READY] == 1)
    _wait(lambda: c[W.CTRL_SUBMITS] > 100)
    submits0 = int(c[W.CTRL_SUBMITS])
    violations, last = 0, 0
    for i in range(100):
        e = g.enter(holder, timeout_us=5_000_000)
        before = c[W.CTRL_SUBMITS]
        if c[W.CTRL_INSIDE] != 0:
            violations += 1
        time.sleep(0.001)
        if c[W.CTRL_INSIDE] != 0 or c[W.CTRL_SUBMITS] != before:
            violations += 1                       # the sibling submitted inside the region
        g.exit(holder, e)
        assert e == last + 1
        last = e
    c[W.CTRL_STOP] = 1
    p.join(20)
    assert p.exitcode == 0
    assert violations == 0
    assert c[W.CTRL_SUBMITS] > submits0           # it kept submitting between regions
    g.close()


def test_sibling_death_during_entry_fails_the_entry(shm):
    path, make = shm
    m, gb = _gate_map(make)
    c = W.ctrl(m, gb)
    g = krex.Gate.attach(m.addr, gb)
    holder = g.register()
    p = _spawn(W.gate_open_submission_then_sleep, path, gb + 64, gb)
    _wait(lambda: c[W.CTRL_READY] == 1)
    result = {}

    def enter():
        t0 = time.monotonic()
        try:
            g.enter(holder, timeout_us=8_000_000)
            result["ok"] = True
        except krex.KrexError as ex:
            result["err"] = str(ex)
        result["s"] = time.monotonic() - t0

    th = threading.Thread(target=enter)
    th.start()
    time.sleep(0.3)
    assert th.is_alive()                          # draining: the sibling's submission is open
    p.kill()
    p.join(10)
    th.join(10)
    assert "STATE" in result.get("err", "") and "died" in result["err"], result
    assert result["s"] < 3.0
    assert g.state()[0] == -1                     # a failing entry reopens the gate
    e = g.enter(holder, timeout_us=2_000_000)     # the dead tenant's slot is reaped
    g.exit(holder, e)
    g.close()


def test_dead_holder_is_recovered_bound_to_holder_and_epoch(shm):
    path, make = shm
    m, gb = _gate_map(make)
    c = W.ctrl(m, gb)
    g = krex.Gate.attach(m.addr, gb)
    me = g.register()
    p = _spawn(W.gate_holder_dies, path, gb + 64, gb)
    p.join(20)
    assert c[W.CTRL_READY] == 1
    dead, e = int(c[W.CTRL_A]), int(c[W.CTRL_B])
    assert g.state()[:2] == (dead, e)             # the gate stays closed after the holder's death
    with pytest.raises(krex.KrexError, match="STATE"):
        g.recover(dead, e + 1)                    # bound to the entry's epoch
    with pytest.raises(krex.KrexError, match="STATE"):
        g.recover(me, e)                          # bound to the holder
    g.recover(dead, e)
    assert g.state()[0] == -1
    e2 = g.enter(me, timeout_us=2_000_000)
    assert e2 == e + 1
    with pytest.raises(krex.KrexError, match="STATE"):
        g.recover(me, e2)                         # the holder is alive
    with pytest.raises(krex.KrexError, match="STATE"):
        g.recover(dead, e)                        # a delayed recovery cannot reopen a later entry
    assert g.state()[:2] == (me, e2)
    g.exit(me, e2)
    g.close()


def test_registration_in_another_process_waits_for_the_gate(shm):
    path, make = shm
    m, gb = _gate_map(make)
    c = W.ctrl(m, gb)
    g = krex.Gate.attach(m.addr, gb)
    holder = g.register()
    e = g.enter(holder)
    p = _spawn(W.gate_register_timed, path, gb + 64, gb)
    _wait(lambda: c[W.CTRL_READY] == 1)
    time.sleep(0.4)
    g.exit(holder, e)
    p.join(20)
    assert p.exitcode == 0
    assert c[W.CTRL_A] > 250_000                  # registered only after the gate reopened
    g.close()
