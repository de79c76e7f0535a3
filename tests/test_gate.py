"""The in-region gate (paper Section 4.2, in-process form) on CPU threads.

Tenants with no stream (NULL) make the drain's stream synchronisation a
no-op, so the protocol's ordering invariants are tested with host threads
only: no GPU, no kernel.
"""
import threading
import time

import pytest

import paper_2609_30057_gb300 as krex


@pytest.fixture
def gate():
    krex.build()
    g = krex.Gate(8)
    yield g
    g.close()


def test_submissions_pass_while_open_and_park_while_held(gate):
    holder, sib = gate.register(), gate.register()
    with gate.submission(sib):
        pass
    epoch = gate.enter(holder)
    assert gate.state()[:2] == (holder, epoch)
    done = threading.Event()

    def sibling():
        with gate.submission(sib, timeout_us=5_000_000):
            done.set()

    th = threading.Thread(target=sibling)
    th.start()
    time.sleep(0.2)
    assert not done.is_set()                 # parked: nothing submitted inside the region
    assert gate.state()[2] == 1
    with gate.submission(holder):           # the holder itself may submit
        pass
    gate.exit(holder, epoch)
    th.join(2)
    assert done.is_set() and gate.state()[0] == -1


def test_entry_drains_an_open_submission(gate):
    holder, sib = gate.register(), gate.register()
    gate.submit_begin(sib)                  # sibling is inside a submission
    entered = threading.Event()

    def enter():
        e = gate.enter(holder, timeout_us=5_000_000)
        entered.set()
        gate.exit(holder, e)

    th = threading.Thread(target=enter)
    th.start()
    time.sleep(0.2)
    assert not entered.is_set()             # the drain waits for the counter to reach 0
    gate.submit_end(sib)
    th.join(2)
    assert entered.is_set()


def test_failing_entry_releases_the_gate(gate):
    holder, sib = gate.register(), gate.register()
    gate.submit_begin(sib)
    t0 = time.time()
    with pytest.raises(krex.KrexError, match="TIMEOUT"):
        gate.enter(holder, timeout_us=100_000)
    assert time.time() - t0 < 2.0
    assert gate.state()[0] == -1            # reopened: measurement never started
    gate.submit_end(sib)
    e = gate.enter(holder, timeout_us=1_000_000)
    gate.exit(holder, e)


def test_exit_is_bound_to_holder_and_epoch(gate):
    a, b = gate.register(), gate.register()
    e1 = gate.enter(a)
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.enter(a)                        # nested entry by the holder
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.exit(b, e1)                     # not the holder
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.exit(a, e1 - 1)                 # stale epoch
    gate.exit(a, e1)
    e2 = gate.enter(b)
    assert e2 == e1 + 1                      # every entry has a fresh epoch
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.exit(a, e1)                     # a delayed exit of the old entry cannot reopen it
    gate.exit(b, e2)


def test_second_holder_waits_for_the_region_lock(gate):
    a, b = gate.register(), gate.register()
    e = gate.enter(a)
    with pytest.raises(krex.KrexError, match="TIMEOUT"):
        gate.enter(b, timeout_us=100_000)
    assert gate.state()[0] == a              # the failed attempt did not touch a's claim
    gate.exit(a, e)
    gate.exit(b, gate.enter(b, timeout_us=1_000_000))


def test_registration_waits_while_the_gate_is_closed(gate):
    a = gate.register()
    e = gate.enter(a)
    got = []
    th = threading.Thread(target=lambda: got.append(gate.register(timeout_us=5_000_000)))
    th.start()
    time.sleep(0.2)
    assert not got
    gate.exit(a, e)
    th.join(2)
    assert len(got) == 1


def test_unregister_rules(gate):
    a, b = gate.register(), gate.register()
    gate.submit_begin(b)
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.unregister(b)
    gate.submit_end(b)
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.submit_end(b)                   # unbalanced end
    e = gate.enter(a)
    with pytest.raises(krex.KrexError, match="STATE"):
        gate.unregister(a)
    gate.exit(a, e)
    gate.unregister(b)


def test_no_sibling_submission_inside_a_region_under_races(gate):
    """Stress the increment-before-check ordering: siblings submit in tight
    loops while a holder enters and exits repeatedly; inside every region no
    sibling may be between submit_begin and submit_end."""
    holder = gate.register()
    sibs = [gate.register() for _ in range(3)]
    inside = [0]
    lock = threading.Lock()
    violations = []
    stop = threading.Event()

    def sibling(t):
        while not stop.is_set():
            gate.submit_begin(t, timeout_us=5_000_000)
            with lock:
                inside[0] += 1
            with lock:
                inside[0] -= 1
            gate.submit_end(t)

    threads = [threading.Thread(target=sibling, args=(t,)) for t in sibs]
    for th in threads:
        th.start()
    for _ in range(200):
        e = gate.enter(holder, timeout_us=5_000_000)
        with lock:
            if inside[0] != 0:
                violations.append(inside[0])
        time.sleep(0.0002)
        with lock:
            if inside[0] != 0:
                violations.append(inside[0])
        gate.exit(holder, e)
    stop.set()
    for th in threads:
        th.join(5)
    assert not violations
    assert gate.state()[1] == 200
