"""Pins for the oracle's Task Scheduler (Algorithms 2-3, Sec. 3.4.1) and
FedAsync aggregation (Algorithm 4) — CPU only.

Worked examples derived by hand from the algorithms live in tests/golden/.
The rest are closed forms (running mean, round robin), invariants (balance,
cap, slot conservation) and brute-force enumeration of small event orders.
"""
import itertools
import os
from collections import deque

import numpy as np
import pytest

from oracle import fo_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
NAMES = {"OK": O.OK, "EMPTY": O.EMPTY, "FULL": O.FULL, "STALE": O.STALE}


def golden_lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [l.split() for l in f if l.strip() and not l.startswith("#")]


# --------------------------------------------------------------------------
# scheduler
# --------------------------------------------------------------------------

def test_tiny_schedule_matches_hand_derived_golden():
    s = O.TaskScheduler(K=4, omega=8, depth=2)
    for f in golden_lines("sched_tiny_order.txt"):
        if f[0] == "enqueue":
            st, slot = s.put(int(f[1]))
            assert (st, slot, int(s.on[int(f[1])])) == (NAMES[f[3]], int(f[4]), int(f[5]))
        else:
            st, k, slot = s.get()
            assert (st, k, slot) == (NAMES[f[2]], int(f[3]), int(f[4]))
            assert s.c == [int(v) for v in f[5:9]]


def replay_slot_reuse_golden(put, get, counters, sender_on):
    """Replays tests/golden/sched_slot_reuse.txt (3 devices, depth 2, omega 3)
    through the given put / get and state readers."""
    for f in golden_lines("sched_slot_reuse.txt"):
        if f[0] == "enqueue":
            k = int(f[1])
            st, slot = put(k)
            assert (st, slot, int(sender_on()[k])) == (NAMES[f[3]], int(f[4]), int(f[5])), f
        else:
            st, k, slot = get()
            assert (st, k, slot) == (NAMES[f[2]], int(f[3]), int(f[4])), f
            assert list(counters()) == [int(v) for v in f[5:8]], f
            assert [int(v) for v in sender_on()] == [int(v) for v in f[9:12]], f


def test_slot_reuse_matches_hand_derived_golden():
    """Freed slots are reused in the order they were freed, a device refused
    with an empty queue is turned on by the next dequeue, and one refused
    with a non-empty queue only by a dequeue of its own."""
    s = O.TaskScheduler(K=3, omega=3, depth=2)
    replay_slot_reuse_golden(s.put, s.get, lambda: s.c, lambda: s.on)


def test_backlogged_queues_are_served_round_robin():
    K = 7
    s = O.TaskScheduler(K, omega=K * 3, depth=3)
    served = []
    for _ in range(40):
        for k in range(K):          # keep every queue backlogged
            if len(s.q[k]) < 2:
                assert s.put(k)[0] == O.OK
        served.append(s.get()[1])
    assert served == [i % K for i in range(40)]


def random_trace(seed, K, n, p_step=0.45):
    r = np.random.default_rng(seed)
    return [("step",) if r.random() < p_step else ("enq", int(r.integers(K))) for _ in range(n)]


def check_invariants(s, omega, depth):
    queued = [slot for q in s.q for slot in q]
    assert len(queued) == len(set(queued))                    # no slot twice
    assert sorted(queued + list(s.free)) == list(range(omega))  # slots conserved
    assert sum(len(q) for q in s.q) <= omega                  # global cap (Sec. 3.4.1)
    assert all(len(q) <= depth for q in s.q)


@pytest.mark.parametrize("seed", range(20))
def test_random_traces_keep_invariants_and_pick_min_counter(seed):
    K, omega, depth = 5, 7, 3
    s = O.TaskScheduler(K, omega, depth)
    fifo = [deque() for _ in range(K)]
    for ev in random_trace(seed, K, 300):
        if ev[0] == "enq":
            st, slot = s.put(ev[1])
            if st == O.OK:
                fifo[ev[1]].append(slot)
        else:
            nonempty = [k for k in range(K) if s.q[k]]
            before = list(s.c)
            st, k, slot = s.get()
            if not nonempty:
                assert st == O.EMPTY and s.c == before
                continue
            assert before[k] == min(before[j] for j in nonempty)
            assert k == min(j for j in nonempty if before[j] == before[k])
            assert slot == fifo[k].popleft()                  # FIFO within a device
        check_invariants(s, omega, depth)


def test_balance_of_continuously_backlogged_devices():
    """With every queue non-empty at every step, max c - min c <= 1."""
    K = 6
    s = O.TaskScheduler(K, omega=24, depth=4)
    r = np.random.default_rng(0)
    for _ in range(500):
        for k in r.permutation(K):
            if not s.q[k]:
                s.put(int(k))
        for _ in range(int(r.integers(1, 4))):
            if all(s.q):
                s.put(int(r.integers(K)))
        assert all(s.q)
        s.get()
        assert max(s.c) - min(s.c) <= 1


def literal_alg3(queues, c):
    """Algorithm 3's activation branch restricted to non-empty queues, written
    as a direct scan (ties to the lowest index)."""
    best = None
    for k in range(len(queues)):
        if queues[k] and (best is None or c[k] < c[best]):
            best = k
    return best


@pytest.mark.parametrize("K", [1, 2, 3])
def test_brute_force_all_short_event_orders(K):
    """Every order of <= 6 events over K <= 3 devices (omega 3, depth 2):
    served device equals a direct scan, sender flags follow Sec. 3.4.1."""
    omega, depth = 3, 2
    alphabet = [("step",)] + [("enq", k) for k in range(K)]
    for n in range(1, 7):
        for seq in itertools.product(alphabet, repeat=n):
            s = O.TaskScheduler(K, omega, depth)
            for ev in seq:
                if ev[0] == "enq":
                    k = ev[1]
                    total, qk = s.queued(), len(s.q[k])
                    st, _ = s.put(k)
                    if total >= omega or qk >= depth:
                        assert st == O.FULL and not s.on[k]
                    else:
                        assert st == O.OK
                        assert s.on[k] == (total + 1 < omega and qk + 1 < depth)
                else:
                    expect = literal_alg3(s.q, s.c)
                    st, k, _ = s.get()
                    if expect is None:
                        assert st == O.EMPTY
                    else:
                        assert k == expect and s.on[k]
                check_invariants(s, omega, depth)


def test_blocked_device_is_turned_on_by_next_dequeue():
    s = O.TaskScheduler(K=3, omega=2, depth=2)
    assert s.put(0)[0] == O.OK and s.put(0)[0] == O.OK     # cap reached by device 0
    assert s.put(1)[0] == O.FULL and not s.on[1]           # device 1 refused, empty queue
    assert list(s.blocked) == [1]
    s.get()
    assert s.on[0] and s.on[1] and not s.blocked
    assert s.put(1)[0] == O.OK


def test_fifo_policy_serves_in_arrival_order():
    s = O.TaskScheduler(K=3, omega=6, depth=3, policy="fifo")
    for k in [2, 2, 0, 1, 2]:
        s.put(k)
    assert [s.get()[1] for _ in range(5)] == [2, 2, 0, 1, 2]
    assert s.get()[0] == O.EMPTY


def test_leave_drains_queue_and_join_does_not_monopolise():
    s = O.TaskScheduler(K=3, omega=9, depth=3)
    for k in (0, 1, 2, 0, 1, 2):
        s.put(k)
    assert s.set_active(2, False) == O.OK
    assert s.put(2)[0] == O.ERR_ARG
    served = [s.get()[1] for _ in range(6)]
    assert sorted(served) == [0, 0, 1, 1, 2, 2]            # device 2's queue drains
    for _ in range(3):
        s.put(0), s.put(1), s.get(), s.get()
    assert s.c[2] < min(s.c[0], s.c[1])
    s.set_active(2, True)
    assert s.c[2] == min(s.c[0], s.c[1])


# --------------------------------------------------------------------------
# aggregation
# --------------------------------------------------------------------------

def test_fedasync_matches_hand_worked_golden():
    lines = golden_lines("fedasync_example.txt")
    g = np.array([float(v) for v in lines[0][1:]])
    agg = O.Aggregator(K=4, max_delay=1)
    assert int(lines[1][1]) == agg.t
    for f in lines[2:]:
        t_k = int(f[1])
        local = np.array([float(v) for v in f[2:5]])
        st, g = agg.aggregate(g, local, t_k)
        assert st == NAMES[f[6]]
        assert np.array_equal(g, np.array([float(v) for v in f[7:10]]))
        assert agg.t == int(f[10])


def test_running_mean_closed_form():
    """All locals trained from version 0 and D >= K: alpha = 1/(t+1), so the
    global after j aggregations is the mean of the first j locals, whatever
    the initial global."""
    r = np.random.default_rng(0)
    K, n = 4, 50
    locals_ = r.standard_normal((K, n)) * 0.05
    g = r.standard_normal(n)
    agg = O.Aggregator(K, max_delay=K)
    for j in range(K):
        st, g = agg.aggregate(g, locals_[j], 0)
        assert st == O.OK
        assert np.allclose(g, locals_[:j + 1].mean(0), rtol=1e-13, atol=1e-16)
    assert agg.round == 1


def test_identity_and_weights_sum_to_one():
    r = np.random.default_rng(1)
    g = r.standard_normal(10)
    agg = O.Aggregator(K=3, max_delay=100)
    for _ in range(5):
        agg.aggregate(g, g, 0)
    st, g2 = agg.aggregate(g, g, 2)
    assert st == O.OK and np.allclose(g2, g, rtol=1e-15)
    c = np.full(7, 3.25)
    st, c2 = agg.aggregate(c, c.copy(), agg.t - 1)
    assert np.allclose(c2, 3.25, rtol=1e-15)


def test_stale_and_invalid_versions():
    agg = O.Aggregator(K=2, max_delay=2)
    g = np.zeros(3)
    for _ in range(4):
        agg.aggregate(g, np.ones(3), agg.t)
    assert agg.t == 4
    st, g2 = agg.aggregate(g, np.ones(3) * 9, 1)          # t - t_k = 3 > D
    assert st == O.STALE and agg.t == 4 and np.array_equal(g2, g)
    assert agg.aggregate(g, g, 5)[0] == O.ERR_ARG          # version from the future
    assert agg.aggregate(g, g, -1)[0] == O.ERR_ARG
