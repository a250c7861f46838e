"""The library's scheduler checks have teeth: copies of the host Task
Scheduler header (paper_2504_13850_gb300/csrc/fo_sched.hpp) with one
plausible mistake each are compiled with g++ into a small host-only shim
(tests/native/sched_shim.cpp) and replayed against the same hand-derived
golden traces and oracle comparisons that check the library.  Every mutant
must fail at least one of them; the unmutated header must pass them all.
CPU only (no CUDA); the builds go to the package's git-ignored _build/."""
import ctypes as C
import os
import shutil
import subprocess

import numpy as np
import pytest

from oracle import fo_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "paper_2504_13850_gb300", "csrc", "fo_sched.hpp")
SHIM = os.path.join(ROOT, "tests", "native", "sched_shim.cpp")
OUT = os.path.join(ROOT, "paper_2504_13850_gb300", "_build", "sched_mutants")

pytestmark = pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")

MUTATIONS = {
    "argmin ties to the highest index": ("(k < 0 || c_[j] < c_[k])", "(k < 0 || c_[j] <= c_[k])"),
    "cap off by one": ("if (total_ >= omega_ || len_[k] >= depth_) {", "if (total_ > omega_ || len_[k] >= depth_) {"),
    "ring depth off by one": ("if (total_ >= omega_ || len_[k] >= depth_) {",
                              "if (total_ >= omega_ || len_[k] > depth_) {"),
    "freed slots reused last-in first-out": ("free_[(free_head_ + free_len_) % omega_] = s;",
                                             "free_head_ = (free_head_ + omega_ - 1) % omega_;\n"
                                             "    free_[free_head_] = s;"),
    "Sender left on at the cap": ("on_[k] = (total_ < omega_ && len_[k] < depth_) ? 1 : 0;",
                                  "on_[k] = (total_ <= omega_ && len_[k] < depth_) ? 1 : 0;"),
    "refused device with an empty queue never turned on": ("blocked_.push_back(k);", ";"),
    "rejoining device keeps its stale counter": ("if (any && c_[k] < lo) c_[k] = lo;", ";"),
    "FIFO policy serves newest first": ("k = arrivals_[arr_head_++];", "k = arrivals_.back();\n      arrivals_.pop_back();"),
    "counter of the wrong device incremented": ("++c_[k];", "++c_[0];"),
}


def build(name, source):
    d = os.path.join(OUT, name.replace(" ", "_"))
    os.makedirs(d, exist_ok=True)
    with open(os.path.join(d, "fo_sched.hpp"), "w") as f:
        f.write(source)
    so = os.path.join(d, "shim.so")
    r = subprocess.run(["g++", "-std=c++17", "-O1", "-shared", "-fPIC", "-I", d, SHIM, "-o", so],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    L = C.CDLL(so)
    L.shim_create.restype = C.c_void_p
    L.shim_create.argtypes = [C.c_int, C.c_int, C.c_int, C.c_int]
    L.shim_destroy.argtypes = [C.c_void_p]
    L.shim_put.argtypes = [C.c_void_p, C.c_int, C.POINTER(C.c_int32)]
    L.shim_get.argtypes = [C.c_void_p, C.POINTER(C.c_int), C.POINTER(C.c_int32)]
    L.shim_peek.argtypes = [C.c_void_p, C.c_int, C.POINTER(C.c_int32)]
    L.shim_set_active.argtypes = [C.c_void_p, C.c_int, C.c_int]
    L.shim_counters.argtypes = [C.c_void_p, C.c_void_p]
    L.shim_sender.argtypes = [C.c_void_p, C.c_void_p]
    L.shim_queued.argtypes = [C.c_void_p]
    return L


class Shim:
    """The fo_sched_* calls' return conventions over a shim build."""

    def __init__(self, L, K, omega, depth, policy="counter"):
        self.L, self.K = L, K
        self.h = L.shim_create(K, omega, depth, 0 if policy == "counter" else 1)

    def __del__(self):
        self.L.shim_destroy(self.h)

    def put(self, k):
        slot = C.c_int32(-1)
        rc = self.L.shim_put(self.h, k, C.byref(slot)) if 0 <= k < self.K else -1
        return rc, slot.value, (int(self.sender_status()[k]) if 0 <= k < self.K else -1)

    def peek(self, k):
        slot = C.c_int32(-1)
        rc = self.L.shim_peek(self.h, k, C.byref(slot))
        return rc, slot.value

    def get(self):
        k, slot = C.c_int(-1), C.c_int32(-1)
        rc = self.L.shim_get(self.h, C.byref(k), C.byref(slot))
        return (O.OK, k.value, slot.value) if rc == 0 else (O.EMPTY, -1, -1)

    def set_active(self, k, active):
        return O.OK if self.L.shim_set_active(self.h, k, int(active)) == 0 else O.ERR_ARG

    def counters(self):
        out = np.zeros(self.K, np.uint64)
        self.L.shim_counters(self.h, out.ctypes.data)
        return [int(v) for v in out]

    def sender_status(self):
        out = np.zeros(self.K, np.uint8)
        self.L.shim_sender(self.h, out.ctypes.data)
        return [int(v) for v in out]

    def queued(self):
        return self.L.shim_queued(self.h)


NAMES = {"OK": O.OK, "EMPTY": O.EMPTY, "FULL": O.FULL}


def golden(name):
    with open(os.path.join(ROOT, "tests", "golden", name)) as f:
        return [l.split() for l in f if l.strip() and not l.startswith("#")]


def check_tiny_golden(L):
    s = Shim(L, 4, 8, 2)
    for p in golden("sched_tiny_order.txt"):
        if p[0] == "enqueue":
            assert s.put(int(p[1])) == (NAMES[p[3]], int(p[4]), int(p[5])), p
        else:
            assert s.get() == (NAMES[p[2]], int(p[3]), int(p[4])), p
            assert s.counters() == [int(v) for v in p[5:9]], p


def check_slot_reuse_golden(L):
    from test_oracle_sched_agg import replay_slot_reuse_golden
    s = Shim(L, 3, 3, 2)
    replay_slot_reuse_golden(lambda k: s.put(k)[:2], s.get, s.counters, s.sender_status)


def check_random_traces(L):
    for policy in ("counter", "fifo"):
        for seed in range(6):
            r = np.random.default_rng(seed)
            K, depth = int(r.integers(1, 9)), int(r.integers(1, 5))
            omega = int(r.integers(1, K * depth + 3))
            a, o = Shim(L, K, omega, depth, policy), O.TaskScheduler(K, omega, depth, policy)
            for _ in range(400):
                u = r.random()
                if u < 0.45:
                    k = int(r.integers(K))
                    rc, slot, on = a.put(k)
                    assert (rc, slot) == o.put(k) and on == int(o.on[k])
                elif u < 0.9:
                    assert a.get() == o.get()
                else:
                    k, act = int(r.integers(K)), bool(r.integers(2))
                    assert a.set_active(k, act) == o.set_active(k, act)
                assert a.counters() == o.c and a.sender_status() == [int(v) for v in o.on]
                assert a.queued() == o.queued()


def check_peek_predicts_put(L):
    """An upload's slot is filled before the scheduler commits it: peek(k)
    must give put(k)'s outcome and slot exactly, and change nothing."""
    for policy in ("counter", "fifo"):
        for seed in range(4):
            r = np.random.default_rng(100 + seed)
            K, depth = int(r.integers(1, 7)), int(r.integers(1, 4))
            omega = int(r.integers(1, K * depth + 2))
            a = Shim(L, K, omega, depth, policy)
            for _ in range(300):
                u = r.random()
                if u < 0.5:
                    k = int(r.integers(K))
                    state = (a.counters(), a.sender_status(), a.queued())
                    prc, pslot = a.peek(k)
                    assert (a.counters(), a.sender_status(), a.queued()) == state
                    rc, slot, _ = a.put(k)
                    assert prc == {0: 0, 2: 2, -1: -1}.get(rc, rc)
                    if rc == 0:
                        assert slot == pslot
                elif u < 0.9:
                    a.get()
                else:
                    a.set_active(int(r.integers(K)), bool(r.integers(2)))


CHECKS = (check_tiny_golden, check_slot_reuse_golden, check_random_traces, check_peek_predicts_put)


def source():
    with open(HEADER) as f:
        return f.read()


def test_unmutated_header_passes_every_check():
    L = build("unmutated", source())
    for check in CHECKS:
        check(L)


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_planted_mistake_in_the_library_scheduler_is_caught(name):
    old, new = MUTATIONS[name]
    src = source()
    assert src.count(old) == 1, old
    L = build(name, src.replace(old, new))
    caught = []
    for check in CHECKS:
        try:
            check(L)
        except AssertionError:
            caught.append(check.__name__)
    assert caught, f"no check caught: {name}"
