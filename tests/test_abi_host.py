"""The C-ABI library on the CPU: it loads without a GPU, exports every entry
point include/fedoptima.h declares, and its host-side Task Scheduler
(Algorithms 2-3 with the flow control of Sec. 3.4.1) agrees bit for bit with
the oracle's on hand-derived and random traces."""
import os
import re

import numpy as np
import pytest

from oracle import fo_oracle as O
from paper_2504_13850_gb300 import api, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_library():
    build.build()
    yield


def declared_symbols():
    with open(os.path.join(ROOT, "include", "fedoptima.h")) as f:
        text = f.read()
    return sorted(set(re.findall(r"FO_API\s+[\w\s\*]+?\b(fo_\w+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    import ctypes
    L = ctypes.CDLL(api.LIB_PATH)
    names = declared_symbols()
    assert len(names) >= 25
    for n in names:
        assert hasattr(L, n), n
    assert sorted(names) == sorted(api.exported_symbols())


def test_scheduler_matches_golden_trace():
    s = api.Scheduler(4, 8, 2)
    names = {"OK": api.OK, "EMPTY": api.EMPTY, "FULL": api.FULL}
    with open(os.path.join(ROOT, "tests", "golden", "sched_tiny_order.txt")) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            p = line.split()
            if p[0] == "enqueue":
                rc, slot, on = s.put(int(p[1]))
                assert (rc, slot, on) == (names[p[3]], int(p[4]), int(p[5]))
            else:
                rc, k, slot = s.get()
                assert (rc, k, slot) == (names[p[2]], int(p[3]), int(p[4]))
                assert s.counters() == [int(v) for v in p[5:9]]


def test_scheduler_matches_slot_reuse_golden():
    from test_oracle_sched_agg import replay_slot_reuse_golden
    s = api.Scheduler(3, 3, 2)
    replay_slot_reuse_golden(lambda k: s.put(k)[:2], s.get, s.counters, s.sender_status)


@pytest.mark.parametrize("policy", ["counter", "fifo"])
@pytest.mark.parametrize("seed", range(12))
def test_scheduler_matches_oracle_on_random_traces(seed, policy):
    r = np.random.default_rng(seed)
    K = int(r.integers(1, 9))
    depth = int(r.integers(1, 5))
    omega = int(r.integers(1, K * depth + 3))
    pol = api.SCHED_COUNTER if policy == "counter" else api.SCHED_FIFO
    a = api.Scheduler(K, omega, depth, pol)
    o = O.TaskScheduler(K, omega, depth, policy)
    for _ in range(600):
        u = r.random()
        if u < 0.45:
            k = int(r.integers(K))
            rc, slot, on = a.put(k)
            orc, oslot = o.put(k)
            assert (rc, slot, on) == (orc, oslot, int(o.on[k]))
        elif u < 0.9:
            rc, k, slot = a.get()
            orc, ok, oslot = o.get()
            assert (rc, k, slot) == (orc, ok, oslot)
        else:
            k = int(r.integers(K))
            act = bool(r.integers(2))
            assert a.set_active(k, act) == o.set_active(k, act)
        assert a.counters() == o.c
        assert a.sender_status() == [int(v) for v in o.on]
        assert a.queued() == o.queued()


def test_scheduler_rejects_bad_arguments():
    s = api.Scheduler(3, 4, 2)
    assert s.put(3)[0] == api.ERR_ARG
    assert s.put(-1)[0] == api.ERR_ARG
    assert s.get()[0] == api.EMPTY
    assert s.set_active(7, 1) == api.ERR_ARG


def test_scheduler_matches_oracle_on_zipf_trace_of_100_devices():
    """The 100-device workload: Zipf(1.2) Poisson arrivals, depth 4,
    omega = 400.  Bit-exact against the oracle; the counter-based policy
    keeps the consumption counts of the backlogged devices within one of
    each other, while FIFO follows the arrival skew."""
    from paper_2504_13850_gb300 import workloads as W
    cfg = W.CONFIGS["scale"]
    K, omega, depth = cfg["K"], cfg["omega"], cfg["depth"]
    a = api.Scheduler(K, omega, depth)
    o = O.TaskScheduler(K, omega, depth)
    f = O.TaskScheduler(K, omega, depth, "fifo")
    order = W.arrival_order(cfg["rates"], 6000, cfg["seed"])
    for i, k in enumerate(order):
        assert a.put(k)[:2] == o.put(k)
        f.put(k)
        if i % 2 == 1:            # the server consumes one batch per two uploads
            assert a.get() == o.get()
            f.get()
    assert a.counters() == o.c
    served = [c for c in o.c if c > 0]
    fifo_served = [c for c in f.c if c > 0]
    assert max(o.c) - min(served) <= max(fifo_served) - min(fifo_served)


def test_scheduler_size_limits_and_depth_above_omega():
    """K and omega beyond FO_MAX_DEVICES / FO_MAX_OMEGA are refused before
    anything is allocated; a ring depth far above omega never binds (the
    global cap is met first), so the trace equals the oracle's with that
    depth, without rings of that depth being allocated."""
    import ctypes
    L = api.lib()
    h = ctypes.c_void_p()
    assert L.fo_sched_create((1 << 20) + 1, 4, 2, api.SCHED_COUNTER, ctypes.byref(h)) == api.ERR_ARG
    assert L.fo_sched_create(4, (1 << 24) + 1, 2, api.SCHED_COUNTER, ctypes.byref(h)) == api.ERR_ARG
    assert L.fo_sched_create(4, 4, 0, api.SCHED_COUNTER, ctypes.byref(h)) == api.ERR_ARG
    r = np.random.default_rng(7)
    K, omega, depth = 5, 7, 1 << 30
    a = api.Scheduler(K, omega, depth)
    o = O.TaskScheduler(K, omega, depth)
    for _ in range(400):
        if r.random() < 0.55:
            k = int(r.integers(K))
            rc, slot, on = a.put(k)
            assert (rc, slot, on) == (*o.put(k), int(o.on[k]))
        else:
            assert a.get() == o.get()
        assert a.counters() == o.c


def test_every_entry_point_cites_its_passage_or_says_it_has_none():
    """Each FO_API declaration follows a comment block that cites the
    paper's section, algorithm, equation or table defining the operation,
    or states that the paper has no counterpart."""
    with open(os.path.join(ROOT, "include", "fedoptima.h")) as f:
        lines = f.read().split("\n")
    blocks, cur = [], None
    for i, line in enumerate(lines):
        if "/*" in line:
            cur = [line]
        elif cur is not None:
            cur.append(line)
        if cur is not None and "*/" in line:
            blocks.append((i, "\n".join(cur)))
            cur = None
    cite = re.compile(r"Sec\.|Alg|Eqs?\.|Table|no\s+(\*\s+)?counterpart|paper has no")
    missing = []
    for i, line in enumerate(lines):
        if line.startswith("FO_API"):
            before = [b for b in blocks if b[0] < i]
            if not before or not cite.search(before[-1][1]):
                missing.append(re.search(r"(fo_\w+)\s*\(", line).group(1))
    assert not missing, missing


def test_missing_library_fails_loudly(monkeypatch):
    """Without the built library every entry point raises: there is no
    fallback path (CPU or otherwise) behind the binding."""
    monkeypatch.setattr(api, "_lib", None)
    monkeypatch.setattr(api, "LIB_PATH", os.path.join(ROOT, "_no_such_dir", "libfedoptima.so"))
    with pytest.raises(api.FedOptimaError, match="missing"):
        api.lib()
    with pytest.raises(api.FedOptimaError):
        api.Scheduler(2, 2, 1)
    from paper_2504_13850_gb300 import workloads as W
    with pytest.raises(api.FedOptimaError):
        api.Server.from_config(W.CONFIGS["tiny"])
