"""The library's host Task Scheduler (Algorithms 2-3, flow control of Sec.
3.4.1, join / leave) against the oracle's under arbitrary interleavings of
uploads, server steps and devices leaving or rejoining, explored by
hypothesis' stateful testing: every return value, slot index, counter,
Sender Status and queue length must agree after every event."""
import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import settings, strategies as st  # noqa: E402
from hypothesis.stateful import RuleBasedStateMachine, initialize, invariant, rule  # noqa: E402

from oracle import fo_oracle as O  # noqa: E402
from paper_2504_13850_gb300 import api, build  # noqa: E402

build.build()


class SchedulerAgreement(RuleBasedStateMachine):
    @initialize(K=st.integers(1, 6), omega=st.integers(1, 10), depth=st.integers(1, 4),
                fifo=st.booleans())
    def setup(self, K, omega, depth, fifo):
        self.K = K
        self.lib = api.Scheduler(K, omega, depth, api.SCHED_FIFO if fifo else api.SCHED_COUNTER)
        self.ref = O.TaskScheduler(K, omega, depth, "fifo" if fifo else "counter")

    @rule(k=st.integers(0, 5))
    def upload(self, k):
        k %= self.K
        rc, slot, on = self.lib.put(k)
        orc, oslot = self.ref.put(k)
        assert (rc, slot) == (orc, oslot)
        assert on == int(self.ref.on[k])

    @rule()
    def step(self):
        assert self.lib.get() == self.ref.get()

    @rule(k=st.integers(0, 5), active=st.booleans())
    def join_or_leave(self, k, active):
        k %= self.K
        assert self.lib.set_active(k, active) == self.ref.set_active(k, active)

    @invariant()
    def same_state(self):
        if not hasattr(self, "ref"):
            return
        assert self.lib.counters() == self.ref.c
        assert self.lib.sender_status() == [int(v) for v in self.ref.on]
        assert self.lib.queued() == self.ref.queued()


SchedulerAgreement.TestCase.settings = settings(max_examples=150, stateful_step_count=60, deadline=None)
test_scheduler_agrees_with_oracle_under_any_interleaving = SchedulerAgreement.TestCase
