"""Counter-based vs FIFO task scheduling (the paper's scheduler comparison,
Sec. 4): on the 100-device Zipf(1.2) trace the counter-based policy spreads
the server's iterations more evenly than FIFO, which follows the arrival
skew.  Host-only (fo_sched_*)."""
import numpy as np

from paper_2504_13850_gb300 import api, study
from paper_2504_13850_gb300 import workloads as W


def test_gini_of_known_distributions():
    assert study.gini([3, 3, 3, 3]) == 0.0
    assert study.gini([0, 0, 0, 8]) == 0.75          # (n - 1) / n for one non-zero value
    assert abs(study.gini([1, 2, 3, 4]) - 0.25) < 1e-12


def test_counter_policy_is_more_balanced_than_fifo():
    r = study.scheduler_balance("scale", uploads=6000)
    assert r["counter"]["gini"] < r["fifo"]["gini"]
    assert r["counter"]["max_share"] < r["fifo"]["max_share"]
    assert r["counter"]["max_minus_min_served"] < r["fifo"]["max_minus_min_served"]


def test_counter_policy_equalises_backlogged_devices():
    # every device uploads at the same rate and the server is the bottleneck:
    # all queues stay backlogged and the counters end within one of each other
    cfg = dict(W.CONFIGS["scale"], rates=[1.0] * 100)
    c = study.consumption(api.SCHED_COUNTER, cfg, 4000, seed=9)
    assert c.max() - c.min() <= 1
