"""Pre-processor split selection (Sec. 3.2, Eqs. 4-6): the oracle pinned to a
hand-worked example and to limiting cases, and the C ABI (host-only)
checked against the oracle."""
import json
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.join(os.path.dirname(__file__), "..", "oracle"))
import fo_oracle as O  # noqa: E402

from paper_2504_13850_gb300 import api  # noqa: E402

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "split_selection.json")))


@pytest.mark.parametrize("case", GOLD["cases"], ids=lambda c: c["name"])
def test_hand_worked_example(case):
    l, cost = O.split_point(GOLD["O_flop"], GOLD["S_bytes"], case["b_Bps"], GOLD["o_flops"], case["allowed"])
    assert l == case["split"]
    assert cost == pytest.approx(case["cost_s"], rel=1e-12)
    rc, l2, c2 = api.select_split(GOLD["O_flop"], GOLD["S_bytes"], case["b_Bps"], GOLD["o_flops"], case["allowed"])
    assert rc == api.OK and l2 == case["split"] and c2 == pytest.approx(case["cost_s"], rel=1e-12)


def _instance(seed, L=12, K=6):
    rng = np.random.default_rng(seed)
    return (rng.uniform(1e8, 5e9, L), rng.uniform(1e5, 5e7, L), rng.uniform(1e7, 1e9, K),
            rng.uniform(1e10, 1e12, K))


def test_infinite_bandwidth_splits_after_the_first_candidate():
    # no transfer cost: the training time only grows with l
    Ol, Sl, b, o = _instance(1)
    allowed = np.zeros(len(Ol), np.uint8)
    allowed[[3, 5, 9]] = 1
    assert O.split_point(Ol, Sl, np.full_like(b, 1e300), o)[0] == 1
    assert O.split_point(Ol, Sl, np.full_like(b, 1e300), o, allowed)[0] == 4


def test_infinite_compute_splits_at_the_smallest_activation():
    Ol, Sl, b, o = _instance(2)
    l, cost = O.split_point(Ol, Sl, b, np.full_like(o, 1e300))
    assert l == int(np.argmin(Sl)) + 1
    assert cost == pytest.approx(Sl.min() / b.min(), rel=1e-12)


def test_slowest_device_decides():
    # adding a device that is faster everywhere changes nothing
    Ol, Sl, b, o = _instance(3)
    l0, c0 = O.split_point(Ol, Sl, b, o)
    l1, c1 = O.split_point(Ol, Sl, np.append(b, b.max() * 10), np.append(o, o.max() * 10))
    assert (l0, c0) == (l1, c1)


def test_scaling_all_rates_scales_the_cost_only():
    Ol, Sl, b, o = _instance(4)
    l0, c0 = O.split_point(Ol, Sl, b, o)
    l1, c1 = O.split_point(Ol, Sl, 4 * b, 4 * o)
    assert l1 == l0 and c1 == pytest.approx(c0 / 4, rel=1e-12)


@pytest.mark.parametrize("seed", range(20))
def test_abi_matches_oracle(seed):
    Ol, Sl, b, o = _instance(100 + seed)
    allowed = None if seed % 2 else (np.random.default_rng(seed).random(len(Ol)) < 0.5).astype(np.uint8)
    if allowed is not None and not allowed.any():
        allowed[-1] = 1
    l, cost = O.split_point(Ol, Sl, b, o, allowed)
    rc, l2, c2 = api.select_split(Ol, Sl, b, o, allowed)
    assert rc == api.OK and l2 == l and c2 == pytest.approx(cost, rel=1e-12)


def test_bad_arguments():
    ok = ([1.0, 2.0], [3.0, 1.0], [1.0], [1.0])
    assert api.select_split([], [], [1.0], [1.0])[0] == api.ERR_ARG
    assert api.select_split([1.0, -1.0], ok[1], ok[2], ok[3])[0] == api.ERR_ARG
    assert api.select_split(ok[0], ok[1], [0.0], ok[3])[0] == api.ERR_ARG
    assert api.select_split(ok[0], ok[1], ok[2], [-1.0])[0] == api.ERR_ARG
    assert api.select_split(*ok, allowed=[0, 0])[0] == api.ERR_ARG
    assert api.select_split(*ok)[0] == api.OK


def test_ties_go_to_the_smallest_split():
    """Every split point costs exactly the same (compute far faster than the
    link, every layer's output the same size): the reading takes the
    smallest l, or the smallest allowed one when a mask is given."""
    Oflop, S = [1.0, 1.0, 1.0, 1.0], [4096.0] * 4
    b, o = [1e6, 2e6], [1e30, 1e30]
    l, cost = O.split_point(Oflop, S, b, o)
    assert (l, cost) == (1, 4096.0 / 1e6)
    assert O.split_point(Oflop, S, b, o, [0, 0, 1, 1]) == (3, 4096.0 / 1e6)
    rc, l2, c2 = api.select_split(Oflop, S, b, o, None)
    assert (rc, l2, c2) == (api.OK, 1, 4096.0 / 1e6)
    rc, l2, c2 = api.select_split(Oflop, S, b, o, [0, 0, 1, 1])
    assert (rc, l2) == (api.OK, 3)
