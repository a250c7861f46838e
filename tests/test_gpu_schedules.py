"""The step graph's schedule does not change the arithmetic: with the weight
gradients on the side stream (default) or all kernels on one stream
(FO_NO_SIDE), the same trace gives bit-identical parameters, momentum and
losses (every reduction has a fixed order, and each stream lane has its own
split-K workspace)."""
import os

import numpy as np
import pytest

from harness import replay_gpu
from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def run(cfg, events, side):
    old = os.environ.pop("FO_NO_SIDE", None)
    try:
        if not side:
            os.environ["FO_NO_SIDE"] = "1"
        s, log = replay_gpu(cfg, events)
        n = sum(1 for e in log if e[0] == "step" and e[1] == api.OK)
        out = (s.get_params(), s.get_momentum(), s.read_losses(0, n), log)
        s.close()
        return out
    finally:
        os.environ.pop("FO_NO_SIDE", None)
        if old is not None:
            os.environ["FO_NO_SIDE"] = old


@pytest.mark.parametrize("name", ["vgg", "resnet", "transformer"])
def test_side_stream_is_bit_identical(name):
    cfg = W.CONFIGS[name]
    events = [("enq", k) for k in range(min(cfg["K"], 3))] + [("step",)] * 3
    a = run(cfg, events, side=True)
    b = run(cfg, events, side=False)
    assert a[3] == b[3]
    for x, y in zip(a[:3], b[:3]):
        assert np.array_equal(x, y)
