"""The five bf16 workloads at their full sizes, in the launch configuration
the benchmark times (same server plan, tiles and cluster splits): scheduler
outcomes bit-exact, and two teacher-forced steps against the exact fp64
oracle: loss 1e-2, parameters 2e-2, and the update and the gradient of
every parameter tensor within the bound of harness.grad_bound."""
import pytest

from harness import check_teacher_forced, teacher_forced
from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def events(cfg, uploaders, steps):
    """A few devices upload one batch each (round robin), then steps."""
    return [("enq", k) for k in range(uploaders)] + [("step",)] * steps


@pytest.mark.parametrize("name", ["vgg", "resnet", "transformer", "scale", "mobilenet"])
def test_full_size_teacher_forced(name):
    cfg = W.CONFIGS[name]
    ev = events(cfg, min(cfg["K"], 3), 2)
    _, _, recs = teacher_forced(cfg, ev)
    assert len(recs) == 2
    check_teacher_forced(recs)
