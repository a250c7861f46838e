"""Server training steps on the GPU against the oracle on the same seeded
traces: scheduler outcomes and slot indices bit-exact, per-step loss within
1e-2 relative, parameters within 2e-2 normwise relative on the bf16 path and
1e-4 on the fp32 path (the tolerances of the method's statement of the
problem), and the parameter update theta_new - theta_old within a tolerance
derived below.

Update tolerance (fp32 path).  Each gradient is formed from a chain of a
few fp32 roundings (2^-24) over sums of <= 4096 terms, < 1e-5 normwise;
1e-4 is used.  The bf16 path is checked step by step (teacher forced)
against the exact oracle: loss, parameters, the gradient of every
parameter tensor and the update, with the bound derived in
harness.grad_bound.
"""
import numpy as np
import pytest

from harness import check_teacher_forced, normwise, replay_gpu, replay_oracle, teacher_forced
from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def small(kind):
    """Shrunk bf16 configurations of each architecture family that still span
    several tensor-core tiles and a ragged tail."""
    if kind == "vgg":
        b = W._Builder()
        t = b.add("conv", 0, cin=64, cout=128, k=3, stride=1, bias=1)
        t = b.add("relu", t)
        t = b.add("conv", t, cin=128, cout=128, k=3, stride=1, bias=1)
        t = b.add("relu", t)
        t = b.add("maxpool2", t)
        t = b.add("conv", t, cin=128, cout=256, k=3, stride=1, bias=1)
        t = b.add("relu", t)
        t = b.add("maxpool2", t)
        t = b.add("flatten", t)
        t = b.add("linear", t, cin=256 * 4 * 4, cout=128, bias=1)
        t = b.add("relu", t)
        b.add("linear", t, cin=128, cout=10, bias=1)
        return W.shrink(W.CONFIGS["vgg"], ops=b.ops, batch=12, in_hwc=(16, 16, 64), K=3,
                        omega=6, depth=2)
    if kind == "resnet":
        b = W._Builder()
        t = W._basic_block(b, 0, 64, 128, 2)
        t = W._basic_block(b, t, 128, 128, 1)
        t = b.add("avgpool", t)
        b.add("linear", t, cin=128, cout=100, bias=1)
        return W.shrink(W.CONFIGS["resnet"], ops=b.ops, batch=10, in_hwc=(16, 16, 64), K=3,
                        omega=6, depth=2)
    if kind == "transformer":
        return W.shrink(W.CONFIGS["transformer"],
                        ops=W.transformer_ops(d=128, heads=2, ffn=256, blocks=2),
                        batch=6, in_hwc=(128, 1, 128), K=3, omega=6, depth=2)
    raise ValueError(kind)


def prefill_then_steps(cfg, steps):
    ev = [("enq", k) for _ in range(cfg["depth"]) for k in range(cfg["K"])]
    return ev + [("step",)] * steps


def compare(cfg, events, loss_tol, param_tol, upd_tol=None, theta0=None):
    s, glog = replay_gpu(cfg, events, theta0)
    o, olog = replay_oracle(cfg, events, theta0)
    assert glog == olog                           # scheduler outcomes, slots: bit-exact
    nsteps = sum(1 for e in glog if e[0] == "step" and e[1] == api.OK)
    losses = s.read_losses(0, nsteps)
    ol = np.array(o.losses)
    assert np.all(np.abs(losses - ol) <= loss_tol * np.abs(ol)), (losses, ol)
    theta = s.get_params()
    theta0 = (W.init_params(cfg) if theta0 is None else theta0).astype(np.float64)
    assert normwise(theta, o.theta) <= param_tol
    if upd_tol is not None:
        assert normwise(theta - theta0, o.theta - theta0) <= upd_tol
        assert normwise(s.get_momentum(), o.v) <= upd_tol
    return s, o


def test_tiny_config_fp32_full_trace():
    cfg = W.CONFIGS["tiny"]
    events = prefill_then_steps(cfg, 9)           # 8 steps + one on empty queues
    s, o = compare(cfg, events, loss_tol=1e-4, param_tol=1e-4, upd_tol=1e-4)
    assert [int(c) for c in s.counters()] == o.sched.c == [2, 2, 2, 2]


@pytest.mark.parametrize("kind", ["vgg", "resnet", "transformer"])
def test_small_bf16_configs_teacher_forced(kind):
    """Every step from the GPU's own state: loss, parameters, update and the
    gradient of every parameter tensor against one exact oracle step.  At
    lr 1e-3 the loss stays near ln C over the six steps (at lr 0.01 the
    small VGG-style network reaches a loss of 11 by its fourth step, where
    the softmax is saturated and the gradient ill-conditioned)."""
    cfg = W.shrink(small(kind), lr=1e-3)
    _, _, recs = teacher_forced(cfg, prefill_then_steps(cfg, 6))
    assert len(recs) == 6
    check_teacher_forced(recs)


def decision_free(kind):
    """Conv / linear stacks without ReLU or max-pool: the tensor-core
    forward, input-gradient and weight-gradient kernels (tile widths 64-256,
    K split over clusters) checked without decision flips."""
    b = W._Builder()
    if kind == "conv16":
        t = b.add("conv", 0, cin=64, cout=128, k=3, stride=1, bias=1)
        t = b.add("conv", t, cin=128, cout=128, k=3, stride=1, bias=1)
        t = b.add("flatten", t)
        t = b.add("linear", t, cin=16 * 16 * 128, cout=128, bias=1)
        b.add("linear", t, cin=128, cout=10, bias=1)
        return W.shrink(W.CONFIGS["vgg"], ops=b.ops, batch=12, in_hwc=(16, 16, 64), K=3, omega=6, depth=2,
                        lr=1e-3)
    if kind == "conv8":
        t = b.add("conv", 0, cin=128, cout=256, k=3, stride=1, bias=1)
        t = b.add("conv", t, cin=256, cout=512, k=3, stride=1, bias=1)
        t = b.add("conv", t, cin=512, cout=256, k=3, stride=1, bias=1)
        t = b.add("flatten", t)
        t = b.add("linear", t, cin=8 * 8 * 256, cout=256, bias=1)
        b.add("linear", t, cin=256, cout=10, bias=1)
        return W.shrink(W.CONFIGS["vgg"], ops=b.ops, batch=20, in_hwc=(8, 8, 128), K=3, omega=6, depth=2,
                        lr=1e-3)
    if kind == "strided":
        t = b.add("conv", 0, cin=64, cout=128, k=3, stride=2, bias=1)      # 16x16 -> 8x8
        t = b.add("conv", t, cin=128, cout=128, k=1, stride=1, bias=1)
        t = b.add("conv", t, cin=128, cout=256, k=3, stride=2, bias=1)     # 8x8 -> 4x4
        t = b.add("flatten", t)
        t = b.add("linear", t, cin=4 * 4 * 256, cout=128, bias=1)
        b.add("linear", t, cin=128, cout=10, bias=1)
        return W.shrink(W.CONFIGS["resnet"], ops=b.ops, batch=16, in_hwc=(16, 16, 64), K=3, omega=6, depth=2,
                        lr=1e-3, classes=10)
    if kind == "resblock":
        t1 = b.add("conv", 0, cin=64, cout=64, k=3, stride=1, bias=0)
        t2 = b.add("conv", t1, cin=64, cout=128, k=3, stride=2, bias=0)
        t3 = b.add("affine", t2, c=128)
        t4 = b.add("conv", t1, cin=64, cout=128, k=1, stride=2, bias=0)    # first into t1's gradient
        t5 = b.add("add", t3, in1=t4)
        t6 = b.add("conv", t5, cin=128, cout=128, k=3, stride=1, bias=0)
        t = b.add("flatten", t6)
        t = b.add("linear", t, cin=8 * 8 * 128, cout=64, bias=1)
        b.add("linear", t, cin=64, cout=10, bias=1)
        return W.shrink(W.CONFIGS["resnet"], ops=b.ops, batch=8, in_hwc=(16, 16, 64), K=3, omega=6, depth=2,
                        lr=1e-3, classes=10)
    raise ValueError(kind)


@pytest.mark.parametrize("kind", ["conv16", "conv8", "strided", "resblock"])
def test_decision_free_teacher_forced(kind):
    cfg = decision_free(kind)
    _, _, recs = teacher_forced(cfg, prefill_then_steps(cfg, 4))
    assert len(recs) == 4
    check_teacher_forced(recs)
    for r in recs:   # no decisions: every tensor within the stated 2e-2 itself
        assert max(r["exact"]["tensor_grad_err"].values()) <= 2e-2, r["exact"]["tensor_grad_err"]


@pytest.mark.parametrize("kind", ["vgg", "resnet", "transformer"])
def test_small_bf16_configs_free_running(kind):
    """Two free-running steps from the same initial weights against the exact
    oracle at the stated tolerances (loss 1e-2, parameters 2e-2).  The small
    configurations train with a loss that grows (lr 0.01, momentum 0.9 on
    random labels), so two trajectories that differ by bf16 rounding
    separate by more than 1e-2 after a few steps; the per-step tolerance is
    gated step by step from a shared state in the teacher-forced test."""
    cfg = small(kind)
    compare(cfg, prefill_then_steps(cfg, 2), loss_tol=1e-2, param_tol=2e-2)


def test_arrival_trace_with_refusals_matches_oracle():
    """A Poisson arrival trace over devices of four speed groups, with the
    global cap reached: refusals, sender flags and served order bit-exact."""
    cfg = W.shrink(W.CONFIGS["tiny"], K=6, omega=5, depth=2,
                   rates=W.group_rates(6))
    ev = W.trace(cfg, n_steps=12, uploads_per_step=2, prefill=False)
    compare(cfg, ev, loss_tol=1e-4, param_tol=1e-4, upd_tol=1e-4)


def test_activation_memory_is_independent_of_devices():
    """Eq. 3: server activation memory is omega batches, whatever K is."""
    cfg = W.CONFIGS["tiny"]
    a = api.Server.from_config(cfg, K=4, omega=8)
    b = api.Server.from_config(cfg, K=100, omega=8)
    assert a.activation_bytes() == b.activation_bytes()
    B, (H, Wd, Ci) = cfg["batch"], cfg["in_hwc"]
    assert a.activation_bytes() >= 8 * B * H * Wd * Ci * 4


def test_empty_and_bad_calls():
    cfg = W.CONFIGS["tiny"]
    s = api.Server.from_config(cfg)
    assert s.server_step()[0] == api.EMPTY
    x, _, labels, _ = W.device_batch(cfg, 0, 0)
    assert s.enqueue_activations(7, x, labels)[0] == api.ERR_ARG
    s.set_device_active(2, False)
    assert s.enqueue_activations(2, x, labels)[0] == api.ERR_ARG


@pytest.mark.parametrize("name", ["tiny", "vgg"])
def test_uploads_into_slots_still_being_read(name):
    """Backlogged queues: after every step the next upload goes into the slot
    that step has just freed while its kernels may still be running, so the
    upload is staged on the device and moved in after the step.  Outcomes
    bit-exact, losses and parameters at the path's tolerances."""
    cfg = W.CONFIGS[name]
    if name == "vgg":
        cfg = W.shrink(cfg, K=3, omega=3, depth=1)
    ev = [("enq", k) for k in range(cfg["K"])]
    for j in range(8):
        ev += [("step",), ("enq", j % cfg["K"])]
    if cfg["dtype"] == W.F32:
        s, _ = compare(cfg, ev, loss_tol=1e-4, param_tol=1e-4, upd_tol=1e-4)
        assert s.read_losses(0, 8).shape == (8,)
    else:
        _, _, recs = teacher_forced(cfg, ev)
        assert len(recs) == 8
        check_teacher_forced(recs)
