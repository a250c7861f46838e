"""The bf16 parity gates have teeth: a training step with a planted mistake
fails harness.gate_failures against the exact fp64 oracle, while a correct
bf16-storage step passes.

Runs on the CPU.  The oracle's bf16-storage reading stands in for the GPU
path (it stores every tensor in bf16 the way the kernels do), and each
mistake is planted in that stand-in's output, the way a kernel bug would
show in the parameters and momentum read back from the GPU: a parameter
tensor whose gradient is lost, a gradient with the wrong sign, an update
that is skipped or applied at twice the learning rate, and momentum that is
dropped.  Both a network with ReLU / max-pool decisions and a
decision-free one are covered, on a first step (v0 = 0) and a second step
(v0 != 0).
"""
import numpy as np
import pytest

from harness import batch_for, gate_failures, param_slices, step_record
from oracle import fo_oracle as O
from paper_2504_13850_gb300 import workloads as W


def relu_pool_net():
    b = W._Builder()
    t = b.add("conv", 0, cin=16, cout=32, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("conv", t, cin=32, cout=32, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("flatten", t)
    t = b.add("linear", t, cin=2 * 2 * 32, cout=32, bias=1)
    t = b.add("relu", t)
    b.add("linear", t, cin=32, cout=10, bias=1)
    return W.shrink(W.CONFIGS["vgg"], ops=b.ops, batch=8, in_hwc=(8, 8, 16), K=2, omega=4, depth=2, lr=1e-3)


def decision_free_net():
    b = W._Builder()
    t = b.add("conv", 0, cin=16, cout=32, k=3, stride=1, bias=1)
    t = b.add("conv", t, cin=32, cout=32, k=3, stride=2, bias=1)
    t = b.add("flatten", t)
    t = b.add("linear", t, cin=4 * 4 * 32, cout=32, bias=1)
    b.add("linear", t, cin=32, cout=10, bias=1)
    return W.shrink(W.CONFIGS["vgg"], ops=b.ops, batch=8, in_hwc=(8, 8, 16), K=2, omega=4, depth=2, lr=1e-3)


def records(cfg, plant=None, steps=2):
    """Teacher-forced records of `steps` steps with the bf16-storage reading
    as the path under test; `plant(th0, v0, th1, v1, slices, lr, mu)`
    returns the path's (th1, v1) with a mistake in them."""
    ops, lr, mu = cfg["ops"], cfg["lr"], cfg["momentum"]
    slices = param_slices(ops)
    th = W.init_params(cfg).astype(np.float64)
    v = np.zeros_like(th)
    out = []
    for j in range(steps):
        x, _, y, ln = batch_for(cfg, j % cfg["K"], j)
        o = O.Server(ops, cfg["K"], cfg["omega"], cfg["depth"], th, lr, mu)
        ob = O.Server(ops, cfg["K"], cfg["omega"], cfg["depth"], th, lr, mu, storage="bf16")
        for srv in (o, ob):
            srv.theta, srv.v = th.copy(), v.copy()
            srv.enqueue(0, x, y, ln)
            srv.step()
        th1, v1 = ob.theta.copy(), ob.v.copy()
        if plant is not None:
            th1, v1 = plant(th, v, th1, v1, slices, lr, mu)
        out.append(step_record(j, ob.losses[-1], th, v, th1, v1, o, ob, mu, slices))
        th, v = th1, v1
    return out


def _tensor(slices, name):
    return dict(slices)[name]


def lose_gradient(name):
    def plant(th0, v0, th1, v1, slices, lr, mu):
        sl = _tensor(slices, name)
        v1, th1 = v1.copy(), th1.copy()
        v1[sl] = mu * v0[sl]
        th1[sl] = th0[sl] - lr * v1[sl]
        return th1, v1
    return plant


def flip_gradient(name):
    def plant(th0, v0, th1, v1, slices, lr, mu):
        sl = _tensor(slices, name)
        g = v1[sl] - mu * v0[sl]
        v1, th1 = v1.copy(), th1.copy()
        v1[sl] = mu * v0[sl] - g
        th1[sl] = th0[sl] - lr * v1[sl]
        return th1, v1
    return plant


def skip_update(th0, v0, th1, v1, slices, lr, mu):
    return th0.copy(), v1


def double_lr(th0, v0, th1, v1, slices, lr, mu):
    return th0 - 2 * lr * v1, v1


def drop_momentum(th0, v0, th1, v1, slices, lr, mu):
    g = v1 - mu * v0
    return th0 - lr * g, g


NETS = {"relu_pool": relu_pool_net, "decision_free": decision_free_net}


@pytest.mark.parametrize("net", sorted(NETS))
def test_correct_bf16_step_passes(net):
    for r in records(NETS[net]()):
        assert not gate_failures(r), gate_failures(r)


@pytest.mark.parametrize("net", sorted(NETS))
def test_every_lost_tensor_gradient_is_caught(net):
    cfg = NETS[net]()
    for name, _ in param_slices(cfg["ops"]):
        recs = records(cfg, lose_gradient(name), steps=1)
        bad = gate_failures(recs[0])
        assert any(b[0] == "grad " + name for b in bad), (name, bad)


@pytest.mark.parametrize("net", sorted(NETS))
def test_every_wrong_signed_tensor_gradient_is_caught(net):
    cfg = NETS[net]()
    for name, _ in param_slices(cfg["ops"]):
        bad = gate_failures(records(cfg, flip_gradient(name), steps=1)[0])
        assert any(b[0] == "grad " + name for b in bad), (name, bad)


@pytest.mark.parametrize("net", sorted(NETS))
@pytest.mark.parametrize("plant", [skip_update, double_lr])
def test_wrong_update_is_caught(net, plant):
    for r in records(NETS[net](), plant):
        assert any(b[0] == "update" for b in gate_failures(r)), gate_failures(r)


@pytest.mark.parametrize("net", sorted(NETS))
def test_dropped_momentum_is_caught_on_the_second_step(net):
    recs = records(NETS[net](), drop_momentum)
    assert not gate_failures(recs[0])          # v0 = 0: the same step
    assert gate_failures(recs[1])
