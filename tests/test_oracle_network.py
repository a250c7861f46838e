"""Pins for the oracle's whole server step (CPU only).

The network forward/backward is checked against an independent statement
of the same architecture in PyTorch fp64 autograd (a library cross-check:
PyTorch's conv/pool/norm/GELU/softmax kernels and its reverse-mode AD), and
by central finite differences of the oracle's own loss on tiny shapes.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import fo_oracle as O
from paper_2504_13850_gb300 import workloads as W


def torch_loss(ops, flat, x, labels, lengths):
    """Independent PyTorch statement of the op-list semantics."""
    p = torch.tensor(flat, dtype=torch.float64, requires_grad=True)
    views, off = {}, 0
    for i, name, shape in O.param_shapes(ops):
        n = int(np.prod(shape))
        views[(i, name)] = p[off:off + n].view(shape)
        off += n
    T = [torch.tensor(x, dtype=torch.float64)]
    ln = None if lengths is None else torch.tensor(lengths)
    for i, op in enumerate(ops):
        kd, a = op["kind"], T[op["in0"]]
        if kd == "conv":
            w = views[(i, "W")].permute(0, 3, 1, 2)
            b = views.get((i, "b"))
            y = F.conv2d(a.permute(0, 3, 1, 2), w, b, stride=op["stride"], padding=op["k"] // 2)
            y = y.permute(0, 2, 3, 1)
        elif kd == "affine":
            y = a * views[(i, "scale")] + views[(i, "shift")]
        elif kd == "relu":
            y = F.relu(a)
        elif kd == "maxpool2":
            y = F.max_pool2d(a.permute(0, 3, 1, 2), 2).permute(0, 2, 3, 1)
        elif kd == "add":
            y = a + T[op["in1"]]
        elif kd == "avgpool":
            y = a.mean(dim=(1, 2))
        elif kd == "flatten":
            y = a.reshape(a.shape[0], -1)
        elif kd == "linear":
            y = F.linear(a, views[(i, "W")], views.get((i, "b")))
        elif kd == "layernorm":
            y = F.layer_norm(a, (op["c"],), views[(i, "gamma")], views[(i, "beta")], eps=1e-5)
        elif kd == "gelu":
            y = F.gelu(a)
        elif kd == "attention":
            B, L, d, h = a.shape[0], a.shape[1], op["c"], op["heads"]
            t = a.reshape(B, L, 3 * d)
            q, k, v = [t[..., j * d:(j + 1) * d].reshape(B, L, h, d // h).transpose(1, 2) for j in range(3)]
            mask = torch.arange(L)[None, :] >= ln[:, None]
            att = F.scaled_dot_product_attention(q, k, v, attn_mask=~mask[:, None, None, :])
            y = att.transpose(1, 2).reshape(B, L, 1, d)
        elif kd == "meanpool":
            m = (torch.arange(a.shape[1])[None, :] < ln[:, None]).to(a.dtype)
            y = (a[:, :, 0, :] * m[..., None]).sum(1) / ln[:, None].to(a.dtype)
        elif kd == "dwconv":
            w = views[(i, "W")].unsqueeze(1)                  # [C, 1, k, k]: groups = C
            y = F.conv2d(a.permute(0, 3, 1, 2), w, views.get((i, "b")), stride=op["stride"],
                         padding=op["k"] // 2, groups=op["c"]).permute(0, 2, 3, 1)
        elif kd == "hswish":
            y = F.hardswish(a)
        elif kd == "hsigmoid":
            y = F.hardsigmoid(a)
        elif kd == "chmul":
            y = a * T[op["in1"]][:, None, None, :]
        else:
            raise ValueError(kd)
        T.append(y)
    loss = F.cross_entropy(T[-1], torch.tensor(labels, dtype=torch.long))
    loss.backward()
    return float(loss.detach()), p.grad.numpy()


def small_vgg():
    b = W._Builder()
    t = b.add("conv", 0, cin=4, cout=6, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("conv", t, cin=6, cout=6, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("conv", t, cin=6, cout=8, k=3, stride=1, bias=1)
    t = b.add("relu", t)
    t = b.add("maxpool2", t)
    t = b.add("flatten", t)
    t = b.add("linear", t, cin=8 * 2 * 2, cout=7, bias=1)
    t = b.add("relu", t)
    b.add("linear", t, cin=7, cout=5, bias=1)
    return b.ops


def small_resnet():
    b = W._Builder()
    t = W._basic_block(b, 0, 4, 6, 2)
    t = W._basic_block(b, t, 6, 6, 1)
    t = b.add("avgpool", t)
    b.add("linear", t, cin=6, cout=5, bias=1)
    return b.ops


def small_mobilenet():
    b = W._Builder()
    t = W._bneck(b, 0, 4, 12, 6, 3, 2)
    t = W._bneck(b, t, 6, 16, 6, 5, 1)
    t = b.add("avgpool", t)
    b.add("linear", t, cin=6, cout=5, bias=1)
    return b.ops


def small_transformer():
    return W.transformer_ops(d=8, heads=2, ffn=12, blocks=2, classes=2)


CASES = {
    "tiny_cnn": (W.tiny_cnn_ops(), (16, 16, 32), False, 10),
    "vgg": (small_vgg(), (8, 8, 4), False, 5),
    "resnet": (small_resnet(), (8, 8, 4), False, 5),
    "mobilenet": (small_mobilenet(), (8, 8, 4), False, 5),
    "transformer": (small_transformer(), (6, 1, 8), True, 2),
}


def make_case(name, B=3, seed=0):
    ops, hwc, seq, classes = CASES[name]
    cfg = {"ops": ops, "seed": seed, "batch": B, "in_hwc": hwc, "seq": seq,
           "classes": classes, "dtype": W.F32}
    theta = W.init_params(cfg).astype(np.float64)
    r = np.random.default_rng(seed + 100)
    theta += 0.05 * r.standard_normal(theta.shape)      # non-trivial biases/affines
    x, _, labels, lengths = W.device_batch(cfg, 0, 0)
    if seq:
        lengths = np.array([2, 6, 4])[:B]
    else:
        x = x + 0.1 * r.standard_normal(x.shape)       # move off ReLU kinks of the input
    return ops, theta, x, labels, lengths


@pytest.mark.parametrize("name", list(CASES))
def test_network_matches_torch_autograd(name):
    ops, theta, x, labels, lengths = make_case(name)
    loss, g = O.loss_and_grad(ops, theta, x, labels, lengths)
    tl, tg = torch_loss(ops, theta, x, labels, lengths)
    assert abs(loss - tl) <= 1e-12 * abs(tl)
    # the first layer's input gradient is not part of g; every param grad is.
    # PyTorch's hard-sigmoid backward scales by a single-precision 1/6 even in
    # float64 (a 3e-8 relative error), so the MobileNet case agrees to ~1e-9;
    # the finite-difference test below pins it independently.
    tol = 1e-7 if name == "mobilenet" else 1e-10
    assert np.linalg.norm(g - tg) <= tol * np.linalg.norm(tg)


@pytest.mark.parametrize("name", ["vgg", "resnet", "transformer", "mobilenet"])
def test_network_finite_differences(name):
    ops, theta, x, labels, lengths = make_case(name, seed=1)
    _, g = O.loss_and_grad(ops, theta, x, labels, lengths)
    r = np.random.default_rng(5)
    idx = r.choice(theta.size, size=40, replace=False)
    h = 1e-6
    num = []
    for i in idx:
        tp, tm = theta.copy(), theta.copy()
        tp[i] += h
        tm[i] -= h
        num.append((O.loss_and_grad(ops, tp, x, labels, lengths)[0]
                    - O.loss_and_grad(ops, tm, x, labels, lengths)[0]) / (2 * h))
    num = np.array(num)
    assert np.linalg.norm(g[idx] - num) <= 1e-6 * np.linalg.norm(num)


def test_server_step_is_sgd_momentum_of_the_gradient():
    ops, theta, x, labels, lengths = make_case("vgg")
    v0 = np.random.default_rng(3).standard_normal(theta.shape)
    loss, th1, v1, g = O.server_step(ops, theta, v0, x, labels, lengths, 0.01, 0.9)
    assert np.allclose(v1, 0.9 * v0 + g, rtol=1e-15)
    assert np.allclose(th1, theta - 0.01 * v1, rtol=1e-15)


def test_param_layout_matches_workload_counts():
    for name, cfg in W.CONFIGS.items():
        n = sum(int(np.prod(s)) for _, _, s in O.param_shapes(cfg["ops"]))
        assert n == W.num_params(cfg["ops"])
    assert W.num_params(W.CONFIGS["vgg"]["ops"]) == 8_625_162
    assert W.num_params(W.CONFIGS["resnet"]["ops"]) == 10_544_740
    assert W.num_params(W.CONFIGS["transformer"]["ops"]) == 12_611_586
    assert W.num_params(W.CONFIGS["tiny"]["ops"]) == 59_466


def test_flat_layout_is_the_documented_order():
    """The flat parameter order the C header documents, written out by hand
    for one op of every parameterised kind: conv W[cout][k][k][cin] then b;
    affine scale then shift; depthwise W[c][k][k] then b; layernorm gamma
    then beta; linear W[cout][cin] then b; ops without a bias have none."""
    ops = [{"kind": "conv", "in0": 0, "cin": 2, "cout": 3, "k": 3, "stride": 1, "bias": 1},
           {"kind": "affine", "in0": 1, "c": 3},
           {"kind": "dwconv", "in0": 2, "c": 3, "k": 5, "stride": 1, "bias": 1},
           {"kind": "conv", "in0": 3, "cin": 3, "cout": 4, "k": 1, "stride": 1, "bias": 0},
           {"kind": "relu", "in0": 4},
           {"kind": "layernorm", "in0": 5, "c": 4},
           {"kind": "flatten", "in0": 6},
           {"kind": "linear", "in0": 7, "cin": 4, "cout": 2, "bias": 1}]
    assert O.param_shapes(ops) == [
        (0, "W", (3, 3, 3, 2)), (0, "b", (3,)),
        (1, "scale", (3,)), (1, "shift", (3,)),
        (2, "W", (3, 5, 5)), (2, "b", (3,)),
        (3, "W", (4, 1, 1, 3)),
        (5, "gamma", (4,)), (5, "beta", (4,)),
        (7, "W", (2, 4)), (7, "b", (2,))]
    flat = np.arange(54 + 3 + 6 + 75 + 3 + 12 + 8 + 8 + 2, dtype=np.float64)
    p = O.unflatten(ops, flat)
    assert p[(0, "b")].tolist() == [54.0, 55.0, 56.0]
    assert p[(0, "W")][1, 0, 2, 1] == 1 * 18 + 0 * 6 + 2 * 2 + 1
    assert np.array_equal(O.flatten(ops, p), flat)


def test_server_trains_on_the_batch_the_scheduler_served():
    """The event-replay server trains each step on the oldest queued batch
    of the device the scheduler picked (FIFO within a device), from the
    parameters the previous step left."""
    ops = small_vgg()
    r = np.random.default_rng(11)
    theta0 = O.flatten(ops, {k: 0.3 * r.standard_normal(s) for k, s in
                             (((i, n), s) for i, n, s in O.param_shapes(ops))})
    K, lr, mu = 3, 0.01, 0.9
    srv = O.Server(ops, K, omega=5, depth=2, theta0=theta0, lr=lr, mu=mu)
    sent = {k: [] for k in range(K)}

    def upload(k):
        x = np.maximum(r.standard_normal((2, 8, 8, 4)), 0.0)
        y = r.integers(0, 5, 2)
        st, _ = srv.enqueue(k, x, y)
        if st == O.OK:
            sent[k].append((x, y))

    for k in (0, 1, 0, 2, 1):
        upload(k)
    theta, v = theta0.copy(), np.zeros_like(theta0)
    for step in range(8):
        if step == 3:
            upload(2)
            upload(0)
        st, k, _ = srv.step()
        if st != O.OK:
            break
        x, y = sent[k].pop(0)
        loss, theta, v, _ = O.server_step(ops, theta, v, x, y, None, lr, mu)
        assert srv.losses[-1] == loss
        assert np.array_equal(srv.theta, theta) and np.array_equal(srv.v, v)
    assert all(not q for q in sent.values())
