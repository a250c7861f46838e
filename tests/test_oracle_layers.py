"""Pins for the oracle's layer arithmetic (CPU only).

Each layer of the oracle is checked against something other than itself:
brute-force loops written from the textbook definition, central finite
differences of its own forward pass (pins every backward), closed forms
and invariants, and an independent PyTorch fp64 autograd statement of the
whole network.
"""
import itertools
import math

import numpy as np
import pytest

from oracle import fo_oracle as O
from paper_2504_13850_gb300 import workloads as W


def rng(seed=0):
    return np.random.default_rng(seed)


def fd_grad(f, x, h=1e-6, idx=None):
    """Central finite differences of scalar f at x (all or selected entries)."""
    x = np.array(x, np.float64)
    flat = x.reshape(-1)
    idx = range(flat.size) if idx is None else idx
    out = {}
    for i in idx:
        old = flat[i]
        flat[i] = old + h
        fp = f(x)
        flat[i] = old - h
        fm = f(x)
        flat[i] = old
        out[i] = (fp - fm) / (2 * h)
    return out


def assert_fd(f, x, analytic, rel=1e-6, n=40, seed=0):
    analytic = np.asarray(analytic).reshape(-1)
    idx = rng(seed).choice(analytic.size, size=min(n, analytic.size), replace=False)
    num = fd_grad(f, x, idx=idx)
    a = np.array([analytic[i] for i in idx])
    b = np.array([num[i] for i in idx])
    err = np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-12)
    assert err < rel, (err, a[:5], b[:5])


# --------------------------------------------------------------------------
# convolution
# --------------------------------------------------------------------------

def brute_conv(x, w, b, stride, pad):
    """Direct loops over every output element and tap, with explicit bounds
    checks standing in for zero padding."""
    N, H, Wd, C = x.shape
    O_, k, _, _ = w.shape
    Ho = (H + 2 * pad - k) // stride + 1
    Wo = (Wd + 2 * pad - k) // stride + 1
    y = np.zeros((N, Ho, Wo, O_))
    for n, i, j, o in itertools.product(range(N), range(Ho), range(Wo), range(O_)):
        acc = 0.0 if b is None else b[o]
        for r, s, c in itertools.product(range(k), range(k), range(C)):
            hh, ww = i * stride + r - pad, j * stride + s - pad
            if 0 <= hh < H and 0 <= ww < Wd:
                acc += x[n, hh, ww, c] * w[o, r, s, c]
        y[n, i, j, o] = acc
    return y


@pytest.mark.parametrize("k,stride", [(3, 1), (3, 2), (1, 1), (1, 2)])
def test_conv_fwd_matches_brute_force(k, stride):
    r = rng(1)
    x = r.standard_normal((2, 6, 6, 3))
    w = r.standard_normal((4, k, k, 3))
    b = r.standard_normal(4)
    y = O.conv_fwd(x, w, b, stride, k // 2)
    assert np.allclose(y, brute_conv(x, w, b, stride, k // 2), rtol=1e-12, atol=1e-12)


def test_conv_single_channel_is_scipy_correlate():
    scipy_signal = pytest.importorskip("scipy.signal")
    r = rng(2)
    x = r.standard_normal((1, 7, 5, 1))
    w = r.standard_normal((1, 3, 3, 1))
    y = O.conv_fwd(x, w, None, 1, 1)
    ref = scipy_signal.correlate2d(x[0, :, :, 0], w[0, :, :, 0], mode="same")
    assert np.allclose(y[0, :, :, 0], ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("k,stride", [(3, 1), (3, 2), (1, 2)])
def test_conv_bwd_finite_differences(k, stride):
    r = rng(3)
    x = r.standard_normal((2, 6, 6, 3))
    w = r.standard_normal((4, k, k, 3))
    b = r.standard_normal(4)
    pad = k // 2
    R = r.standard_normal(O.conv_fwd(x, w, b, stride, pad).shape)
    dx, dw, db = O.conv_bwd(x, w, R, stride, pad, True)
    assert_fd(lambda xx: np.sum(O.conv_fwd(xx, w, b, stride, pad) * R), x, dx)
    assert_fd(lambda ww: np.sum(O.conv_fwd(x, ww, b, stride, pad) * R), w, dw)
    assert_fd(lambda bb: np.sum(O.conv_fwd(x, w, bb, stride, pad) * R), b, db)
    assert O.conv_bwd(x, w, R, stride, pad, False)[0] is None


# --------------------------------------------------------------------------
# pooling, relu, affine, linear
# --------------------------------------------------------------------------

def test_maxpool_tie_goes_to_first_in_row_major_order():
    x = np.zeros((1, 2, 2, 1))
    x[0, 0, 1, 0] = x[0, 1, 0, 0] = 5.0          # tie between (0,1) and (1,0)
    dy = np.ones((1, 1, 1, 1))
    dx = O.maxpool2_bwd(x, dy)
    assert dx[0, 0, 1, 0] == 1.0 and dx.sum() == 1.0
    assert O.maxpool2_fwd(x)[0, 0, 0, 0] == 5.0


def test_maxpool_brute_force_and_fd():
    r = rng(4)
    x = r.standard_normal((2, 4, 6, 3))
    y = O.maxpool2_fwd(x)
    for n, i, j, c in itertools.product(range(2), range(2), range(3), range(3)):
        assert y[n, i, j, c] == max(x[n, 2 * i + a, 2 * j + b, c] for a in (0, 1) for b in (0, 1))
    R = r.standard_normal(y.shape)
    assert_fd(lambda xx: np.sum(O.maxpool2_fwd(xx) * R), x, O.maxpool2_bwd(x, R))


def test_relu_derivative_at_zero_is_zero():
    x = np.array([-1.0, 0.0, 2.0])
    assert list(O.relu_bwd(x, np.ones(3))) == [0.0, 0.0, 1.0]


def test_affine_and_linear_fd():
    r = rng(5)
    x = r.standard_normal((2, 3, 3, 4))
    sc, sh = r.standard_normal(4), r.standard_normal(4)
    R = r.standard_normal(x.shape)
    dx, dsc, dsh = O.affine_bwd(x, sc, R)
    assert_fd(lambda t: np.sum(O.affine_fwd(t, sc, sh) * R), x, dx)
    assert_fd(lambda t: np.sum(O.affine_fwd(x, t, sh) * R), sc, dsc)
    assert_fd(lambda t: np.sum(O.affine_fwd(x, sc, t) * R), sh, dsh)
    xl = r.standard_normal((3, 2, 5))
    w, b = r.standard_normal((4, 5)), r.standard_normal(4)
    R = r.standard_normal((3, 2, 4))
    dx, dw, db = O.linear_bwd(xl, w, R, True)
    assert_fd(lambda t: np.sum(O.linear_fwd(t, w, b) * R), xl, dx)
    assert_fd(lambda t: np.sum(O.linear_fwd(xl, t, b) * R), w, dw)
    assert_fd(lambda t: np.sum(O.linear_fwd(xl, w, t) * R), b, db)
    # brute force of one output entry
    assert np.isclose(O.linear_fwd(xl, w, b)[1, 0, 2], sum(xl[1, 0, c] * w[2, c] for c in range(5)) + b[2])


def test_avgpool_and_flatten():
    r = rng(6)
    x = r.standard_normal((2, 3, 4, 5))
    y = O.avgpool_fwd(x)
    assert np.allclose(y[1, 2], x[1, :, :, 2].sum() / 12)
    R = r.standard_normal(y.shape)
    assert_fd(lambda t: np.sum(O.avgpool_fwd(t) * R), x, O.avgpool_bwd(x, R))


# --------------------------------------------------------------------------
# transformer pieces
# --------------------------------------------------------------------------

def test_layernorm_invariants_and_fd():
    r = rng(7)
    x = r.standard_normal((2, 5, 1, 8)) * 3 + 1
    y, cache = O.layernorm_fwd(x, np.ones(8), np.zeros(8))
    assert np.allclose(y.mean(-1), 0, atol=1e-12)
    # biased variance, eps = 1e-5: var(y) = var / (var + eps)
    v = x.var(-1)
    assert np.allclose(y.var(-1), v / (v + 1e-5), rtol=1e-12)
    g, bt = r.standard_normal(8), r.standard_normal(8)
    y, cache = O.layernorm_fwd(x, g, bt)
    R = r.standard_normal(y.shape)
    dx, dg, db = O.layernorm_bwd(cache, g, R)
    assert_fd(lambda t: np.sum(O.layernorm_fwd(t, g, bt)[0] * R), x, dx)
    assert_fd(lambda t: np.sum(O.layernorm_fwd(x, t, bt)[0] * R), g, dg)
    assert_fd(lambda t: np.sum(O.layernorm_fwd(x, g, t)[0] * R), bt, db)


def test_gelu_values_and_fd():
    xs = np.array([-3.0, -1.0, 0.0, 0.5, 2.0, 6.0])
    ref = np.array([v * 0.5 * (1 + math.erf(v / math.sqrt(2))) for v in xs])
    assert np.allclose(O.gelu_fwd(xs), ref, rtol=1e-14, atol=1e-15)
    assert O.gelu_fwd(np.array([0.0]))[0] == 0.0
    assert np.isclose(O.gelu_bwd(np.array([0.0]), np.ones(1))[0], 0.5)
    assert np.isclose(O.gelu_fwd(np.array([10.0]))[0], 10.0)
    x = rng(8).standard_normal(30)
    R = rng(9).standard_normal(30)
    assert_fd(lambda t: np.sum(O.gelu_fwd(t) * R), x, O.gelu_bwd(x, R))


def test_attention_special_cases():
    r = rng(10)
    B, L, d, h = 2, 5, 8, 2
    qkv = r.standard_normal((B, L, 1, 3 * d))
    # zero queries: every head averages the values of the valid keys
    q0 = qkv.copy()
    q0[..., :d] = 0
    lengths = np.array([3, 5])
    out, _ = O.attention_fwd(q0, lengths, d, h)
    for b in range(B):
        vmean = qkv[b, :lengths[b], 0, 2 * d:].mean(0)
        assert np.allclose(out[b, :, 0, :], vmean[None, :], rtol=1e-12)
    # masked keys and values have no influence
    out1, _ = O.attention_fwd(qkv, lengths, d, h)
    q2 = qkv.copy()
    q2[0, 3:, 0, d:] = 1e3
    out2, _ = O.attention_fwd(q2, lengths, d, h)
    assert np.allclose(out1, out2, rtol=1e-12)
    # a single valid key returns its value
    out3, _ = O.attention_fwd(qkv, np.array([1, 1]), d, h)
    assert np.allclose(out3[0, :, 0, :], qkv[0, 0, 0, 2 * d:][None, :])


def test_attention_brute_force_one_row():
    r = rng(11)
    B, L, d, h = 1, 4, 6, 2
    dh = d // h
    qkv = r.standard_normal((B, L, 1, 3 * d))
    out, _ = O.attention_fwd(qkv, np.array([3]), d, h)
    i, head = 2, 1
    q = qkv[0, i, 0, head * dh:(head + 1) * dh]
    sc = [np.dot(q, qkv[0, j, 0, d + head * dh:d + (head + 1) * dh]) / math.sqrt(dh) for j in range(3)]
    m = max(sc)
    w = [math.exp(s - m) for s in sc]
    ref = sum(w[j] * qkv[0, j, 0, 2 * d + head * dh:2 * d + (head + 1) * dh] for j in range(3)) / sum(w)
    assert np.allclose(out[0, i, 0, head * dh:(head + 1) * dh], ref, rtol=1e-12)


def test_attention_fd():
    r = rng(12)
    B, L, d, h = 2, 4, 8, 2
    qkv = r.standard_normal((B, L, 1, 3 * d))
    lengths = np.array([2, 4])
    out, cache = O.attention_fwd(qkv, lengths, d, h)
    R = r.standard_normal(out.shape)
    dqkv = O.attention_bwd(cache, R, d, h)
    assert_fd(lambda t: np.sum(O.attention_fwd(t, lengths, d, h)[0] * R), qkv, dqkv, n=60)


def test_meanpool():
    r = rng(13)
    x = r.standard_normal((2, 5, 1, 3))
    lengths = np.array([2, 5])
    y = O.meanpool_fwd(x, lengths)
    assert np.allclose(y[0], (x[0, 0, 0] + x[0, 1, 0]) / 2)
    R = r.standard_normal(y.shape)
    dx = O.meanpool_bwd(x, lengths, R)
    assert np.all(dx[0, 2:] == 0)
    assert_fd(lambda t: np.sum(O.meanpool_fwd(t, lengths) * R), x, dx)


# --------------------------------------------------------------------------
# loss and optimizer
# --------------------------------------------------------------------------

def test_ce_zero_logits_closed_form():
    B, C = 4, 10
    labels = np.array([0, 3, 9, 3])
    loss, dz = O.softmax_ce(np.zeros((B, C)), labels)
    assert math.isclose(loss, math.log(C), rel_tol=1e-14)
    ref = np.full((B, C), 1.0 / C)
    ref[np.arange(B), labels] -= 1.0
    assert np.allclose(dz, ref / B, rtol=1e-14, atol=1e-16)


def test_ce_fd_and_shift_invariance():
    r = rng(14)
    z = r.standard_normal((3, 5))
    labels = np.array([1, 4, 0])
    loss, dz = O.softmax_ce(z, labels)
    assert math.isclose(O.softmax_ce(z + 7.0, labels)[0], loss, rel_tol=1e-12)
    # logits far beyond exp's range: the loss and its gradient are unchanged
    # (a softmax that does not subtract the row maximum overflows here)
    lz, dzz = O.softmax_ce(z + 1000.0, labels)
    assert math.isclose(lz, loss, rel_tol=1e-9) and np.allclose(dzz, dz, rtol=1e-9, atol=1e-15)
    brute = np.mean([math.log(sum(math.exp(v) for v in z[b])) - z[b, labels[b]] for b in range(3)])
    assert math.isclose(loss, brute, rel_tol=1e-12)
    assert_fd(lambda t: O.softmax_ce(t, labels)[0], z, dz)


def test_sgd_momentum_constant_gradient_closed_form():
    g = np.array([0.5, -2.0, 1e-3])
    theta0 = np.array([1.0, 2.0, 3.0])
    lr, mu = 0.01, 0.9
    th, v = theta0.copy(), np.zeros(3)
    for n in range(1, 21):
        th, v = O.sgd_momentum(th, v, g, lr, mu)
        assert np.allclose(v, g * (1 - mu ** n) / (1 - mu), rtol=1e-13)
    # theta_n = theta_0 - lr * g * sum_{i=1..n} (1 - mu^i)/(1 - mu)
    s = sum((1 - mu ** i) / (1 - mu) for i in range(1, 21))
    assert np.allclose(th, theta0 - lr * g * s, rtol=1e-13)


# --------------------------------------------------------------------------
# bf16 storage reading
# --------------------------------------------------------------------------

def test_to_bf16_matches_bit_rounding_and_torch():
    import torch
    r = rng(20)
    x = (r.standard_normal(10000) * np.exp(r.uniform(-20, 20, 10000))).astype(np.float32)
    ref_bits, _ = W.round_to_bf16(x)[0], None
    assert np.array_equal(O.to_bf16(x.astype(np.float64)), ref_bits.astype(np.float64))
    t = torch.tensor(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.to_bf16(x.astype(np.float64)), t)


def test_to_bf16_ties_to_even():
    one = 1.0
    assert O.to_bf16(np.array([one + 2.0 ** -8]))[0] == 1.0               # tie -> even (1.0)
    assert O.to_bf16(np.array([one + 3 * 2.0 ** -8]))[0] == 1.0 + 2.0 ** -6  # tie -> even
    assert O.to_bf16(np.array([one + 2.0 ** -8 + 2.0 ** -30]))[0] == 1.0 + 2.0 ** -7
    assert O.to_bf16(np.array([0.0, -0.0]))[1] == 0.0


def test_bf16_storage_rounds_every_stored_tensor():
    from test_oracle_network import make_case
    ops, theta, x, labels, lengths = make_case("vgg")
    params = O.unflatten(ops, theta)
    T, _ = O.forward(ops, params, O.to_bf16(x), lengths, storage="bf16")
    for t in T[1:-1]:
        assert np.array_equal(O.to_bf16(t), t)
    assert not np.array_equal(O.to_bf16(T[-1]), T[-1])     # logits stay unrounded
    T64, _ = O.forward(ops, params, O.to_bf16(x), lengths)
    rel = np.linalg.norm(T[-1] - T64[-1]) / np.linalg.norm(T64[-1])
    assert 1e-5 < rel < 3e-2


def test_bf16_reading_keeps_the_classifier_weights_fp32():
    """In the bf16-storage reading every stored tensor and every hidden
    conv / linear weight is rounded, but the logits layer reads the fp32
    master weights (the classifier kernel does), so its output equals the
    fp64 product of the rounded input with the unrounded weights."""
    ops = [{"kind": "flatten", "in0": 0},
           {"kind": "linear", "in0": 1, "cin": 6, "cout": 3, "bias": 1}]
    r = rng(30)
    w = r.standard_normal((3, 6))
    w[0, 0] = 1.0 + 2.0 ** -12                    # not a bf16 value
    b = r.standard_normal(3)
    x = r.standard_normal((2, 1, 2, 3))
    params = {(1, "W"): w, (1, "b"): b}
    T, _ = O.forward(ops, params, x, None, storage="bf16")
    assert np.array_equal(T[-1], O.to_bf16(x).reshape(2, 6) @ w.T + b)
    hidden = [{"kind": "flatten", "in0": 0},
              {"kind": "linear", "in0": 1, "cin": 6, "cout": 3, "bias": 0},
              {"kind": "linear", "in0": 2, "cin": 3, "cout": 2, "bias": 0}]
    w2 = r.standard_normal((2, 3))
    T, _ = O.forward(hidden, {(1, "W"): w, (2, "W"): w2}, x, None, storage="bf16")
    h = O.to_bf16(O.to_bf16(x).reshape(2, 6) @ O.to_bf16(w).T)
    assert np.array_equal(T[2], h) and np.array_equal(T[3], h @ w2.T)
