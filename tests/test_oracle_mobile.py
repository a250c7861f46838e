"""Pins for the oracle's MobileNetV3 pieces (CPU only): depthwise
convolution against the (already pinned) full convolution with a
block-diagonal weight, hard swish / hard sigmoid closed forms, and finite
differences of the channel scaling."""
import numpy as np
import pytest

from oracle import fo_oracle as O


def _block_diag(wd, C):
    k = wd.shape[1]
    w = np.zeros((C, k, k, C))
    for c in range(C):
        w[c, :, :, c] = wd[c]
    return w


@pytest.mark.parametrize("k,stride", [(3, 1), (3, 2), (5, 1), (5, 2)])
def test_depthwise_is_a_block_diagonal_convolution(k, stride):
    r = np.random.default_rng(k * 10 + stride)
    N, H, W, C = 2, 7, 6, 5
    x = r.standard_normal((N, H, W, C))
    wd = r.standard_normal((C, k, k))
    b = r.standard_normal(C)
    y = O.dwconv_fwd(x, wd, b, stride, k // 2)
    yf = O.conv_fwd(x, _block_diag(wd, C), b, stride, k // 2)
    np.testing.assert_allclose(y, yf, rtol=1e-12, atol=1e-12)
    dy = r.standard_normal(y.shape)
    dx, dw, db = O.dwconv_bwd(x, wd, dy, stride, k // 2, True)
    dxf, dwf, dbf = O.conv_bwd(x, _block_diag(wd, C), dy, stride, k // 2, True)
    np.testing.assert_allclose(dx, dxf, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dw, np.stack([dwf[c, :, :, c] for c in range(C)]), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(db, dbf, rtol=1e-12, atol=1e-12)


def test_hard_swish_and_sigmoid_values():
    x = np.array([-4.0, -3.0, -1.5, 0.0, 1.0, 3.0, 4.0])
    np.testing.assert_allclose(O.hswish_fwd(x), [0.0, 0.0, -1.5 * 1.5 / 6, 0.0, 4.0 / 6, 3.0, 4.0])
    np.testing.assert_allclose(O.hsigmoid_fwd(x), [0.0, 0.0, 0.25, 0.5, 4.0 / 6, 1.0, 1.0])
    # derivatives away from the kinks, by central differences
    h = 1e-6
    for xv in (-5.0, -2.2, -0.4, 0.9, 2.7, 5.0):
        fd = (O.hswish_fwd(np.array([xv + h])) - O.hswish_fwd(np.array([xv - h]))) / (2 * h)
        assert O.hswish_bwd(np.array([xv]), np.array([1.0]))[0] == pytest.approx(fd[0], abs=1e-8)
        fd = (O.hsigmoid_fwd(np.array([xv + h])) - O.hsigmoid_fwd(np.array([xv - h]))) / (2 * h)
        assert O.hsigmoid_bwd(np.array([xv]), np.array([1.0]))[0] == pytest.approx(fd[0], abs=1e-8)


def test_channel_scaling_gradients():
    r = np.random.default_rng(7)
    x = r.standard_normal((2, 3, 4, 5))
    s = r.standard_normal((2, 5))
    dy = r.standard_normal(x.shape)
    dx, ds = O.chmul_bwd(x, s, dy)
    f = lambda xx, ss: float((O.chmul_fwd(xx, ss) * dy).sum())
    h = 1e-6
    for idx in [(0, 1, 2, 3), (1, 0, 3, 0)]:
        e = np.zeros_like(x)
        e[idx] = h
        assert dx[idx] == pytest.approx((f(x + e, s) - f(x - e, s)) / (2 * h), rel=1e-6)
    for idx in [(0, 2), (1, 4)]:
        e = np.zeros_like(s)
        e[idx] = h
        assert ds[idx] == pytest.approx((f(x, s + e) - f(x, s - e)) / (2 * h), rel=1e-6)



def test_kink_derivatives_are_the_stated_one_sided_limits():
    """At exactly -3 and 3 the derivative is a convention (any value between
    the one-sided derivatives is a subgradient).  The one taken here, by the
    oracle and the kernels alike, is checked against one-sided finite
    differences: hard swish uses its interior formula on the closed interval
    [-3, 3] (the right derivative at -3, the left one at 3); hard sigmoid
    uses 1/6 only strictly inside, so at both kinks it takes the outer
    one-sided derivative, 0.  PyTorch 2.11 agrees on hard sigmoid but gives
    hard swish the open interval (0 at -3, 1 at 3)."""
    h = 1e-7
    one = np.ones(1)

    def right(f, x):
        return float((f(np.array([x + h])) - f(np.array([x])))[0] / h)

    def left(f, x):
        return float((f(np.array([x])) - f(np.array([x - h])))[0] / h)

    assert O.hswish_bwd(np.array([-3.0]), one)[0] == pytest.approx(right(O.hswish_fwd, -3.0), abs=1e-6)
    assert O.hswish_bwd(np.array([3.0]), one)[0] == pytest.approx(left(O.hswish_fwd, 3.0), abs=1e-6)
    assert O.hsigmoid_bwd(np.array([-3.0]), one)[0] == pytest.approx(left(O.hsigmoid_fwd, -3.0), abs=1e-6)
    assert O.hsigmoid_bwd(np.array([3.0]), one)[0] == pytest.approx(right(O.hsigmoid_fwd, 3.0), abs=1e-6)
