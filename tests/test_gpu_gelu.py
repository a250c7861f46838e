"""The GELU kernels (the transformer's feed-forward activation, x Phi(x))
against the exact definition.  The kernels evaluate the normal distribution
function with a rational approximation of absolute error below 7.5e-8
(Abramowitz & Stegun 26.2.17), so:

* forward: every stored bf16 output lies within one rounding step of the
  exact value, 2^-8 |GELU(x)| (the bf16 spacing is at most 2^-7 |y|, and the
  approximation can move a value across a rounding boundary), plus 1e-6 for
  the approximation near zero and in the left tail;
* backward: the whole teacher-forced step (gradients of the linear layers
  on both sides of the GELU) under the gates of harness.gate_failures, and
  the fp32 path's full trace at 1e-4.

The network's first layer has its weights scaled by 4, so that the GELU's
inputs spread to about +-16 and cover both tails and the region around 0
(the classifier's by 1/4, so that the loss stays near ln 10)."""
import numpy as np
import pytest
from scipy.special import ndtr

from harness import check_teacher_forced, normwise, teacher_forced
from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W
from test_gpu_train import compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def gelu_ops(width=512):
    b = W._Builder()
    t = b.add("flatten", 0)
    t = b.add("linear", t, cin=4 * 4 * 16, cout=width, bias=1)
    t = b.add("gelu", t)
    b.add("linear", t, cin=width, cout=10, bias=1)
    return b.ops


def gelu_cfg(dtype, width=512):
    return W.shrink(W.CONFIGS["mobilenet"], ops=gelu_ops(width), classes=10, batch=64, in_hwc=(4, 4, 16), K=2,
                    omega=4, depth=2, dtype=dtype, lr=1e-3)


def wide_theta(cfg, width=512):
    th = W.init_params(cfg).copy()
    n1 = 4 * 4 * 16 * width
    th[:n1] *= 4.0                                      # the first linear layer's weights
    th[n1 + width:n1 + width + width * 10] *= 0.25      # the classifier's, so the logits stay near the start's scale
    return th


def _device_bf16(ptr, n):
    import torch

    class _Arr:
        __cuda_array_interface__ = {"shape": (int(n),), "typestr": "<i2", "data": (ptr, False), "version": 3}
    t = torch.as_tensor(_Arr(), device=torch.device("cuda", 0)).clone()
    return t.view(torch.bfloat16).float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("width", [512, 520])
def test_gelu_forward_is_the_rounded_exact_value(width):
    """Width 520: the last 32-column chunk of the GELU-storing epilogue is
    mostly past the end of the output (and a whole chunk of the last tile
    is)."""
    cfg = gelu_cfg(W.BF16, width)
    ev = [("enq", 0), ("enq", 1), ("step",), ("step",)]
    s, _, recs = teacher_forced(cfg, ev, theta0=wide_theta(cfg, width))
    assert len(recs) == 2
    x_ptr, x_dims, _ = s.tensor(2)          # the first linear layer's output: the GELU's input
    y_ptr, y_dims, dt = s.tensor(3)
    assert x_dims == y_dims and dt == api.DTYPE_BF16
    n = int(np.prod(y_dims))
    x, y = _device_bf16(x_ptr, n), _device_bf16(y_ptr, n)
    assert np.max(x) > 10 and np.min(x) < -10 and np.mean(np.abs(x) < 0.5) > 0.05
    exact = x * ndtr(x)
    err = np.abs(y - exact)
    bound = 2.0 ** -8 * np.abs(exact) + 1e-6
    assert np.all(err <= bound), (x[err > bound][:8], y[err > bound][:8], exact[err > bound][:8])
    check_teacher_forced(recs)


@pytest.mark.parametrize("width", [512, 520])
def test_gelu_backward_teacher_forced_bf16(width):
    """520 columns: a ragged last output tile in the linear layers on both
    sides of the GELU, and a bias gradient whose last 256-column block of
    the column sums holds one 8-column group."""
    cfg = gelu_cfg(W.BF16, width)
    ev = [("enq", k) for _ in range(2) for k in range(2)] + [("step",)] * 4
    _, _, recs = teacher_forced(cfg, ev, theta0=wide_theta(cfg, width))
    assert len(recs) == 4
    check_teacher_forced(recs)


def test_gelu_fp32_full_trace():
    """Losses and parameters at 1e-4; the momentum (the sum of the steps'
    gradients) at 1e-4 too.  The update theta - theta0 is not gated here:
    with the first layer's weights scaled by 4 an fp32 weight's spacing is
    ~3e-8 against updates of ~1e-4, so its rounding alone is ~1e-4 of the
    update."""
    cfg = gelu_cfg(W.F32)
    ev = [("enq", k) for _ in range(2) for k in range(2)] + [("step",)] * 4
    s, o = compare(cfg, ev, loss_tol=1e-4, param_tol=1e-4, theta0=wide_theta(cfg))
    assert normwise(s.get_momentum(), o.v) <= 1e-4
