"""MobileNetV3 bottleneck layers on the GPU against the oracle: depthwise
convolution (strides 1 and 2, with and without bias), hard swish, hard
sigmoid and the squeeze-and-excite channel scaling, inside small networks
that still span several tiles and ragged channel tails, on both precisions.

fp32 path: the full trace (scheduler outcomes bit-exact, loss 1e-4,
parameters, update and momentum 1e-4 normwise: fp32 roundings over sums of
at most a few thousand terms).  bf16 path: teacher-forced steps against the
exact oracle with the gates of harness.gate_failures (the hard sigmoid's
derivative jumps at -3 and 3 and the SE block has a ReLU, so decisions at
those kinks can flip: the allowance of harness.grad_bound applies).
"""
import pytest

from harness import check_teacher_forced, teacher_forced
from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W
from test_gpu_train import compare, prefill_then_steps

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def small_mobile(dtype):
    """Two bottlenecks (5x5 stride 2 with SE and hard swish; 3x3 stride 1
    with ReLU, a biased depthwise conv and a residual) and the head."""
    b = W._Builder()
    t = W._bneck(b, 0, 24, 72, 40, 5, 2)
    u = b.add("conv", t, cin=40, cout=120, k=1, stride=1, bias=0)
    u = b.add("affine", u, c=120)
    u = b.add("relu", u)
    u = b.add("dwconv", u, c=120, k=3, stride=1, bias=1)
    u = b.add("hswish", u)
    sq = b.add("avgpool", u)
    sq = b.add("linear", sq, cin=120, cout=30, bias=1)
    sq = b.add("relu", sq)
    sq = b.add("linear", sq, cin=30, cout=120, bias=1)
    sq = b.add("hsigmoid", sq)
    u = b.add("chmul", u, in1=sq)
    u = b.add("conv", u, cin=120, cout=40, k=1, stride=1, bias=0)
    u = b.add("affine", u, c=40)
    t = b.add("add", u, in1=t)
    t = b.add("conv", t, cin=40, cout=96, k=1, stride=1, bias=0)
    t = b.add("affine", t, c=96)
    t = b.add("hswish", t)
    t = b.add("avgpool", t)
    t = b.add("linear", t, cin=96, cout=64, bias=1)
    t = b.add("hswish", t)
    b.add("linear", t, cin=64, cout=10, bias=1)
    return W.shrink(W.CONFIGS["mobilenet"], ops=b.ops, classes=10, batch=10, in_hwc=(7, 7, 24), K=3, omega=6, depth=2,
                    dtype=dtype)


def test_small_mobile_fp32_full_trace():
    cfg = small_mobile(W.F32)
    compare(cfg, prefill_then_steps(cfg, 6), loss_tol=1e-4, param_tol=1e-4, upd_tol=1e-4)


def test_small_mobile_bf16_teacher_forced():
    cfg = small_mobile(W.BF16)
    _, _, recs = teacher_forced(cfg, prefill_then_steps(cfg, 6))
    assert len(recs) == 6
    check_teacher_forced(recs)


def test_depthwise_gradients_reach_the_input_layer():
    """A depthwise conv reading the uploaded batch (no input gradient) and a
    channel scale whose gate is computed from it (neither passes a gradient
    to the upload): the fp32 trace still matches."""
    b = W._Builder()
    t = b.add("dwconv", 0, c=16, k=5, stride=2, bias=1)
    g = b.add("avgpool", 0)
    g = b.add("hsigmoid", g)
    t2 = b.add("chmul", 0, in1=g)
    t2 = b.add("maxpool2", t2)
    t2 = b.add("dwconv", t2, c=16, k=3, stride=1, bias=0)
    t = b.add("add", t, in1=t2)
    t = b.add("hswish", t)
    t = b.add("flatten", t)
    b.add("linear", t, cin=4 * 4 * 16, cout=10, bias=1)
    cfg = W.shrink(W.CONFIGS["mobilenet"], ops=b.ops, classes=10, batch=6, in_hwc=(8, 8, 16), K=2, omega=4, depth=2,
                   dtype=W.F32)
    compare(cfg, prefill_then_steps(cfg, 4), loss_tol=1e-4, param_tol=1e-4, upd_tol=1e-4)


def test_bad_mobile_shapes_are_refused():
    base = W.CONFIGS["mobilenet"]
    bad = [
        [{"kind": "dwconv", "in0": 0, "c": 100, "k": 5, "stride": 2, "bias": 0}],   # channels
        [{"kind": "dwconv", "in0": 0, "c": 112, "k": 4, "stride": 1, "bias": 0}],   # even k
        [{"kind": "dwconv", "in0": 0, "c": 112, "k": 3, "stride": 3, "bias": 0}],   # stride
        [{"kind": "chmul", "in0": 0, "in1": 0}],                                    # gate not [B,1,1,C]
    ]
    for ops in bad:
        ops = ops + [{"kind": "flatten", "in0": 1}, {"kind": "linear", "in0": 2, "cin": 4 * 4 * 112, "cout": 10,
                                                      "bias": 1}]
        with pytest.raises(RuntimeError):
            api.Server.from_config(W.shrink(base, ops=ops, classes=10))


def test_depthwise_any_kernel_size():
    """Kernel sizes outside the unrolled 3 / 5 (k = 7 stride 1, k = 1
    stride 2) take the generic depthwise kernels; bf16 teacher-forced."""
    b = W._Builder()
    t = b.add("dwconv", 0, c=16, k=7, stride=1, bias=1)
    t = b.add("affine", t, c=16)
    t = b.add("hswish", t)
    t = b.add("dwconv", t, c=16, k=1, stride=2, bias=0)
    t = b.add("hswish", t)
    t = b.add("flatten", t)
    b.add("linear", t, cin=4 * 4 * 16, cout=10, bias=1)
    for dtype in (W.F32, W.BF16):
        cfg = W.shrink(W.CONFIGS["mobilenet"], ops=b.ops, classes=10, batch=6, in_hwc=(8, 8, 16), K=2, omega=4, depth=2,
                       dtype=dtype)
        if dtype == W.F32:
            compare(cfg, prefill_then_steps(cfg, 4), loss_tol=1e-4, param_tol=1e-4, upd_tol=1e-4)
        else:
            _, _, recs = teacher_forced(cfg, prefill_then_steps(cfg, 4))
            check_teacher_forced(recs)
