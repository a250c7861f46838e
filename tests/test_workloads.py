"""The seeded inputs follow the stated recipe (CPU only): activation batches
ReLU(N(0,1)) (image) or N(0,1) (sequence), rounded to bf16 by
round-to-nearest-even for the bf16 workloads, labels uniform over the
classes, lengths uniform over 32..128; device models N(0, 0.05); initial
weights He-normal with zero biases and unit scales; arrivals Poisson with
the four testbed-B groups' rates or Zipf(1.2); the workload table."""
import math

import numpy as np
import pytest

from paper_2504_13850_gb300 import workloads as W


def test_batches_are_deterministic_and_distinct():
    cfg = W.CONFIGS["vgg"]
    a = W.device_batch(cfg, 3, 7)
    b = W.device_batch(cfg, 3, 7)
    assert all(np.array_equal(u, v) for u, v in zip(a[:3], b[:3]))
    for other in (W.device_batch(cfg, 4, 7), W.device_batch(cfg, 3, 8)):
        assert not np.array_equal(a[0], other[0])


def test_image_batches_are_relu_of_a_standard_normal_rounded_to_bf16():
    cfg = W.CONFIGS["vgg"]
    x, bits, labels, lengths = W.device_batch(cfg, 0, 0)
    assert x.shape == (64, 16, 16, 128) and x.dtype == np.float32 and lengths is None
    assert np.array_equal((bits.astype(np.uint32) << 16).view(np.float32), x)
    assert np.array_equal(W.round_to_bf16(x)[0], x)
    n = x.size
    zero = np.mean(x == 0.0)
    assert abs(zero - 0.5) < 4 * math.sqrt(0.25 / n)
    pos = x[x > 0].astype(np.float64)
    assert pos.mean() == pytest.approx(math.sqrt(2 / math.pi), rel=5e-3)    # half-normal mean
    assert pos.var() == pytest.approx(1 - 2 / math.pi, rel=1e-2)
    assert labels.dtype == np.int32 and labels.min() >= 0 and labels.max() < cfg["classes"]


def test_fp32_batches_are_not_rounded():
    x, bits, _, _ = W.device_batch(W.CONFIGS["tiny"], 1, 2)
    assert bits is None and not np.array_equal(W.round_to_bf16(x)[0], x)


def test_sequence_batches():
    cfg = W.CONFIGS["transformer"]
    counts = np.zeros(129, np.int64)
    lab = []
    for j in range(40):
        x, _, labels, lengths = W.device_batch(cfg, j % cfg["K"], j)
        assert x.shape == (32, 128, 1, 512)
        counts += np.bincount(lengths, minlength=129)
        lab.append(labels)
    assert counts[:32].sum() == 0 and counts[32:].min() > 0              # uniform over 32..128
    lab = np.concatenate(lab)
    assert set(np.unique(lab)) == {0, 1} and abs(lab.mean() - 0.5) < 0.1
    assert abs(float(x.mean())) < 0.01 and float(x.var()) == pytest.approx(1.0, rel=0.02)


def test_round_to_bf16_ties_to_even():
    v = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 1.0 + 2.0 ** -8 + 2.0 ** -20],
                 np.float32)
    got, _ = W.round_to_bf16(v)
    assert got.tolist() == [1.0, 1.0 + 2.0 ** -6, -1.0, 1.0 + 2.0 ** -7]


def test_device_and_global_models_are_n_0_005():
    for m in (W.device_model(200_000, 1, 3, 0), W.global_model(200_000, 1)):
        assert m.dtype == np.float32 and abs(float(m.mean())) < 1e-3
        assert float(m.std()) == pytest.approx(0.05, rel=0.01)
    assert not np.array_equal(W.device_model(10, 1, 3, 0), W.device_model(10, 1, 3, 1))


def test_initial_weights_are_he_normal():
    cfg = W.CONFIGS["vgg"]
    theta = W.init_params(cfg)
    off = 0
    for name, shape in W.param_shapes(cfg["ops"]):
        n = int(np.prod(shape))
        t = theta[off:off + n].astype(np.float64)
        off += n
        if name == "W":
            std = math.sqrt(2.0 / np.prod(shape[1:]))
            assert t.std() == pytest.approx(std, rel=max(0.02, 5 / math.sqrt(n)))
        else:
            assert np.all(t == 0.0)
    assert off == theta.size
    lt = W.init_params(W.CONFIGS["transformer"])
    shapes = W.param_shapes(W.CONFIGS["transformer"]["ops"])
    off = 0
    for name, shape in shapes:
        n = int(np.prod(shape))
        if name == "gamma":
            assert np.all(lt[off:off + n] == 1.0)
        if name == "beta":
            assert np.all(lt[off:off + n] == 0.0)
        off += n


def test_rates_and_arrivals():
    assert W.group_rates(8) == [240.0] * 2 + [320.0] * 2 + [640.0] * 2 + [921.0] * 2
    z = W.zipf_rates(100)
    assert z[0] == 1.0 and z[9] == pytest.approx(10 ** -1.2)
    rates = W.group_rates(4)
    order = W.arrival_order(rates, 20_000, 0)
    freq = np.bincount(order, minlength=4) / len(order)
    np.testing.assert_allclose(freq, np.array(rates) / sum(rates), atol=0.01)


def test_workload_table():
    want = {   # K, omega, depth, batch, per-sample input, dtype, classes
        "tiny": (4, 8, 2, 16, (16, 16, 32), W.F32, 10),
        "vgg": (10, 40, 4, 64, (16, 16, 128), W.BF16, 10),
        "resnet": (20, 80, 4, 128, (16, 16, 128), W.BF16, 100),
        "transformer": (16, 64, 4, 32, (128, 1, 512), W.BF16, 2),
        "scale": (100, 400, 4, 64, (16, 16, 128), W.BF16, 100),
        "mobilenet": (10, 40, 4, 64, (4, 4, 112), W.BF16, 200),
    }
    for name, (K, omega, depth, batch, hwc, dt, classes) in want.items():
        c = W.CONFIGS[name]
        assert (c["K"], c["omega"], c["depth"], c["batch"], c["in_hwc"], c["dtype"], c["classes"]) == \
            (K, omega, depth, batch, hwc, dt, classes), name
        assert c["lr"] == 0.01 and c["momentum"] == 0.9
    assert W.num_params(W.CONFIGS["mobilenet"]["ops"]) == 3_665_744
    assert W.CONFIGS["vgg"]["agg_params"] == 1_000_000 and W.CONFIGS["tiny"]["agg_params"] == 20_000
