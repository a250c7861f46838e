"""Server creation refuses bad configurations and op lists on the host, before
any CUDA call (shape inference and the configuration checks of
fo_server_create), so these run on the CPU.  Each case names the error text
it must produce.  Every shipped workload passes the same checks: without a GPU
its create stops at stream creation (FO_ERR_CUDA), never at FO_ERR_ARG."""
import pytest

from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W


@pytest.fixture(scope="module", autouse=True)
def built_library():
    build.build()
    api.lib()


def create(cfg, **over):
    return api.Server.from_config(cfg, **over)


def refused(match, cfg, **over):
    with pytest.raises(api.FedOptimaError) as e:
        create(cfg, **over)
    assert "ERR_ARG" in str(e.value), str(e.value)
    assert match in str(e.value), str(e.value)


def no_gpu():
    try:
        import torch
        return not torch.cuda.is_available()
    except ImportError:
        return True


TINY = W.CONFIGS["tiny"]          # [16, 16, 32] input, 10 classes


def head(in0, cin, classes=10):
    return [{"kind": "flatten", "in0": in0}, {"kind": "linear", "in0": in0 + 1, "cin": cin, "cout": classes, "bias": 1}]


@pytest.mark.parametrize("field,value", [
    ("K", 0), ("K", (1 << 20) + 1), ("omega", 0), ("omega", (1 << 24) + 1), ("depth", 0),
    ("batch", 0), ("batch", 1025), ("num_classes", 0), ("dtype", "f16"), ("max_delay", -1), ("policy", 2),
])
def test_bad_server_configuration(field, value):
    if field == "dtype":
        # the binding maps anything but "bf16" to fp32; pass the raw code instead
        L = api.lib()
        import ctypes as C
        ops = api.ops_to_c(TINY["ops"])
        opt = api.fo_optimizer(0.01, 0.9)
        cfg = api.fo_server_cfg(4, 8, 2, 16, 16, 16, 32, 10, 7, 0, 2**31 - 1, 0)
        h = C.c_void_p()
        assert L.fo_server_create(ops, len(TINY["ops"]), C.byref(opt), C.byref(cfg), C.byref(h)) == api.ERR_ARG
        return
    refused("bad server configuration", TINY, **{field: value})


def test_input_larger_than_int32_per_sample():
    refused("activation elements per sample", TINY, in_hwc=(65536, 65536, 1))


@pytest.mark.parametrize("ops,match", [
    ([{"kind": "relu", "in0": 1}] + head(1, 16 * 16 * 32), "bad in0"),
    ([{"kind": "conv", "in0": 0, "cin": 16, "cout": 8, "k": 3, "stride": 1, "bias": 0}] + head(1, 16 * 16 * 8),
     "bad conv"),
    ([{"kind": "conv", "in0": 0, "cin": 32, "cout": 8, "k": 5, "stride": 1, "bias": 0}] + head(1, 16 * 16 * 8),
     "bad conv"),
    ([{"kind": "conv", "in0": 0, "cin": 32, "cout": 8, "k": 3, "stride": 3, "bias": 0}] + head(1, 6 * 6 * 8),
     "bad conv"),
    ([{"kind": "affine", "in0": 0, "c": 31}] + head(1, 16 * 16 * 32), "affine channels"),
    ([{"kind": "maxpool2", "in0": 0}, {"kind": "maxpool2", "in0": 1}, {"kind": "maxpool2", "in0": 2},
      {"kind": "maxpool2", "in0": 3}, {"kind": "maxpool2", "in0": 4}] + head(5, 32), "maxpool odd size"),
    ([{"kind": "relu", "in0": 0}, {"kind": "add", "in0": 1, "in1": 3}] + head(2, 16 * 16 * 32), "bad in1"),
    ([{"kind": "maxpool2", "in0": 0}, {"kind": "add", "in0": 1, "in1": 0}] + head(2, 8 * 8 * 32),
     "add shapes differ"),
    ([{"kind": "flatten", "in0": 0}, {"kind": "linear", "in0": 1, "cin": 100, "cout": 10, "bias": 1}],
     "linear cin"),
    ([{"kind": "layernorm", "in0": 0, "c": 32}, {"kind": "layernorm", "in0": 1, "c": 30}] + head(2, 16 * 16 * 32),
     "layernorm channels"),
    ([{"kind": "attention", "in0": 0, "cin": 32, "heads": 1}] + head(1, 16 * 16 * 32), "attention shape"),
    ([{"kind": "meanpool", "in0": 0}] + head(1, 16 * 32), "meanpool shape"),
    ([{"kind": "dwconv", "in0": 0, "c": 32, "k": 9, "stride": 1, "bias": 0}] + head(1, 16 * 16 * 32),
     "bad depthwise conv"),
    ([{"kind": "dwconv", "in0": 0, "c": 32, "k": 3, "stride": 2, "bias": 0}, {"kind": "chmul", "in0": 0, "in1": 1}]
     + head(2, 16 * 16 * 32), "channel scale must be [B, 1, 1, C]"),
    ([{"kind": "relu", "in0": 0}, {"kind": "avgpool", "in0": 1}], "the last op must be a linear layer"),
    (head(0, 16 * 16 * 32, classes=7), "the last op must be a linear layer"),
    ([{"kind": "conv", "in0": 0, "cin": 32, "cout": 1 << 24, "k": 1, "stride": 1, "bias": 0}]
     + head(1, 16 * 16 * 32), "elements per sample"),
])
def test_bad_op_lists(ops, match):
    refused(match, TINY, ops=ops)


def test_unknown_op_kind():
    import ctypes as C
    L = api.lib()
    ops = api.ops_to_c(head(0, 16 * 16 * 32))
    ops[0].kind = 99
    opt = api.fo_optimizer(0.01, 0.9)
    cfg = api.fo_server_cfg(4, 8, 2, 16, 16, 16, 32, 10, 0, 0, 2**31 - 1, 0)
    h = C.c_void_p()
    assert L.fo_server_create(ops, 2, C.byref(opt), C.byref(cfg), C.byref(h)) == api.ERR_ARG
    assert b"unknown kind" in L.fo_last_error()


@pytest.mark.skipif(not no_gpu(), reason="checks the host-side validation only where no GPU can be reached")
@pytest.mark.parametrize("name", list(W.CONFIGS))
def test_every_workload_passes_validation(name):
    with pytest.raises(api.FedOptimaError) as e:
        create(W.CONFIGS[name])
    assert "ERR_CUDA" in str(e.value), str(e.value)
