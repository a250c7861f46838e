"""Devices and server on one GPU (the live VGG-style pipeline): each device's
network (M_dk + auxiliary network) trains as its own fo_server and uploads
the split-point activation of each local iteration to the server; models go
through FedAsync aggregation.  Checks the pipeline end to end and the
uploaded activation against the oracle."""
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.join(os.path.dirname(__file__), "..", "oracle"))
import fo_oracle as O  # noqa: E402

pytestmark = pytest.mark.gpu


def test_split_activation_matches_oracle():
    import torch
    from paper_2504_13850_gb300 import api
    from paper_2504_13850_gb300 import workloads as W
    cfg = W.CONFIGS["vgg_device"]
    d = api.Server.from_config(cfg)
    theta = W.init_params(cfg)
    d.set_params(theta)
    x, bits, labels, _ = W.device_batch(cfg, 3, 0)
    dev = torch.device("cuda", 0)
    up = torch.from_numpy(np.ascontiguousarray(bits.view(np.int16))).to(dev)
    assert d.enqueue_activations(0, up, torch.from_numpy(labels).to(dev))[0] == api.OK
    assert d.server_step()[0] == api.OK
    d.synchronize()
    ptr, dims, dt = d.tensor(W.VGG_DEVICE_SPLIT)
    assert dims == (64, 16, 16, 128) and dt == api.DTYPE_BF16
    # read the device tensor through the CUDA array interface
    class _Arr:
        __cuda_array_interface__ = {"shape": (int(np.prod(dims)),), "typestr": "<i2", "data": (ptr, False),
                                    "version": 3}
    flat = torch.as_tensor(_Arr(), device=dev).clone()
    ref_T, _ = O.forward(cfg["ops"], O.unflatten(cfg["ops"], theta.astype(np.float64)), x, None, storage="bf16")
    ref = ref_T[W.VGG_DEVICE_SPLIT].reshape(-1)
    g = flat.view(torch.bfloat16).float().cpu().numpy().astype(np.float64)
    err = np.linalg.norm(g - ref) / np.linalg.norm(ref)
    assert err < 1e-2, err


def test_live_pipeline_trains_devices_and_server():
    import torch
    from paper_2504_13850_gb300 import live
    p = live.LivePipeline()
    p.run(80, agg_every=4)
    p.finish()
    st = p.stats
    assert st["device_iterations"] > 20 and st["uploads"] > 20 and st["server_steps"] > 20
    assert st["aggregations"] > 0
    losses = p.server.read_losses(0, st["server_steps"])
    assert np.all(np.isfinite(losses))
    assert np.all(np.isfinite(p.global_model.cpu().numpy()))
    # every server iteration consumed one upload of a device that is still queued or done
    assert st["server_steps"] <= st["uploads"]
