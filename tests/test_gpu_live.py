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


def _device_floats(ptr, n, dev):
    """A copy of n fp32 values at a device pointer (CUDA array interface)."""
    import torch

    class _Arr:
        __cuda_array_interface__ = {"shape": (int(n),), "typestr": "<f4", "data": (ptr, False), "version": 3}
    return torch.as_tensor(_Arr(), device=dev).clone().cpu().numpy().astype(np.float64)


def test_live_device_iteration_and_aggregation_match_the_oracle():
    """Algorithm 1 inside the live pipeline, teacher-forced: after a warm-up
    of the whole pipeline, one device iteration (M_dk forward, auxiliary
    network, local loss f_d, backward, SGD-momentum) from the device's own
    parameters and momentum is compared with one exact oracle step on the
    same local batch, under the gates of harness.gate_failures; the model it
    then sends is aggregated into the global device model (Algorithm 4,
    aggregation branch), compared with the oracle's Aggregator at 1e-6."""
    import torch
    from harness import batch_for, gate_failures, param_slices, step_record
    from paper_2504_13850_gb300 import api, live
    dev = torch.device("cuda", 0)
    p = live.LivePipeline()
    p.run(30, agg_every=4)
    p.finish()
    dcfg, ops, mu = p.dcfg, p.dcfg["ops"], p.dcfg["momentum"]
    slices = param_slices(ops)
    checked = 0
    for k in range(p.K):
        if not p.server.sender_status()[k]:
            continue
        d = p.devices[k]
        j = p.local_steps[k] % len(p.data[k])
        x_dev, lab_dev = p.data[k][j]
        th0 = d.get_params().astype(np.float64)
        v0 = d.get_momentum().astype(np.float64)
        assert d.enqueue_activations(0, x_dev, lab_dev)[0] == api.OK
        assert d.server_step()[0] == api.OK
        d.synchronize()
        p.local_steps[k] += 1
        # the device's loss ring holds its own iterations: this one is the newest
        loss = float(d.read_losses(p.local_steps[k] - 1, 1)[0])
        th1 = d.get_params().astype(np.float64)
        v1 = d.get_momentum().astype(np.float64)
        x, _, y, _ = batch_for(dcfg, k, j)
        o = O.Server(ops, 1, 1, 1, th0, dcfg["lr"], mu)
        ob = O.Server(ops, 1, 1, 1, th0, dcfg["lr"], mu, storage="bf16")
        for srv in (o, ob):
            srv.theta, srv.v = th0.copy(), v0.copy()
            srv.enqueue(0, x, y)
            srv.step()
        rec = step_record(0, loss, th0, v0, th1, v1, o, ob, mu, slices)
        assert not gate_failures(rec), gate_failures(rec)
        # the device sends its model: FedAsync update of the global device model
        local_ptr, n = d.params_device()
        g_before = p.global_model.cpu().numpy().astype(np.float64)
        local = _device_floats(local_ptr, n, dev)
        t, _ = p.server.version()
        tk = p.version[k]
        rc, t_new = p.server.aggregate(p.global_model, local_ptr, k, tk)
        assert rc == api.OK and t_new == t + 1
        p.server.synchronize()
        agg = O.Aggregator(p.K, 2**31 - 1)
        agg.t = t
        st, expect = agg.aggregate(g_before, local, tk)
        assert st == O.OK
        got = p.global_model.cpu().numpy().astype(np.float64)
        assert np.linalg.norm(got - expect) <= 1e-6 * np.linalg.norm(expect)
        assert np.all(np.abs(got - expect) <= 1e-6 * (np.abs(g_before) + np.abs(local)) + 1e-30)
        checked += 1
        if checked == 2:
            break
    assert checked == 2
    p.close()
