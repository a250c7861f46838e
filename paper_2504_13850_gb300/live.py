"""Devices and server on one GPU: the VGG-style split run end to end.

Each of the server's K devices is its own fo_server holding M_dk and the
default auxiliary network (``workloads.vgg_device_ops``).  One device event
follows Algorithm 1: the device trains one iteration on a batch of its local
(synthetic) data with its local loss f_d, and uploads the split-point
activation of that iteration, with its labels, to the server's queue
(Algorithm 2; a device the flow control has turned off skips its turn).
Every ``agg_every`` local iterations the device sends its model (M_dk and the
auxiliary network, one flat vector) for FedAsync aggregation (Algorithm 4)
and continues from the returned global model.  The server trains on its
queues in the Task Scheduler's order (Algorithm 3), one iteration per event.
Device and server work run on their own CUDA streams, so they overlap.
"""
import time

import numpy as np

from . import api
from . import workloads as W


class LivePipeline:
    def __init__(self, server_cfg="vgg", device_cfg="vgg_device", split=W.VGG_DEVICE_SPLIT, pool=4, seed=0):
        import torch
        self.torch = torch
        self.scfg, self.dcfg = W.CONFIGS[server_cfg], W.CONFIGS[device_cfg]
        self.K, self.split = self.scfg["K"], split
        dev = torch.device("cuda", torch.cuda.current_device())
        self.server = api.Server.from_config(self.scfg)
        self.server.set_params(W.init_params(self.scfg))
        theta0 = W.init_params(self.dcfg)
        self.devices = []
        for _ in range(self.K):
            d = api.Server.from_config(self.dcfg)
            d.set_params(theta0)
            self.devices.append(d)
        # local data of each device: a pool of batches resident in HBM
        self.data = []
        for k in range(self.K):
            batches = []
            for j in range(pool):
                x, bits, labels, _ = W.device_batch(self.dcfg, k, j)
                up = bits.view(np.int16) if bits is not None else x
                batches.append((torch.from_numpy(np.ascontiguousarray(up)).to(dev),
                                torch.from_numpy(labels).to(dev)))
            self.data.append(batches)
        # the global device model (padded device layout) and each device's version t_k
        ptr, n = self.devices[0].params_device()
        self.n_dev_params = n
        self.global_model = torch.empty(n, dtype=torch.float32, device=dev)
        self.devices[0].store_params_device(self.global_model.data_ptr(), n)
        self.devices[0].synchronize()
        self.version = [0] * self.K
        self.local_steps = [0] * self.K
        self.order = W.arrival_order(self.scfg["rates"], 1_000_000, self.scfg["seed"] + seed)
        self.pos = 0
        self.a_stream = torch.cuda.ExternalStream(self.server.agg_stream(), device=dev)
        self.stats = {"device_iterations": 0, "uploads": 0, "refused": 0, "skipped_off": 0, "server_steps": 0,
                      "aggregations": 0, "stale": 0}

    def event(self, agg_every):
        """One device event and one server iteration."""
        k = self.order[self.pos % len(self.order)]
        self.pos += 1
        if self.server.sender_status()[k]:
            d = self.devices[k]
            x, labels = self.data[k][self.local_steps[k] % len(self.data[k])]
            rc, _ = d.enqueue_activations(0, x, labels)
            assert rc == api.OK, rc
            rc, _, _ = d.server_step()                      # M_dk + auxiliary network, local loss
            assert rc == api.OK, rc
            d.synchronize()
            self.stats["device_iterations"] += 1
            self.local_steps[k] += 1
            ptr, _, _ = d.tensor(self.split)                # the split-point activation of that iteration
            rc, _ = self.server.enqueue_activations(k, ptr, labels)
            if rc == api.OK:
                self.stats["uploads"] += 1
            else:
                self.stats["refused"] += 1
            if self.local_steps[k] % agg_every == 0:
                local_ptr, _ = d.params_device()
                rc, t = self.server.aggregate(self.global_model, local_ptr, k, self.version[k])
                if rc == api.STALE:
                    self.stats["stale"] += 1
                else:
                    self.stats["aggregations"] += 1
                self.version[k], _ = self.server.version()
                # the device continues from the global model once the update is done
                ev = self.torch.cuda.Event()
                ev.record(self.a_stream)
                ev.synchronize()
                d.load_params_device(self.global_model.data_ptr(), self.n_dev_params)
        else:
            self.stats["skipped_off"] += 1
        rc, _, _ = self.server.server_step()
        if rc == api.OK:
            self.stats["server_steps"] += 1

    def run(self, events, agg_every=8):
        for _ in range(events):
            self.event(agg_every)

    def close(self):
        """Destroys the servers before the buffers they used."""
        self.finish()
        for d in self.devices:
            d.close()
        self.server.close()
        self.devices, self.data, self.global_model = [], [], None

    def finish(self):
        self.server.synchronize()
        for d in self.devices:
            d.synchronize()
        self.server.check_error()
        for d in self.devices:
            d.check_error()


def measure(events=400, warmup=40, agg_every=8):
    """Wall-clock throughput of the live pipeline: server and device
    training samples per second."""
    import torch
    p = LivePipeline()
    p.run(warmup, agg_every)
    p.finish()
    s0 = dict(p.stats)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    p.run(events, agg_every)
    p.finish()
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    d = {k: p.stats[k] - s0[k] for k in p.stats}
    B = p.scfg["batch"]
    p.close()
    return {"events": events, "seconds": round(dt, 4),
            "server_samples_per_s": round(d["server_steps"] * B / dt, 1),
            "device_samples_per_s": round(d["device_iterations"] * p.dcfg["batch"] / dt, 1),
            "counts": d, "devices": p.K, "agg_every": agg_every,
            "device_network": "conv3x3 3->128, ReLU, maxpool2 (M_dk, split output [16,16,128]) + aux conv3x3 "
                              "128->128, ReLU, avgpool, FC 128->10; batch 64 of [32,32,3]"}
