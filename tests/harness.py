"""Trace replay on both sides (the CUDA library through the C ABI, and the
oracle) from the same seeded inputs, for the parity tests."""
import numpy as np

from oracle import fo_oracle as O
from paper_2504_13850_gb300 import workloads as W


def gpu_available():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


def batch_for(cfg, k, j):
    x, bits, labels, lengths = W.device_batch(cfg, k, j)
    upload = bits if cfg["dtype"] == W.BF16 else x
    return x, np.ascontiguousarray(upload), labels, lengths


def replay_gpu(cfg, events, theta0=None, server=None):
    """Replays ("enq", k) / ("step",) events through the C ABI.  Returns the
    server and the log of outcomes."""
    from paper_2504_13850_gb300 import api
    s = server or api.Server.from_config(cfg)
    if server is None:
        s.set_params(W.init_params(cfg) if theta0 is None else theta0)
    log, nb = [], {}
    for ev in events:
        if ev[0] == "enq":
            k = ev[1]
            j = nb.get(k, 0)
            nb[k] = j + 1
            _, up, labels, lengths = batch_for(cfg, k, j)
            rc, on = s.enqueue_activations(k, up, labels, lengths)
            log.append(("enq", k, rc, on))
        elif ev[0] == "step":
            rc, k, slot = s.server_step()
            log.append(("step", rc, k, slot))
    return s, log


def replay_oracle(cfg, events, theta0=None, max_steps=None):
    """The same events through the oracle (fp64).  Slot indices come from the
    oracle's own scheduler."""
    theta = W.init_params(cfg) if theta0 is None else theta0
    srv = O.Server(cfg["ops"], cfg["K"], cfg["omega"], cfg["depth"], theta, cfg["lr"],
                   cfg["momentum"])
    log, nb, steps = [], {}, 0
    for ev in events:
        if ev[0] == "enq":
            k = ev[1]
            j = nb.get(k, 0)
            nb[k] = j + 1
            x, _, labels, lengths = batch_for(cfg, k, j)
            rc, slot = srv.enqueue(k, x, labels, lengths)
            log.append(("enq", k, rc, int(srv.sched.on[k])))
        elif ev[0] == "step":
            if max_steps is not None and steps >= max_steps:
                break
            rc, k, slot = srv.step()
            steps += rc == O.OK
            log.append(("step", rc, k, slot))
    return srv, log


def normwise(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))
