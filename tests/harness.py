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


def param_slices(ops):
    out, off = [], 0
    for i, name, shape in O.param_shapes(ops):
        n = int(np.prod(shape))
        out.append((f"{i}:{ops[i]['kind']}.{name}", slice(off, off + n)))
        off += n
    return out


def teacher_forced(cfg, events, max_steps=None):
    """GPU and oracle in lockstep: before every step the oracle takes the
    GPU's theta and momentum, then both run the same scheduled batch.  Two
    oracle readings run side by side: the exact fp64 definition, and the
    bf16-storage reading (the kernel's precision for every stored tensor, so
    that ReLU / max-pool decisions are taken alike).  Returns per-step records
    with the loss, parameter and per-tensor gradient errors against each
    (gradient recovered exactly as g = v_new - mu v_old)."""
    from paper_2504_13850_gb300 import api
    s = api.Server.from_config(cfg)
    theta0 = W.init_params(cfg)
    s.set_params(theta0)
    storage = "bf16" if cfg["dtype"] == W.BF16 else None
    mk = lambda st: O.Server(cfg["ops"], cfg["K"], cfg["omega"], cfg["depth"], theta0, cfg["lr"],
                             cfg["momentum"], storage=st)
    o, ob = mk(None), mk(storage)
    mu = cfg["momentum"]
    nb, recs, steps = {}, [], 0
    slices = param_slices(cfg["ops"])
    for ev in events:
        if ev[0] == "enq":
            k = ev[1]
            j = nb.get(k, 0)
            nb[k] = j + 1
            x, up, labels, lengths = batch_for(cfg, k, j)
            g_out = s.enqueue_activations(k, up, labels, lengths)
            o_rc, _ = o.enqueue(k, x, labels, lengths)
            ob.enqueue(k, x, labels, lengths)
            assert (g_out[0], g_out[1]) == (o_rc, int(o.sched.on[k]))
            continue
        if max_steps is not None and steps >= max_steps:
            break
        th0 = s.get_params().astype(np.float64)
        v0 = s.get_momentum().astype(np.float64)
        for srv in (o, ob):
            srv.theta, srv.v = th0.copy(), v0.copy()
        g_rc, gk, gslot = s.server_step()
        o_rc, ok, oslot = o.step()
        ob.step()
        assert (g_rc, gk, gslot) == (o_rc, ok, oslot)
        if g_rc != api.OK:
            continue
        loss = float(s.read_losses(steps, 1)[0])
        th1 = s.get_params().astype(np.float64)
        v1 = s.get_momentum().astype(np.float64)
        recs.append(step_record(steps, loss, th0, v0, th1, v1, o, ob, mu, slices))
        steps += 1
    return s, o, recs


def step_record(step, loss, th0, v0, th1, v1, o, ob, mu, slices):
    """One teacher-forced step's errors.  `th1, v1, loss` are the path under
    test, `o` the exact oracle and `ob` its bf16-storage reading, both
    stepped from (th0, v0).  The gradient is recovered exactly from the
    momentum, g = v1 - mu v0.  "reading" records how far the bf16-storage
    reading's own gradient lies from the exact one (per tensor and whole):
    the distance that storing the path's tensors in bf16 moves the
    definition by, which sets the allowance for decision flips."""
    g_gpu = v1 - mu * v0
    g_ex = o.v - mu * v0
    g_rd = ob.v - mu * v0
    rec = {"step": step, "loss": loss,
           "g_norm": float(np.linalg.norm(g_ex)), "v_norm": float(np.linalg.norm(o.v)),
           "reading": {"whole": normwise(g_rd, g_ex),
                       "tensor": {n: normwise(g_rd[sl], g_ex[sl]) for n, sl in slices}}}
    for tag, srv, g_ref in (("exact", o, g_ex), ("stored", ob, g_rd)):
        rec[tag] = {
            "loss": srv.losses[-1],
            "param_err": normwise(th1, srv.theta),
            "update_err": normwise(th1 - th0, srv.theta - th0),
            "grad_err": normwise(g_gpu, g_ref),
            "tensor_grad_err": {n: normwise(g_gpu[sl], g_ref[sl]) for n, sl in slices},
        }
    return rec
