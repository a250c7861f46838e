"""Task-scheduler balance study (the paper's comparison of its counter-based
Task Scheduler with a FIFO scheduler, Sec. 4 'Task scheduling mechanisms'):
replays a seeded upload trace through the library's host scheduler
(fo_sched_*) under both policies and reports how evenly the server's
training iterations are spread over the devices."""
import numpy as np

from . import api
from . import workloads as W


def gini(x):
    """Gini coefficient of non-negative values (0 = all equal)."""
    x = np.asarray(x, np.float64)
    if x.sum() == 0:
        return 0.0
    return float(np.abs(x[:, None] - x[None, :]).sum() / (2.0 * len(x) * x.sum()))


def consumption(policy, cfg, uploads, seed, uploads_per_step=2):
    """Per-device count of server iterations fed by each device when the
    devices upload as the config's Poisson processes and the server takes
    one batch per `uploads_per_step` uploads; refused uploads (flow control)
    are dropped."""
    s = api.Scheduler(cfg["K"], cfg["omega"], cfg["depth"], policy)
    for i, k in enumerate(W.arrival_order(cfg["rates"], uploads, seed)):
        s.put(k)
        if i % uploads_per_step == uploads_per_step - 1:
            s.get()
    return np.asarray(s.counters(), np.int64)


def scheduler_balance(name="scale", uploads=6000):
    """Balance of counter-based vs FIFO scheduling on a workload's trace."""
    cfg = W.CONFIGS[name]
    out = {"trace": f"{name}: {cfg['K']} devices, omega {cfg['omega']}, depth {cfg['depth']}, {uploads} "
                    f"Poisson uploads (seed {cfg['seed']}), one server iteration per two uploads"}
    for label, policy in (("counter", api.SCHED_COUNTER), ("fifo", api.SCHED_FIFO)):
        c = consumption(policy, cfg, uploads, cfg["seed"])
        served = c[c > 0]
        out[label] = {"gini": round(gini(c), 4), "served_devices": int(len(served)),
                      "max_minus_min_served": int(served.max() - served.min()) if len(served) else 0,
                      "max_share": round(float(c.max() / c.sum()), 4)}
    return out
