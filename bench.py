#!/usr/bin/env python
"""Benchmark of the FedOptima server-side hot path on GB300.

One step = the whole hot path for one uploaded batch: the Task Scheduler
serves the device with the smallest consumption counter (Algorithm 3), the
server trains M_s on that batch (forward, softmax cross-entropy, backward,
SGD-momentum: Algorithm 4, training branch), the device whose sender was
turned on uploads its next batch into the freed HBM slot (Algorithm 2 with
the flow control of Sec. 3.4.1), and one device-side model is aggregated
FedAsync-style (Algorithm 4, aggregation branch).

Workload: the VGG-style server part (10 devices, bf16 activations
[64,128,16,16], 8,625,162 parameters; device model 1,000,000 fp32
parameters), with synthetic seeded inputs.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

For N > 1 (torchrun, one rank per GPU) every rank runs an independent
replica of the server: the server step is one sequential SGD chain and does
not shard, so the ranks exchange nothing but the timing.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "server-side train samples/s at 1 GB300; % bf16 tensor peak; aggregation HBM GB/s"
UNIT = "samples/s"
WORKLOAD = "vgg"
WORKLOAD_DESC = ("VGG-style server part: 10 devices, bf16 activations [64,128,16,16] = ReLU(N(0,1)), "
                 "2x(conv3x3 ->256, ReLU), maxpool2, 2x(conv3x3 ->512, ReLU), maxpool2, FC 8192->512->10, "
                 "softmax-CE, SGD lr 0.01 momentum 0.9; 1M-param device model aggregated each step")
OTHER_DESC = {
    "resnet": "ResNet-18 stages 3-4 server part: 20 devices, bf16 activations [128,128,16,16] = ReLU(N(0,1)), "
              "basic blocks 128->256 (stride 2), 256, 256->512 (stride 2), 512 with folded batch norms, avgpool, "
              "FC 512->100, softmax-CE, SGD lr 0.01 momentum 0.9",
    "transformer": "Transformer encoder server part: 16 devices, bf16 activations [32,128,512] ~ N(0,1) with "
                   "lengths 32..128, 4 pre-LN blocks (8 heads, FFN 2048, GELU), masked mean-pool, FC 512->2, "
                   "softmax-CE, SGD lr 0.01 momentum 0.9",
    "scale": "ResNet-18 stages 3-4 server part with 100 devices (Zipf rates), bf16 activations [64,128,16,16], "
             "omega 400, FC 512->100, softmax-CE, SGD lr 0.01 momentum 0.9",
    "mobilenet": "MobileNetV3-Large server part: 10 devices, bf16 activations [64,112,4,4] = ReLU(N(0,1)), "
                 "BNECK-5-160 x3 (first stride 2; 1x1 expand, 5x5 depthwise, squeeze-and-excite, 1x1 project, "
                 "hard swish), CONV-1-960, avgpool, FC 960->1280, hard swish, FC 1280->200, softmax-CE, "
                 "SGD lr 0.01 momentum 0.9",
}


def workload_desc(name):
    return WORKLOAD_DESC if name == WORKLOAD else OTHER_DESC.get(name, name)


FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=WORKLOAD)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-agg-sweep", action="store_true")
    p.add_argument("--no-live", action="store_true",
                   help="skip the live pipeline (devices' networks training on the same GPU)")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.proc:
            return None
        self.f.flush()
        with open(self.f.name) as fh:
            rows = [r.split(",") for r in fh.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, r[5:9]):
                if v.strip() == "Active":
                    reasons.add(n)
        if not sm:
            return None
        loaded = [v for v in sm if v >= 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if n_gpus > 0 else "gloo"
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, value, device):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(world, value, device):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def oracle_samples_per_s(cfg, n_steps, batch):
    """The oracle as it stands, timed on this host's cores: n_steps server
    steps at `batch` samples each (a bounded sample of the workload)."""
    import numpy as np
    from oracle import fo_oracle as O
    from paper_2504_13850_gb300 import workloads as W
    theta = W.init_params(cfg).astype(np.float64)
    v = np.zeros_like(theta)
    t0 = time.perf_counter()
    for j in range(n_steps):
        x, _, y, ln = W.device_batch(cfg, j % cfg["K"], j, batch=batch)
        _, theta, v, _ = O.server_step(cfg["ops"], theta, v, x, y, ln, cfg["lr"], cfg["momentum"])
    dt = time.perf_counter() - t0
    return n_steps * batch / dt, dt


def oracle_sample(cfg, batch, seconds=12.0, min_steps=2, max_steps=50):
    """The oracle timed over whole server steps at `batch` samples each,
    until about `seconds` of CPU work have run (at least `min_steps`).
    Returns (samples/s, steps, elapsed seconds)."""
    import numpy as np
    from oracle import fo_oracle as O
    from paper_2504_13850_gb300 import workloads as W
    theta = W.init_params(cfg).astype(np.float64)
    v = np.zeros_like(theta)
    dt, j = 0.0, 0
    while j < max_steps and (j < min_steps or dt < seconds):
        x, _, y, ln = W.device_batch(cfg, j % cfg["K"], j, batch=batch)
        t0 = time.perf_counter()
        _, theta, v, _ = O.server_step(cfg["ops"], theta, v, x, y, ln, cfg["lr"], cfg["momentum"])
        dt += time.perf_counter() - t0
        j += 1
    return j * batch / dt, j, dt


def run_reference(args):
    world, rank, _ = dist_setup(0)
    if rank != 0:
        return
    from paper_2504_13850_gb300 import workloads as W
    cfg = W.CONFIGS[args.workload]
    # Each step runs the oracle on a bounded sample of the step's batch, sized
    # so that warm-up plus timed steps take about 90 s of CPU work.
    probe = 4
    _, t_probe = oracle_samples_per_s(cfg, 1, probe)
    per_sample = t_probe / probe
    batch = int(max(1, min(cfg["batch"], 90.0 / (per_sample * (args.steps + args.warmup)))))
    oracle_samples_per_s(cfg, max(1, args.warmup), batch)
    v, dt = oracle_samples_per_s(cfg, args.steps, batch)
    cores = os.cpu_count()
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": workload_desc(args.workload), "sample": f"{batch} of the {cfg['batch']} samples per step"},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{args.steps} oracle server steps at batch {batch} (numpy fp64, BLAS threads = cores)"},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args):
    import numpy as np
    import torch

    from paper_2504_13850_gb300 import api, build
    from paper_2504_13850_gb300 import workloads as W

    world, rank, local = dist_setup(args.gpus)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    build.build()
    api.lib()
    cfg = W.CONFIGS[args.workload]
    B, (H, Wd, C) = cfg["batch"], cfg["in_hwc"]
    srv = api.Server.from_config(cfg)
    srv.set_params(W.init_params(cfg))
    stream = torch.cuda.ExternalStream(srv.stream(), device=dev)

    # Resident inputs: a pool of uploaded batches and device models in HBM.
    P = 8
    pool = []
    for j in range(P):
        x, bits, labels, lengths = W.device_batch(cfg, j % cfg["K"], 10_000 + j)
        up = bits.view(np.int16) if bits is not None else x
        pool.append((torch.from_numpy(np.ascontiguousarray(up)).to(dev),
                     torch.from_numpy(labels).to(dev),
                     None if lengths is None else torch.from_numpy(lengths).to(dev)))
    n_model = cfg["agg_params"]
    g_model = torch.from_numpy(W.global_model(n_model, cfg["seed"])).to(dev)
    locals_ = [torch.from_numpy(W.device_model(n_model, cfg["seed"], j, 0)).to(dev) for j in range(2)]
    order = W.arrival_order(cfg["rates"], 200_000, cfg["seed"] + rank)
    pos = [0]

    def next_uploader():
        on = srv.sender_status()
        for _ in range(100_000):
            k = order[pos[0] % len(order)]
            pos[0] += 1
            if on[k]:
                return k
        return int(np.argmax(on))

    # Backlog: every device fills its ring (the steady state of a loaded server).
    for r in range(cfg["depth"]):
        for k in range(cfg["K"]):
            a, lb, ln = pool[(r * cfg["K"] + k) % P]
            srv.enqueue_activations(k, a, lb, ln)

    it = [0]
    done = [0]                      # server steps run so far (loss ring index)

    def step(host=None):
        i = it[0]
        it[0] += 1
        rc, k, slot = srv.server_step()
        assert rc == api.OK, rc
        done[0] += 1
        u = next_uploader()
        if host is None:
            a, lb, ln = pool[i % P]
            rc, _ = srv.enqueue_activations(u, a, lb, ln)
            local = locals_[i % 2]
        else:
            a, lb, ln = host["batches"][i % len(host["batches"])]
            rc, _ = srv.enqueue_activations(u, a, lb, ln)
            # the device model comes up on a copy stream into one of two
            # staging buffers, after the aggregation that last read it
            b = i % 2
            cs = host["copy"]
            cs.wait_event(host["read"][b])
            with torch.cuda.stream(cs):
                host["stage"][b].copy_(host["models"][b], non_blocking=True)
                host["landed"][b].record(cs)
            stream.wait_event(host["landed"][b])
            local = host["stage"][b]
        assert rc == api.OK, rc
        t, _ = srv.version()
        rc, _ = srv.aggregate(g_model, local, u, max(0, t - 3))
        assert rc == api.OK, rc
        if host is not None:
            host["read"][i % 2].record(stream)
            # every step's loss comes back to the host; step i's is read while
            # step i + 1 runs (fo_read_losses waits for that step only)
            if done[0] >= 2:
                host["loss"] = srv.read_losses(done[0] - 2, 1)

    # ---------------- device-resident timed region
    for _ in range(args.warmup):
        step()
    srv.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        barrier(world)
        torch.cuda.synchronize()
        k0 = srv.kernels_launched()
        ev0.record(stream)
        w0 = time.perf_counter()
        for _ in range(args.steps):
            step()
        ev1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - w0
        barrier(world)
    srv.check_error()
    ms_dev = ev0.elapsed_time(ev1)
    launches = srv.kernels_launched() - k0
    ms_max = max_over_ranks(world, ms_dev, dev)
    samples = sum_over_ranks(world, float(args.steps * B), dev)
    value = samples / (ms_max / 1e3)

    # ---------------- per-kernel times: the same steps again, each launch
    # bracketed by CUDA events on the compute stream (a separate timed region,
    # so the events do not perturb the value above)
    n_prof = min(args.steps, 200)
    srv.profile(True)
    srv.profile_reset()
    torch.cuda.synchronize()
    for _ in range(n_prof):
        step()
    ktimes = srv.kernel_times()
    srv.profile(False)
    srv.check_error()

    # ---------------- end to end through the C ABI from pinned host memory
    e2e = None
    if not args.no_e2e:
        host = {"batches": [], "models": [], "stage": [torch.empty(n_model, device=dev) for _ in range(2)],
                "copy": torch.cuda.Stream(device=dev), "landed": [torch.cuda.Event() for _ in range(2)],
                "read": [torch.cuda.Event() for _ in range(2)]}
        for a, lb, ln in pool[:4]:
            host["batches"].append((a.cpu().pin_memory(), lb.cpu().pin_memory(),
                                    None if ln is None else ln.cpu().pin_memory()))
        host["models"] = [m.cpu().pin_memory() for m in locals_]
        h2d = (host["batches"][0][0].numel() * host["batches"][0][0].element_size() + 4 * B
               + (4 * B if cfg["seq"] else 0) + 4 * n_model)
        srv.synchronize()
        for _ in range(max(1, args.warmup)):
            step(host)
        n_e2e = min(args.steps, 100)
        barrier(world)
        torch.cuda.synchronize()
        ev0.record(stream)
        for _ in range(n_e2e):
            step(host)
        host["loss"] = srv.read_losses(done[0] - 1, 1)   # the last step's loss, inside the timed region
        ev1.record(stream)
        torch.cuda.synchronize()
        barrier(world)
        ms_e = max_over_ranks(world, ev0.elapsed_time(ev1), dev)
        e2e = {"value": sum_over_ranks(world, float(n_e2e * B), dev) / (ms_e / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": 4}

    # ---------------- aggregation bandwidth sweep (standalone FedAsync update)
    agg = None
    if rank == 0 and not args.no_agg_sweep:
        n = 200_000_000
        try:
            ga = torch.randn(n, device=dev) * 0.05
            la = torch.randn(n, device=dev) * 0.05
            pk, which = peaks()
            sweep = []
            for m in (1_000_000, 4_000_000, 16_000_000, 64_000_000, n):
                g_m, l_m = ga[:m], la[:m]
                for _ in range(3):
                    api.axpby_async(g_m, l_m, 0.25, srv.stream())
                best = 1e30
                for _ in range(10):
                    ev0.record(stream)
                    api.axpby_async(g_m, l_m, 0.25, srv.stream())
                    ev1.record(stream)
                    torch.cuda.synchronize()
                    best = min(best, ev0.elapsed_time(ev1))
                # 12 bytes per parameter; below ~126 MB of traffic the vectors stay in L2
                sweep.append({"params": m, "gbs": round(12.0 * m / (best / 1e3) / 1e9, 1),
                              "l2_resident": 12 * m < 126 * 2**20})
            gbs = sweep[-1]["gbs"]
            agg = {"params": n, "gbs": gbs, "frac": round(gbs / pk["hbm_gbs"], 4),
                   "peak_gbs": pk["hbm_gbs"], "peak": which, "bytes_per_param": 12,
                   "sweep": sweep, "best_of": 10}
            del ga, la
            torch.cuda.empty_cache()
        except torch.cuda.OutOfMemoryError:
            agg = None

    if rank != 0:
        return
    pk, which = peaks()
    # dominant kernel class of the step, by total time
    dom = max(ktimes.items(), key=lambda kv: kv[1][1])
    name, (nl, ms_k, fl_k, by_k) = dom
    if fl_k > 0:
        peak = pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
        achieved = fl_k / (ms_k / 1e3) / 1e12
        roof = {"kernel": name, "bound": "tensor", "achieved": round(achieved, 2), "peak": peak,
                "unit": "TFLOP/s", "frac": round(achieved / peak, 4), "traffic": traffic_for(name),
                "peak_kind": f"{which} sustained bf16", "launches": nl, "ms_total": round(ms_k, 3)}
    else:
        peak = pk["hbm_gbs"]
        achieved = by_k / (ms_k / 1e3) / 1e9
        roof = {"kernel": name, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": traffic_for(name),
                "peak_kind": f"{which} copy", "launches": nl, "ms_total": round(ms_k, 3)}
    step_flops = sum(v[2] for v in ktimes.values()) / n_prof
    step_ms = ms_dev / args.steps
    tensor_frac = step_flops / (step_ms / 1e3) / 1e12 / pk.get("bf16_tflops_sustained", pk["bf16_tflops"])
    tensor_frac_burst = step_flops / (step_ms / 1e3) / 1e12 / pk["bf16_tflops"]
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        v_cpu, n_cpu, dt_cpu = oracle_sample(cfg, B)
        cpu = {"value": round(v_cpu, 3), "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"{n_cpu} oracle server steps at batch {B} ({dt_cpu:.1f} s, numpy fp64, BLAS threads = cores)"}
    from paper_2504_13850_gb300 import study
    sched = study.scheduler_balance("scale", uploads=6000)   # host-only: counter vs FIFO scheduling
    wsb = srv.device_bytes()
    live_line = None
    if rank == 0 and not args.no_live and args.workload == "vgg":
        # a second workload: the VGG-style split with every device's network
        # training on the same GPU and feeding the server (measured after the
        # timed region, so it does not perturb `value`)
        try:
            from paper_2504_13850_gb300 import live
            live_line = live.measure(events=400, warmup=40, agg_every=8)
        except Exception as e:   # reported, not fatal: the headline above stands alone
            live_line = {"error": f"{type(e).__name__}: {e}"}
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": workload_desc(args.workload), "global_batch": B * world, "devices": cfg["K"],
                   "omega": cfg["omega"], "parallelism": f"replicas{world}",
                   "l2": f"not flushed: each step touches the server's {wsb / 1e6:.0f} MB of parameters, "
                         f"momentum, gradients, activations and scratch, above the 126 MB L2"},
        "e2e": e2e,
        "gpu_launches": int(launches),
        "roofline": roof,
        "step_tensor_frac": round(tensor_frac, 4),
        "step_tensor_frac_burst": round(tensor_frac_burst, 4),
        "step_gflop": round(step_flops / 1e9, 2),
        "aggregation": agg,
        "scheduler_balance": sched,
        "live_pipeline": live_line,
        "cpu_baseline": cpu,
        "clocks": clk.summary(),
        "host_wall_ms_per_step": round(1e3 * wall / args.steps, 4),
        "kernels_profiled_steps": n_prof,
        "kernels": {k: {"launches": v[0], "ms": round(v[1], 3),
                        "tflops": round(v[2] / (v[1] / 1e3) / 1e12, 1) if v[2] and v[1] else None,
                        "gbs": round(v[3] / (v[1] / 1e3) / 1e9, 1) if v[3] and v[1] else None}
                    for k, v in sorted(ktimes.items(), key=lambda kv: -kv[1][1])},
    }
    print(json.dumps(line), flush=True)


def traffic_for(kernel):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if the
    kernel source has not changed since it was captured (else None)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(path):
        return None
    for line in open(path):
        f = line.split()
        if len(f) >= 3 and not line.startswith("#") and f[0] == kernel:
            src = os.path.join(ROOT, "paper_2504_13850_gb300", "csrc", f[1].split(":")[0])
            if os.path.exists(src):
                h = hashlib.sha1(open(src, "rb").read()).hexdigest()[:12]
                if h == f[1].split(":")[1]:
                    return float(f[2])
    return None


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
