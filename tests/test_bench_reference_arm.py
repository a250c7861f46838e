"""The benchmark's reference arm on CPU: `bench.py --impl reference` times
the oracle on the host cores and prints one JSON line with the same metric,
unit and direction as the GPU arm, plus its `cpu_baseline` and a host-only
`e2e` block.  Under torchrun with two ranks only rank 0 prints; both exit 0.
Run on the smallest workload (4 devices, batch 16) so the oracle finishes in
seconds."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ARGS = ["--impl", "reference", "--workload", "tiny", "--steps", "2", "--warmup", "1"]


def json_lines(out):
    return [json.loads(l) for l in out.splitlines() if l.startswith("{")]


def env():
    e = dict(os.environ)
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK", "MASTER_ADDR", "MASTER_PORT"):
        e.pop(k, None)
    e["CUDA_VISIBLE_DEVICES"] = ""
    return e


def check_line(d, n_gpus):
    sys.path.insert(0, ROOT)
    import bench
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["higher_is_better"] is True and d["scaling"] == "weak"
    assert d["n_gpus"] == n_gpus and d["steps"] == 2 and d["warmup"] == 1
    assert d["value"] > 0 and d["ms_per_step"] > 0
    assert d["vs_baseline"] is None and d["dtype"] == "f64" and d["data"] == "synthetic"
    assert "workload" in d["config"] and "sample" in d["config"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["unit"] == d["unit"]
    assert cb["cores"] >= 1 and cb["sample"]
    e2e = d["e2e"]
    assert e2e == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, "bench.py"] + ARGS, cwd=ROOT, env=env(), capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = json_lines(r.stdout)
    assert len(lines) == 1
    check_line(lines[0], 1)


def test_reference_arm_under_two_ranks_prints_once():
    pytest.importorskip("torch.distributed.run")
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), "bench.py", "--gpus", "2"] + ARGS
    r = subprocess.run(cmd, cwd=ROOT, env=env(), capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = json_lines(r.stdout)
    assert len(lines) == 1
    check_line(lines[0], 2)


def test_cpu_baseline_sample_runs_until_its_time_budget():
    """The GPU arm's `cpu_baseline` times whole oracle steps until about the
    requested seconds of CPU work have run (at least two steps)."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2504_13850_gb300 import workloads as W
    cfg = W.CONFIGS["tiny"]
    v, n, dt = bench.oracle_sample(cfg, cfg["batch"], seconds=0.3)
    assert n >= 2 and dt >= 0.3 and v == pytest.approx(n * cfg["batch"] / dt)
    v, n, dt = bench.oracle_sample(cfg, 4, seconds=0.0)
    assert n == 2 and v > 0
    v, n, dt = bench.oracle_sample(cfg, 4, seconds=1e9, max_steps=3)
    assert n == 3
