"""The benchmark's multi-rank plumbing on CPU (gloo, world size 2): the
server step does not shard, so N GPUs run N independent replicas and the
ranks only exchange the timing (max over ranks) and the work done (sum over
ranks).  Checked here with two processes and the gloo backend."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.multiprocessing as mp  # noqa: E402


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    import torch.distributed as dist
    w, r, local = bench.dist_setup(0)            # no GPU: gloo
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(w)
    ms = 10.0 + rank                              # a slower rank sets the job's time
    samples = 64.0 * (rank + 1)
    out[rank] = (bench.max_over_ranks(w, ms, "cpu"), bench.sum_over_ranks(w, samples, "cpu"))
    bench.barrier(w)
    dist.destroy_process_group()


def test_two_replicas_reduce_time_by_max_and_work_by_sum():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(worker, args=(world, free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1] == (11.0, 64.0 + 128.0)


def test_single_rank_needs_no_process_group(monkeypatch):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.dist_setup(1) == (1, 0, 0)
    assert bench.max_over_ranks(1, 3.5, "cpu") == 3.5
    assert bench.sum_over_ranks(1, 7.0, "cpu") == 7.0
