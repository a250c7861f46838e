"""FedAsync aggregation on the GPU (fo_aggregate / fo_axpby_async) against
the oracle (Algorithm 4, aggregation branch), fp64 reference, 1e-6
relative.  Elementwise bound derived from the fp32 arithmetic of
fmaf(alpha, l - g, g): |err| <= 2 ulp of (|g| + |l|), i.e. 1e-6 (|g| + |l|)."""
import numpy as np
import pytest
import torch

from harness import normwise
from oracle import fo_oracle as O
from paper_2504_13850_gb300 import api, build
from paper_2504_13850_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    api.lib()


def agg(s, g, l, k, version):
    """fo_aggregate ordered after the caller's torch work on its inputs and
    completed before the caller reads the result (the aggregation runs on the
    server's own stream)."""
    torch.cuda.synchronize()
    out = s.aggregate(g, l, k, version)
    s.synchronize()
    return out


def tiny_server(max_delay=2**31 - 1):
    return api.Server.from_config(W.CONFIGS["tiny"], max_delay=max_delay)


def check(gpu, ref, g_old, l):
    gpu = np.asarray(gpu, np.float64)
    assert normwise(gpu, ref) <= 1e-6
    bound = 1e-6 * (np.abs(g_old) + np.abs(l)) + 1e-30
    assert np.all(np.abs(gpu - ref) <= bound)


def test_tiny_config_each_device_once_is_running_mean():
    """Each device's model once, all trained from version 0: per step the GPU
    result is checked elementwise against Algorithm 4 applied to the GPU's own
    previous global (teacher forced), and the whole chain normwise against the
    oracle's chain and the closed form (running mean of the locals)."""
    cfg = W.CONFIGS["tiny"]
    n = cfg["agg_params"]
    s = tiny_server()
    g0 = W.global_model(n, cfg["seed"])
    gd = torch.tensor(g0, device="cuda")
    chain = O.Aggregator(cfg["K"], 2**31 - 1)
    g_chain = g0.astype(np.float64)
    locs = []
    for k in range(cfg["K"]):
        l = W.device_model(n, cfg["seed"], k, 0)
        locs.append(l)
        g_before = gd.cpu().numpy().astype(np.float64)
        step = O.Aggregator(cfg["K"], 2**31 - 1)
        step.t = k
        _, ref = step.aggregate(g_before, l, 0)
        rc, t = agg(s, gd, torch.tensor(l, device="cuda"), k, 0)
        assert rc == api.OK and t == k + 1
        check(gd.cpu().numpy(), ref, g_before, l)
        _, g_chain = chain.aggregate(g_chain, l, 0)
        assert normwise(gd.cpu().numpy(), g_chain) <= 1e-6
        assert normwise(gd.cpu().numpy(), np.mean(np.array(locs, np.float64), 0)) <= 1e-6
    assert s.version() == (4, 1)


@pytest.mark.parametrize("n,offset", [(1, 0), (7, 1), (8, 0), (1000, 3), (1_000_003, 0), (4_194_304, 2)])
def test_ragged_sizes_and_unaligned_pointers(n, offset):
    r = np.random.default_rng(n)
    g = r.standard_normal(n + offset).astype(np.float32)
    l = r.standard_normal(n + offset).astype(np.float32)
    gd = torch.tensor(g, device="cuda")
    ld = torch.tensor(l, device="cuda")
    s = tiny_server()
    # advance t so that alpha is not 1: three identity aggregations first
    for _ in range(3):
        agg(s, gd[offset:], gd[offset:].clone(), 0, s.version()[0])
    g_mid = gd.cpu().numpy()[offset:].astype(np.float64)
    rc, t = agg(s, gd[offset:], ld[offset:], 1, 1)        # t = 3, t_k = 1 -> alpha = 1/3
    assert rc == api.OK and t == 4
    ref = (1 / 3) * l[offset:].astype(np.float64) + (1 - 1 / 3) * g_mid
    check(gd.cpu().numpy()[offset:], ref, g_mid, l[offset:])
    assert np.array_equal(gd.cpu().numpy()[:offset], g[:offset])   # nothing before the view


def test_identity_is_bit_exact():
    r = np.random.default_rng(1)
    g = torch.tensor(r.standard_normal(123_457).astype(np.float32), device="cuda")
    before = g.clone()
    s = tiny_server()
    for v in range(5):
        agg(s, g, g.clone(), 0, max(0, s.version()[0] - v % 3))
    assert torch.equal(g, before)


def test_stale_and_invalid_versions():
    s = tiny_server(max_delay=2)
    g = torch.zeros(1000, device="cuda")
    l = torch.ones(1000, device="cuda")
    for _ in range(4):
        agg(s, g, l, 0, s.version()[0])
    t = s.version()[0]
    before = g.clone()
    rc, nv = agg(s, g, l * 5, 1, t - 3)
    assert rc == api.STALE and nv == t and s.version()[0] == t
    torch.cuda.synchronize()
    assert torch.equal(g, before)
    assert agg(s, g, l, 1, t + 1)[0] == api.ERR_ARG
    assert agg(s, g, l, 1, -1)[0] == api.ERR_ARG
    assert agg(s, g, l, 99, t)[0] == api.ERR_ARG


@pytest.mark.parametrize("n", [16_000_000, 200_000_000])
def test_large_models_sampled(n):
    """Full sweep sizes: exact check on a sample of indices, plus the weights
    summing to one (a constant model stays constant)."""
    gen = torch.Generator(device="cuda").manual_seed(n)
    g = torch.randn(n, device="cuda", generator=gen) * 0.05
    l = torch.randn(n, device="cuda", generator=gen) * 0.05
    idx = torch.randint(0, n, (100_000,), device="cuda", generator=gen)
    g_s = g[idx].double().cpu().numpy()
    l_s = l[idx].double().cpu().numpy()
    api.axpby_async(g, l, 0.25)
    torch.cuda.synchronize()
    ref = 0.25 * l_s + 0.75 * g_s
    check(g[idx].cpu().numpy(), ref, g_s, l_s)
    c = torch.full((n,), 3.25, device="cuda")
    api.axpby_async(c, c.clone(), 0.125)
    torch.cuda.synchronize()
    assert bool((c == 3.25).all())
    del g, l, c
    torch.cuda.empty_cache()
