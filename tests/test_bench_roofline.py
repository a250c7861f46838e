"""The roofline arithmetic of bench.py, on made-up kernel times: the
dominant class is the one with the largest total time; `achieved` is its
algorithmic FLOPs (or bytes) over its event time, which is the FLOPs per
launch over the average launch time; `frac` divides by the burst bf16 peak
(or the copy bandwidth for a class with no FLOPs), `frac_sustained` by the
sustained one; the whole step's tensor share divides the step's FLOPs by the
step time."""
import math

import bench

PK = {"hbm_gbs": 6000.0, "bf16_tflops": 2000.0, "bf16_tflops_sustained": 1600.0}


def test_dominant_contraction_class():
    # name: (launches, total ms, total FLOPs, total bytes)
    kt = {"tc_linear_fwd": (16, 0.20, 16 * 6.4e9, 0.0),
          "tc_linear_wgrad": (16, 0.15, 16 * 6.4e9, 0.0),
          "sgd_momentum": (7, 0.05, 0.0, 2.8e8)}
    r = bench.roofline_of(kt, PK, "measured", "no-such-workload")
    assert r["kernel"] == "tc_linear_fwd" and r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    per_launch = 6.4e9 / (0.20 / 16 / 1e3) / 1e12          # FLOPs per launch / mean launch time
    assert math.isclose(r["achieved"], round(per_launch, 2))
    assert math.isclose(r["frac"], round(per_launch / 2000.0, 4))
    assert math.isclose(r["frac_sustained"], round(per_launch / 1600.0, 4))
    assert r["peak"] == 2000.0 and r["launches"] == 16 and r["traffic"] is None


def test_dominant_memory_class():
    kt = {"sgd_momentum": (7, 0.30, 0.0, 1.2e9), "tc_linear_fwd": (16, 0.10, 1e11, 0.0)}
    r = bench.roofline_of(kt, PK, "measured", "no-such-workload")
    assert r["kernel"] == "sgd_momentum" and r["bound"] == "hbm" and r["unit"] == "GB/s"
    gbs = 1.2e9 / (0.30 / 1e3) / 1e9
    assert math.isclose(r["achieved"], round(gbs, 1)) and math.isclose(r["frac"], round(gbs / 6000.0, 4))


def test_kernels_table_and_step_share():
    kt = {"a": (4, 0.5, 2e12, 0.0), "b": (2, 1.0, 0.0, 3e9)}
    t = bench.kernels_table(kt)
    assert list(t) == ["b", "a"]                              # by total time
    assert t["a"]["tflops"] == round(2e12 / 0.5e-3 / 1e12, 1) and t["a"]["gbs"] is None
    assert t["b"]["gbs"] == round(3e9 / 1e-3 / 1e9, 1) and t["b"]["tflops"] is None
    flops, burst, sustained = bench.step_fracs(kt, 10, 0.25, PK)   # 10 profiled steps of 0.25 ms
    assert math.isclose(flops, 2e11)
    assert math.isclose(burst, 2e11 / 0.25e-3 / 1e12 / 2000.0)
    assert math.isclose(sustained, 2e11 / 0.25e-3 / 1e12 / 1600.0)
