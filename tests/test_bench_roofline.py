"""bench.py's roofline bookkeeping on CPU: which roof binds, the achieved
rate over the measured launch time, and the ncu traffic attached to it."""
import pytest

import bench

HBM, TF = 6685.8, 1741.7   # GB/s, TFLOP/s (the measured peaks the bench reads)


def test_hbm_bound_kernel():
    # 1 GB and 1 GFLOP per launch: 0.15 ms on HBM against 0.6 us on the tensor pipe
    r = bench.roofline_of("merge", 0.2, 1.0, {"merge": 1e9}, {"merge": 1e9}, HBM, TF, "measured")
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(1e9 / 0.2e-3 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / HBM)
    assert r["traffic"] is None


def test_tensor_bound_kernel_per_launch():
    # 22 launches per round: the per-launch work is the round's over the launches
    flops, bytes_ = {"gemm_fwd": 22 * 2e12}, {"gemm_fwd": 22 * 1e8}
    r = bench.roofline_of("gemm_fwd", 2.0, 22.0, flops, bytes_, HBM, TF, "measured")
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["flops_per_launch"] == pytest.approx(2e12)
    assert r["achieved"] == pytest.approx(2e12 / 2e-3 / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / TF)


def test_round_kernel_carries_its_ncu_traffic():
    key = ("fused_round", "mlp-784-512-10-W16")
    assert key in bench.NCU_TRAFFIC
    r = bench.roofline_of("fused_round", 0.1, 1.0, {"fused_round": 7.4e9}, {"fused_round": 41.9e6}, HBM, TF,
                          "measured", workload="mlp-784-512-10-W16")
    assert r["bound"] == "hbm"
    assert r["traffic"] == bench.NCU_TRAFFIC[key][0]
    assert r["traffic_source"].startswith("profiles/")


def test_kernel_without_algorithmic_work_has_no_fraction():
    r = bench.roofline_of("round_bookkeeping", 0.01, 1.0, {}, {}, HBM, TF, "measured")
    assert r["frac"] is None and r["achieved"] is None
