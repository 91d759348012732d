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


def test_result_line_carries_every_workload():
    """One JSON line: the headline at the top level, and every workload of the
    run (the three training workloads and the two merge microbenchmarks)
    under roofline/cpu_baseline/e2e "configs", each roofline with its bound,
    rate, peak and fraction; the config dict is the one the reference arm
    prints."""
    import argparse
    import synth
    w = synth.CFG2
    roof = bench.roofline_of("fused_round", 0.1, 1.0, {"fused_round": 7.4e9}, {"fused_round": 41.9e6}, HBM, TF,
                             "measured", workload=w.name)
    e2e = {"value": 4e7, "unit": "samples/s", "h2d_bytes_per_step": 1, "d2h_bytes_per_step": 64}
    side = {}
    for sw, kern in ((synth.CFG1, "softreg_round"), (synth.CFG3, "gemm_dw_sgd")):
        side[sw.name] = {"value": 1e6, "roofline": {"kernel": kern, "bound": "hbm", "achieved": 1.0, "peak": HBM,
                                                    "unit": "GB/s", "frac": 1.0 / HBM, "traffic": None},
                         "e2e": dict(e2e)}
    merge = {m.name: {"GB/s": 6700.0, "frac": 1.0, "ms_median": 1.0, "peak": HBM, "traffic": 6.7e9}
             for m in (synth.CFG4, synth.CFG5)}
    res = {"value": 4e7, "ms_per_step": 0.11, "roofline": roof, "e2e": dict(e2e), "gpu_launches": 80,
           "clocks": None, "merge": merge, "kernels": {}, "samples_per_round": 4544, "T_star": 4340,
           "tau": [5] * 16, "workloads": side}
    cpu = {"value": 2e4, "unit": "samples/s", "cores": 16, "kind": "oracle", "sample": "6 rounds"}
    cpus = {n: dict(cpu) for n in (synth.CFG1.name, synth.CFG3.name, synth.CFG4.name, synth.CFG5.name)}
    args = argparse.Namespace(steps=20, warmup=5)
    line = bench.result_line(args, 1, w, res, cpu, cpus)
    names = {c.name for c in (synth.CFG1, synth.CFG2, synth.CFG3, synth.CFG4, synth.CFG5)}
    assert set(line["roofline"]["configs"]) == names
    assert set(line["cpu_baseline"]["configs"]) == names
    assert set(line["e2e"]["configs"]) == {synth.CFG1.name, synth.CFG2.name, synth.CFG3.name}
    for r in line["roofline"]["configs"].values():
        assert {"bound", "achieved", "peak", "unit", "frac"} <= set(r)
    assert line["roofline"]["configs"][w.name]["tensor_frac"] == pytest.approx(7.4e9 / 1e-4 / 1e12 / TF)
    assert line["config"] == bench.workload_config(w)
    assert "dims" not in line["config"]
