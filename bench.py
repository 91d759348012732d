#!/usr/bin/env python
"""Benchmark of the Oscars hot path on one GB300 (or N independent replicas).

A step is one Oscars round of the 784-512-10 MLP workload with W=16 workers
(batch 64): every worker's tau_i local SGD steps (the schedule of Algorithm 1),
the push, the server merge and global update (Eq. 4) and the pull.  The
headline metric is simulated-worker samples per second (sum_i tau_i * B per
round).  The same JSON line carries the server-merge microbenchmarks (P=25.6M,
W=64 and P=340M, W=8) as GB/s and fraction of HBM bandwidth.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl oscars|reference]
  python bench.py --compare [--compare-configs cfg1,cfg2,cfg3]
  python bench.py --cnn [--steps K] [--warmup W]

--impl reference times the CPU oracle (the plain numpy restatement of the
method) on the same workload and metric.

--compare runs the paper's convergence comparison in simulated time instead:
Oscars rounds against BSP (one step per barrier) and local SGD with a fixed
period I (the median Oscars tau), each for the same simulated time, and
prints one JSON line per workload with the eval-loss curves and the ticks each
scheme needs to reach the loss BSP ends at.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

WORKLOAD = synth.CFG2
WORKLOADS = {w.name: w for w in (synth.CFG1, synth.CFG2, synth.CFG3)}
METRIC = "simulated-worker samples/s (Oscars rounds; merge GB/s alongside)"
UNIT = "samples/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="oscars", choices=["oscars", "reference"])
    ap.add_argument("--workload", default=WORKLOAD.name, choices=sorted(WORKLOADS),
                    help="MLP workload of the round benchmark (default: the 784-512-10 headline); the "
                         "server-merge microbenchmarks run with the headline only")
    ap.add_argument("--no-merge", action="store_true", help="skip the merge microbenchmarks")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--samples-per-worker", type=int, default=0,
                    help="shard rows per worker of the round workload (0: the workload's own; smaller for "
                         "ncu captures that must stay a few GB on the device)")
    ap.add_argument("--no-side", action="store_true",
                    help="skip the other training workloads (softmax regression, 3072-1024-1024-10 MLP)")
    ap.add_argument("--merge-reps", type=int, default=20)
    ap.add_argument("--only", choices=["all", "round", "merge"], default="all",
                    help="round: only the Oscars-round benchmark; merge: only the merge microbenchmarks")
    ap.add_argument("--cnn", action="store_true",
                    help="the convolutional worker workload (resnet-mini-c64-W16) instead of the MLP headline")
    ap.add_argument("--compare", action="store_true",
                    help="simulated time-to-loss comparison of Oscars, BSP and fixed-period local SGD")
    ap.add_argument("--compare-configs", default="cfg1,cfg2,cfg3")
    ap.add_argument("--drift-sigma", type=float, default=0.25,
                    help="--compare: sd of the per-window log-speed step of the drifting-speed scenario")
    ap.add_argument("--merge-sizes", default="",
                    help="comma list of P:W merge cases replacing the two default workloads (profiling)")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained", d["bf16_tflops"]), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


# how the GPU arm keeps timed rounds from reusing L2 (the same string in both
# arms, so that their config dicts are identical)
L2_NOTE = "GPU arm: L2 flushed between timed rounds (512 MB write)"
L2_NOTE_MERGE = "inputs larger than L2 (6.8 and 13.6 GB per launch)"


def library_schedule(w):
    """T*, max wait and tau of the library's own scheduler (Algorithm 1 in
    the C ABI), for the workload's speeds."""
    import paper_2102_08550_gb300 as P
    t = P.oscars_iteration_ticks(synth.speeds(w).tolist(), w.ticks_per_unit)
    T, mw, tau = P.oscars_schedule_solve(t, w.M)
    return int(T), int(mw), np.asarray(tau, np.int64)


def workload_config(w, l2=L2_NOTE):
    speeds = "speeds {" + ", ".join(f"{v:g}" for v in w.speeds) + "}" if w.speeds else "lognormal(0,0.5) speeds"
    return {"workload": f"{w.name} (W={w.num_workers}, dims={'-'.join(map(str, w.dims))}, batch={w.batch}, "
                        f"M={w.M}, {speeds})",
            "W": w.num_workers, "batch": w.batch, "M": w.M, "lr": w.lr,
            "samples_per_worker": w.samples_per_worker, "l2": l2}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    def __init__(self, index: int):
        self.index = index
        self.proc = None
        # raw samples (the JSON line carries their summary); OSCARS_CLOCK_LOG_DIR keeps them elsewhere
        log_dir = os.environ.get("OSCARS_CLOCK_LOG_DIR", tempfile.gettempdir())
        self.path = os.path.join(log_dir, f"oscars_clocks_{os.getpid()}.csv")

    def __enter__(self):
        if self.index < 0:                # sampling off
            return self
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if not self.proc:
            return None
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() in ("active", "1", "0x1"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ------------------------------------------------------------------ GPU arm
def algorithmic_work(w, tau):
    """Per-round algorithmic work of each kernel class of the MLP path:
    {class: (flops, hbm_bytes)}.  Bytes count every operand once at its
    stored width (fp32 master 4 B, bf16 operand copies 2 B), i.e. what a
    kernel must move if nothing stays on chip between launches."""
    B, d = w.batch, w.dims
    L = len(d) - 1
    n = float(np.sum(tau))            # worker-steps per round
    W = w.num_workers
    fl, by = {}, {}

    def add(k, f, b):
        fl[k] = fl.get(k, 0.0) + f
        by[k] = by.get(k, 0.0) + b
    for l in range(L - 1):            # hidden layers on the tensor cores
        i, o = d[l], d[l + 1]
        add("gemm_fwd", n * 2 * B * i * o, n * (o * i * 2 + B * i * 2 + 2 * B * o * 2 + o * 4))
        add("gemm_dw_sgd", n * 2 * B * i * o,
            n * (o * i * (4 + 4 + 2) + o * B * 2 + i * B * 2 + o * (4 + 4 + 4)))
        if l >= 1:
            add("gemm_dh", n * 2 * B * i * o, n * (o * i * 2 + B * o * 2 + B * i * 2 + 2 * B * i * 2 + i * 4))
    H, C = d[L - 1], d[L]
    if L == 1:                        # fp32 softmax regression on the CUDA cores: logits + weight gradient
        add("softreg_round", n * 4 * B * H * C, n * (B * H * 4 + B * 4) + W * (C * H + C) * 4 * 2)
    add("head_fwd", n * 2 * B * H * C, n * (C * H * 2 + B * H * 2 + B * C * 4 + B * 4 + C * 4))
    add("head_bwd", n * 4 * B * H * C,
        n * (B * H * 2 + C * H * (2 + 4 + 4 + 2) + 2 * B * H * 2 + H * 4 + B * C * 4 + C * 8))
    add("stage", 0.0, n * B * (d[0] * 4 + 2 * d[0] * 2 + 8))
    # the fused last layer of the per-layer path does the head's forward and
    # backward in one launch
    fl["head_fused"], by["head_fused"] = fl["head_fwd"] + fl["head_bwd"], by["head_fwd"] + by["head_bwd"]
    # the one-launch round of a 2-layer model does all of the above per step
    # and keeps each worker's model on chip for the round: its work is the sum
    # of the parts, its compulsory bytes the global model read once (the
    # workers share it through L2), every worker's replica written once, and
    # each step's staged inputs (X and X^T bf16, labels)
    if L == 2:
        i = d[0]
        P_model = sum(a * b + b for a, b in zip(d[:-1], d[1:]))
        fl["fused_round"] = fl["gemm_fwd"] + fl["gemm_dw_sgd"] + fl["head_fwd"] + fl["head_bwd"]
        by["fused_round"] = P_model * 4.0 * (1 + W) + n * (2 * B * i * 2 + B * 4)
    P_pad = w.num_params   # padding is < 0.1%
    add("merge", 2.0 * W * P_pad, (W + 2) * P_pad * 4.0)
    add("shadow_refresh", 0.0, P_pad * 6.0)
    return fl, by


# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per launch from one
# ncu capture of the kernel as it stands, with the profile summary that holds
# it; a kernel missing here reports traffic null.
NCU_TRAFFIC = {
    ("fused_round", "mlp-784-512-10-W16"): (15.999488e6, "profiles/fused_round_mlp784-512-10_W16.md"),
}


_ALU_PEAK = None


def alu_peak_tflops():
    """fp32 FFMA peak of the CUDA cores: SMs x 128 FFMA per clock x 2 FLOP x
    the maximum SM clock (nvidia-smi; 2070 MHz if it cannot be read)."""
    global _ALU_PEAK
    if _ALU_PEAK is None:
        import torch
        sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
        mhz = 2070.0
        try:
            out = subprocess.run(["nvidia-smi", "-i", str(torch.cuda.current_device()), "--query-gpu=clocks.max.sm",
                                  "--format=csv,noheader,nounits"], capture_output=True, text=True, timeout=10)
            mhz = float(out.stdout.strip().splitlines()[0])
        except Exception:
            pass
        _ALU_PEAK = (sms * 128 * 2 * mhz * 1e6 / 1e12, f"{sms} SMs x 128 FFMA x 2 x {mhz:.0f} MHz")
    return _ALU_PEAK


def roofline_of(name, ms_per_launch, launches_per_round, flops, bytes_, hbm, tflops, peak_kind, workload=None):
    """Roofline of one kernel class from its algorithmic work per launch and
    its measured duration per launch.  ``bound`` is the roof that binds at
    that work (the larger of flops / bf16 peak and bytes / HBM peak);
    tensor-core kernels also report ``tensor_frac`` (their FLOP rate over the
    bf16 peak) beside an HBM bound, and ``hbm_frac`` beside a tensor bound."""
    f = flops.get(name, 0.0) / launches_per_round
    b = bytes_.get(name, 0.0) / launches_per_round
    t = ms_per_launch / 1e3
    if name == "softreg_round" and f > 0.0:     # fp32 CUDA-core arithmetic
        peak, how = alu_peak_tflops()
        ach = f / t / 1e12
        return {"kernel": name, "bound": "alu", "achieved": ach, "peak": peak, "unit": "TFLOP/s", "frac": ach / peak,
                "peak_kind": f"fp32 FFMA ({how})", "flops_per_launch": f, "bytes_per_launch": b,
                "ms_per_launch": ms_per_launch, "traffic": None}
    if f == 0.0 and b == 0.0:
        return {"kernel": name, "bound": "alu", "achieved": None, "peak": None, "unit": None, "frac": None,
                "ms_per_launch": ms_per_launch, "traffic": None}
    t_flop = f / (tflops * 1e12)
    t_mem = b / (hbm * 1e9)
    tr = NCU_TRAFFIC.get((name, workload))
    traffic = tr[0] if tr else None
    tensor_frac = f / t / 1e12 / tflops if name in TENSOR_KERNELS and f > 0.0 else None
    if t_flop >= t_mem:
        ach = f / t / 1e12
        return {"kernel": name, "bound": "tensor", "achieved": ach, "peak": tflops, "unit": "TFLOP/s",
                "frac": ach / tflops, "peak_kind": f"{peak_kind} bf16 dense (burst)", "flops_per_launch": f,
                "bytes_per_launch": b, "ms_per_launch": ms_per_launch, "traffic": traffic,
                "traffic_source": tr[1] if tr else None, "hbm_frac": b / t / 1e9 / hbm}
    ach = b / t / 1e9
    return {"kernel": name, "bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
            "peak_kind": f"{peak_kind} HBM copy", "flops_per_launch": f, "bytes_per_launch": b,
            "ms_per_launch": ms_per_launch, "traffic": traffic,
            "traffic_source": tr[1] if tr else None, "tensor_frac": tensor_frac,
            "tensor_peak": tflops if tensor_frac is not None else None}


def max_over_ranks(ms: float, world: int, device) -> float:
    """The slowest rank's time (every rank gets it); identity for one rank."""
    if world <= 1:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, world: int, max_ms: float) -> float:
    """Units processed by all ranks divided by the slowest rank's time (weak
    scaling: every rank runs its own replica of the workload)."""
    return units_per_rank * world / (max_ms / 1e3)


def measure_rounds(w, steps, warmup, dev, world=1, local_rank=0, flush=None, clock=True, prof_rounds=None):
    """Oscars rounds of the MLP workload ``w`` on ``dev``: device time of
    ``steps`` rounds (CUDA events, L2 flushed between rounds), then the
    per-kernel split from an instrumented replay."""
    import torch
    import paper_2102_08550_gb300 as P
    hbm, tf_burst, tf_sus, peak_kind = peaks()
    shards = [synth.shard_t(w, k, dev) for k in range(w.num_workers)]
    layers0 = synth.init_layers_np(w)
    init = torch.from_numpy(synth.flatten_layers(layers0)).to(dev)
    stream = torch.cuda.current_stream(dev)

    def make(flags=0):
        return P.OscarsContext(num_workers=w.num_workers, dims=w.dims, batch=w.batch, lr=w.lr, bf16=w.bf16,
                               speed=synth.speeds(w).tolist(), M=w.M, shards=shards, init_params=init,
                               stream=stream.cuda_stream, flags=flags)

    ctx = make()
    sch = ctx.schedule()                 # what the library runs: its own Algorithm 1
    tau = np.asarray(sch["tau"], np.int64)
    T_star = sch["T_star"]
    samples_per_round = int(np.sum(tau)) * w.batch
    if flush is None:
        flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)   # > L2 (129 MB)

    def one_round():
        P.oscars_local_steps(ctx.handle, want_tau=False, want_loss=False)
        P.oscars_push_merge(ctx.handle)

    for _ in range(warmup):
        one_round()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    with ClockSampler(local_rank if clock else -1) as clk:
        for i in range(steps):
            flush.fill_(float(i))            # evict the previous round's state from L2 (untimed)
            evs[i][0].record(stream)
            one_round()
            evs[i][1].record(stream)
        torch.cuda.synchronize()
    total_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in evs), world, dev)
    torch.cuda.synchronize()
    ctx.close()
    value = whole_job_rate(samples_per_round * steps, world, total_ms)

    # ---- per-kernel device time: the same round graph with an event node
    # around every kernel (device timeline, no host launch gaps)
    pctx = make(flags=P.FLAG_PROFILE)
    for _ in range(2):
        P.oscars_local_steps(pctx.handle, want_tau=False, want_loss=False)
        P.oscars_push_merge(pctx.handle)
    torch.cuda.synchronize()
    pctx.profile_reset()
    prof_rounds = prof_rounds or max(3, min(steps, 10))
    for i in range(prof_rounds):
        flush.fill_(float(i))
        P.oscars_local_steps(pctx.handle, want_tau=False, want_loss=False)
        P.oscars_push_merge(pctx.handle)
    prof = pctx.profile()
    torch.cuda.synchronize()
    pctx.close()
    del shards
    launches_per_round = sum(c for _, c in prof.values()) / prof_rounds
    flops, bytes_ = algorithmic_work(w, tau)
    dom = max(prof, key=lambda k: prof[k][0])
    kernels = {}
    tot = sum(x[0] for x in prof.values())
    for k, (ms, cnt) in prof.items():
        r = roofline_of(k, ms / cnt, cnt / prof_rounds, flops, bytes_, hbm, tf_burst, peak_kind)
        kernels[k] = {"ms_per_round": ms / prof_rounds, "launches_per_round": cnt / prof_rounds,
                      "share": ms / tot, "bound": r["bound"], "frac": r["frac"]}
        if k in TENSOR_KERNELS and flops.get(k, 0.0) > 0.0:   # tensor-core work: its fraction of the tensor peak
            tf = flops[k] / (ms / prof_rounds / 1e3) / 1e12
            kernels[k]["tflops"] = tf
            kernels[k]["tensor_frac"] = tf / tf_burst
    gemm = [k for k in kernels if k.startswith("gemm_") or k == "head_fused"]
    if gemm:                            # the grouped worker GEMMs together
        g_ms = sum(prof[k][0] for k in gemm) / prof_rounds
        g_tf = sum(flops.get(k, 0.0) for k in gemm) / (g_ms / 1e3) / 1e12
        kernels["all_gemms"] = {"ms_per_round": g_ms, "share": g_ms * prof_rounds / tot, "tflops": g_tf,
                                "tensor_frac": g_tf / tf_burst}
    roof = roofline_of(dom, prof[dom][0] / prof[dom][1], prof[dom][1] / prof_rounds, flops, bytes_, hbm, tf_burst,
                       peak_kind, w.name)
    return {"value": value, "ms_per_step": total_ms / steps, "roofline": roof, "kernels": kernels,
            "gpu_launches": int(round(launches_per_round * steps)), "clocks": clk.summary() if clock else None,
            "samples_per_round": samples_per_round, "T_star": int(T_star), "tau": [int(v) for v in tau]}


# kernel classes whose FLOPs run on the tensor cores (tcgen05)
TENSOR_KERNELS = ("gemm_fwd", "gemm_dh", "gemm_dw_sgd", "head_fused", "fused_round")

# the training workloads measured beside the headline (absolute samples/s and
# the roofline of their dominant kernel)
SIDE_WORKLOADS = (synth.CFG1, synth.CFG3)


def run_side_workloads(args, dev):
    import torch
    out = {}
    for w in SIDE_WORKLOADS:
        r = measure_rounds(w, max(20, args.steps), max(3, args.warmup), dev, clock=False, prof_rounds=3)
        e2e = None
        if not args.no_e2e:
            shards = [synth.shard_t(w, k, dev) for k in range(w.num_workers)]
            e2e = run_e2e(args, shards, w, np.asarray(r["tau"]), dev, torch.cuda.current_stream(dev))
            del shards
        out[w.name] = {"metric": "simulated-worker samples/s", "value": r["value"], "unit": UNIT,
                       "ms_per_round": r["ms_per_step"], "config": workload_config(w),
                       "dtype": "bf16 (fp32 master, fp32 accumulate)" if w.bf16 else "f32",
                       "roofline": r["roofline"], "kernels": r["kernels"], "samples_per_round": r["samples_per_round"],
                       "e2e": e2e}
        torch.cuda.empty_cache()
    return out


def run_gpu(args, rank, world, local_rank):
    import torch
    from paper_2102_08550_gb300 import _build

    _build.build()
    dev = torch.device(f"cuda:{local_rank}")
    torch.cuda.set_device(dev)
    w = WORKLOADS[args.workload]
    if args.samples_per_worker:
        w = dataclasses.replace(w, samples_per_worker=args.samples_per_worker)
    hbm, tf_burst, tf_sus, peak_kind = peaks()
    stream = torch.cuda.current_stream(dev)
    res = measure_rounds(w, args.steps, args.warmup, dev, world, local_rank)

    # ---- end to end through the C ABI with host-resident inputs
    e2e = None
    if not args.no_e2e:
        shards = [synth.shard_t(w, k, dev) for k in range(w.num_workers)]
        e2e = run_e2e(args, shards, w, np.asarray(res["tau"]), dev, stream, world)
        del shards
        torch.cuda.empty_cache()

    res["e2e"] = e2e
    res["merge"] = None if args.no_merge else run_merge(args, dev, stream, hbm, peak_kind)
    res["workloads"] = (run_side_workloads(args, dev)
                        if world == 1 and args.workload == WORKLOAD.name and not args.no_side else None)
    return res


def run_e2e(args, shards, w, tau, dev, stream, world=1):
    """End to end through the C ABI with the inputs in HOST memory: the
    shards live in pinned host memory and the library's staging kernel reads
    each round's mini-batches straight from there (over the host link), then
    the round runs and the per-worker losses are read back to the host."""
    import torch
    import paper_2102_08550_gb300 as P
    host = [(x.cpu().pin_memory(), y.cpu().pin_memory()) for x, y in shards]
    layers0 = synth.init_layers_np(w)
    init = torch.from_numpy(synth.flatten_layers(layers0)).pin_memory()
    ctx = P.OscarsContext(num_workers=w.num_workers, dims=w.dims, batch=w.batch, lr=w.lr, bf16=w.bf16,
                          speed=synth.speeds(w).tolist(), M=w.M, shards=host, init_params=init,
                          stream=stream.cuda_stream)
    # warm-up: one full pass over every shard.  The first touch of each
    # pinned host page costs extra once per process; the timed rounds measure
    # the steady state and the first pass is reported beside it.
    samples = int(np.sum(tau)) * w.batch
    epoch = max(3, args.warmup, max(int(np.ceil(w.samples_per_worker / (int(t) * w.batch))) for t in tau))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    ctx.train(epoch)
    first_pass = samples * epoch / (time.perf_counter() - t0)
    # timed: one oscars_train call, the API a user trains with.  Every round
    # its W per-worker losses are copied to pinned host memory and read by the
    # host (the library pipelines the rounds one deep).
    steps = max(200, args.steps)      # a wall-clock measurement: tens of milliseconds, not a few
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    log = ctx.train(steps)
    dt = max_over_ranks(time.perf_counter() - t0, world, dev)
    assert len(log) == steps and all(np.isfinite(r["worker_loss"]) for r in log)
    ctx.close()
    h2d = samples * (w.dims[0] * 4 + 4)
    return {"value": whole_job_rate(samples * steps, world, dt * 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": 4 * w.num_workers, "steps": steps, "warmup_rounds": epoch,
            "first_pass_value": first_pass,
            "note": "one oscars_train call, host wall clock; shards in pinned host memory, read by the staging "
                    "kernel; losses read back every round"}


def merge_workloads(args):
    if not args.merge_sizes:
        return [synth.CFG4, synth.CFG5]
    out = []
    for item in args.merge_sizes.split(","):
        Pn, W = (int(v) for v in item.split(":"))
        out.append(synth.MergeWorkload(f"merge-P{Pn}-W{W}", W, Pn, 1e-3, 8, "localsteps"))
    return out


# DRAM bytes per algorithmic byte of the merge kernel, from ncu captures of
# smaller launches of the same kernel with the same worker count (the
# full-size launches are too large to capture; traffic grows in proportion to
# P): (dram__bytes_read.sum + dram__bytes_write.sum) / ((W + 2) * P * 4).
MERGE_TRAFFIC = {
    64: (0.99694, "profiles/merge_vec4_P4M_W64.md (P = 4M, scaled by P)"),
    8: (0.98816, "profiles/merge_vec4_P32M_W8.md (P = 32M, scaled by P)"),
}


def run_merge(args, dev, stream, hbm, peak_kind):
    import torch
    import paper_2102_08550_gb300 as P
    res = {}
    for m in merge_workloads(args):
        W, Pn = m.num_workers, m.num_params
        rule = P.W_LOCALSTEPS if m.weight_rule == "localsteps" else P.W_UNIFORM
        xg0 = synth.merge_xg_t(m, 0, Pn, dev)
        deltas = [synth.merge_delta_t(m, k, 0, Pn, dev) for k in range(W)]
        ctx = P.OscarsContext(num_workers=W, dims=[Pn], model=P.MODEL_FLAT, weight_rule=rule, t_ticks=[1] * W,
                              M=2, init_params=xg0, server_lr=m.server_lr, stream=stream.cuda_stream)
        del xg0
        ctx.set_local_steps(synth.merge_taus(m).tolist())
        ptrs = [d.data_ptr() for d in deltas]
        for _ in range(3):
            P.oscars_push_merge(ctx.handle, ptrs)
        torch.cuda.synchronize()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.merge_reps)]
        for a, b in evs:
            a.record(stream)
            P.oscars_push_merge(ctx.handle, ptrs)
            b.record(stream)
        torch.cuda.synchronize()
        ts = sorted(a.elapsed_time(b) for a, b in evs)
        med = ts[len(ts) // 2]
        alg = (W + 2) * Pn * 4.0
        gbs = alg / (med / 1e3) / 1e9
        tr = MERGE_TRAFFIC.get(W)
        res[m.name] = {"GB/s": gbs, "frac": gbs / hbm, "ms_median": med, "ms_min": ts[0],
                       "bytes_per_launch": alg, "weight_rule": m.weight_rule,
                       "peak": hbm, "peak_kind": f"{peak_kind} HBM copy", "bound": "hbm",
                       "traffic": tr[0] * alg if tr else None, "traffic_source": tr[1] if tr else None,
                       "launches": args.merge_reps, "l2": L2_NOTE_MERGE}
        ctx.close()
        del deltas
        torch.cuda.empty_cache()
    return res


def merge_cpu_baseline(m, dev, budget_s=8.0):
    """The oracle merge (fp64 sum in worker order) on the host cores over a
    bounded prefix of the parameter vector: GB/s of (W + 2) * P_sample * 4
    algorithmic bytes.  The inputs are drawn on the GPU (untimed)."""
    from oracle import merge as omerge
    from oracle import schedule as S
    n = 1 << 20 if m.num_workers > 16 else 1 << 22
    xg = synth.merge_xg_t(m, 0, n, dev).cpu().numpy()
    deltas = [synth.merge_delta_t(m, k, 0, n, dev).cpu().numpy() for k in range(m.num_workers)]
    w = S.merge_weights(m.weight_rule, synth.merge_taus(m))
    omerge.merge_deltas(xg, deltas, w, m.server_lr)          # warm-up
    t0 = time.perf_counter()
    reps = 0
    while True:
        omerge.merge_deltas(xg, deltas, w, m.server_lr)
        reps += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    return {"value": (m.num_workers + 2) * n * 4.0 * reps / dt / 1e9, "unit": "GB/s", "cores": cores_used(),
            "kind": "oracle", "sample": f"{reps} merges of the first {n} of {m.num_params} parameters, "
                                        f"W={m.num_workers} (numpy fp64)"}


# ------------------------------------------------------------------ CPU oracle
def oracle_rounds(w, rounds, budget_s):
    """Run up to ``rounds`` oracle rounds (stopping after budget_s seconds);
    returns (samples, seconds, rounds run)."""
    from oracle import run as orun
    from oracle import bf16 as obf16
    from oracle import schedule as S
    t = S.iteration_ticks(synth.speeds(w), w.ticks_per_unit)
    T, mw, tau = S.schedule(t, w.M)
    rows = min(w.samples_per_worker, rounds * int(tau.max()) * w.batch + w.batch)
    shards = [synth.shard_np(w, k, n=rows) for k in range(w.num_workers)]
    state = orun.init_state(w.dims, synth.init_layers_np(w), t, w.M)
    rnd = obf16.round_bf16 if w.bf16 else obf16.identity
    t0 = time.perf_counter()
    done = 0
    for _ in range(rounds):
        orun.run_round(state, shards, w.batch, w.lr, rnd)
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    return done * int(np.sum(tau)) * w.batch, dt, done


def cores_used():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


COMPARE = {"cfg1": (synth.CFG1, 20), "cfg2": (synth.CFG2, 30), "cfg3": (synth.CFG3, 10)}


def run_compare(args, dev):
    """Eval loss against simulated time for three schemes on one workload,
    all through oscars_train with the same data, init and eval set."""
    import torch
    import paper_2102_08550_gb300 as P
    for key in [k for k in args.compare_configs.split(",") if k]:
        w, oscars_rounds = COMPARE[key]
        speeds = synth.speeds(w).tolist()
        t = P.oscars_iteration_ticks(speeds, w.ticks_per_unit)
        tau_o, B_o = P.oscars_policy_local_steps(P.POLICY_OSCARS, t, w.M)
        I = max(1, int(round(float(np.median(tau_o)))))
        horizon = oscars_rounds * B_o
        shards = [synth.shard_t(w, k, dev) for k in range(w.num_workers)]
        Xe, ye = synth.eval_t(w, dev)
        init = torch.from_numpy(synth.flatten_layers(synth.init_layers_np(w))).to(dev)
        res = {}
        for name, pol, per in (("oscars", P.POLICY_OSCARS, 1), ("bsp", P.POLICY_BSP, 1),
                               (f"local_sgd_I{I}", P.POLICY_LOCAL_SGD, I)):
            tau, B = P.oscars_policy_local_steps(pol, t, w.M, P.SEARCH_CAPPED, per)
            rounds = max(1, horizon // B)
            ctx = P.OscarsContext(num_workers=w.num_workers, dims=w.dims, batch=w.batch, lr=w.lr,
                                  bf16=w.bf16, speed=speeds, ticks_per_unit=w.ticks_per_unit, M=w.M,
                                  shards=shards, init_params=init,
                                  stream=torch.cuda.current_stream(dev).cuda_stream)
            ctx.set_local_steps(tau)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            log = ctx.train(rounds, Xe, ye)
            wall = time.perf_counter() - t0
            ctx.close()
            step = max(1, len(log) // 20)
            res[name] = {"tau": tau, "barrier_ticks": B, "rounds": len(log),
                         "idle_frac": float(1.0 - sum(a * b for a, b in zip(tau, t)) / (B * len(t))),
                         "samples": len(log) * int(sum(tau)) * w.batch, "final_eval_loss": log[-1]["eval_loss"],
                         "curve": [[e["ticks"], round(e["eval_loss"], 6)] for e in log[step - 1::step]],
                         "wall_s": wall, "_log": log}
        target = res["bsp"]["final_eval_loss"]
        for r in res.values():
            log = r.pop("_log")
            r["ticks_to_target"] = next((e["ticks"] for e in log if e["eval_loss"] <= target), None)
        base = res["bsp"]["ticks_to_target"]
        for r in res.values():
            r["speedup_vs_bsp"] = base / r["ticks_to_target"] if r["ticks_to_target"] else None
        print(json.dumps({"mode": "compare", "workload": workload_config(w, "n/a")["workload"],
                          "dtype": "bf16" if w.bf16 else "fp32", "horizon_ticks": horizon,
                          "target_loss": target, "policies": res}))


def run_compare_drift(args, dev, key):
    """Drifting speeds: each worker's speed is constant over windows of T*_0
    ticks (the first Oscars barrier) and takes a log-normal step between
    windows.  Each scheme starts every round with the speeds in force at its
    simulated time: Oscars re-solves Algorithm 1 (oscars_set_iteration_ticks),
    "static" keeps the first round's tau while the round lengths follow the
    true times, BSP runs one step per barrier."""
    import torch
    import paper_2102_08550_gb300 as P
    w, oscars_rounds = COMPARE[key]
    sp = synth.drifting_speeds(w, 4 * oscars_rounds + 1, sigma=args.drift_sigma)
    ts = [P.oscars_iteration_ticks(sp[r].tolist(), w.ticks_per_unit) for r in range(sp.shape[0])]
    tau0, window = P.oscars_policy_local_steps(P.POLICY_OSCARS, ts[0], w.M)
    horizon = oscars_rounds * window
    shards = [synth.shard_t(w, k, dev) for k in range(w.num_workers)]
    Xe, ye = synth.eval_t(w, dev)
    init = torch.from_numpy(synth.flatten_layers(synth.init_layers_np(w))).to(dev)
    res = {}
    for name in ("oscars_adaptive", "oscars_static", "bsp"):
        ctx = P.OscarsContext(num_workers=w.num_workers, dims=w.dims, batch=w.batch, lr=w.lr, bf16=w.bf16,
                              speed=sp[0].tolist(), ticks_per_unit=w.ticks_per_unit, M=w.M, shards=shards,
                              init_params=init, stream=torch.cuda.current_stream(dev).cuda_stream)
        now, log, samples, busy, span = 0, [], 0, 0, 0
        while now < horizon:
            t = ts[min(now // window, len(ts) - 1)]
            ctx.set_iteration_ticks(t)                     # Algorithm 1 on the times in force
            if name == "oscars_static":
                ctx.set_local_steps(tau0)
            elif name == "bsp":
                ctx.set_local_steps([1] * w.num_workers)
            e = ctx.train(1, Xe, ye)[0]
            sch = ctx.schedule()
            now += e["barrier"]
            samples += int(sum(sch["tau"])) * w.batch
            busy += sum(a * b for a, b in zip(sch["tau"], t))
            span += e["barrier"] * w.num_workers
            log.append([now, e["eval_loss"]])
        ctx.close()
        res[name] = {"rounds": len(log), "samples": samples, "idle_frac": 1.0 - busy / span,
                     "final_eval_loss": log[-1][1], "_log": log}
    target = max(r["final_eval_loss"] for r in res.values())
    for r in res.values():
        log = r.pop("_log")
        r["ticks_to_target"] = next((tk for tk, ev in log if ev <= target), None)
        step = max(1, len(log) // 20)
        r["curve"] = [[tk, round(ev, 6)] for tk, ev in log[step - 1::step]]
    print(json.dumps({"mode": "compare-drift", "workload": workload_config(w, "n/a")["workload"],
                      "sigma": args.drift_sigma, "window_ticks": window, "horizon_ticks": horizon,
                      "target_loss": target, "policies": res}))


def cnn_work(w, tau, tiles_per_image=8):
    """Per-round algorithmic FLOPs of the convolutional worker by kernel class
    (multiply-adds x2; the stem counts its real input channels)."""
    n = float(np.sum(tau)) * w.batch            # samples per round
    hw, C, K = w.height * w.width, w.ch, w.dims[-1]
    block = 2.0 * hw * C * 9 * C
    stem = 2.0 * hw * C * 9 * w.in_ch
    return {"conv_fwd": n * (stem + 2 * w.blocks * block),
            "conv_dgrad": n * 2 * w.blocks * block,
            "conv_wgrad": n * (stem + 2 * w.blocks * block),
            "cnn_head": n * 3 * 2 * C * K}


def run_cnn(args, dev):
    """Oscars rounds of the convolutional worker: samples/s with the tensor
    roofline of its convolution kernels."""
    import torch
    import paper_2102_08550_gb300 as P
    w = synth.CFG6
    hbm, tf_burst, tf_sus, peak_kind = peaks()
    T_star, mw, tau = library_schedule(w)
    samples_per_round = int(np.sum(tau)) * w.batch
    shards = [synth.shard_t(w, k, dev) for k in range(w.num_workers)]
    # canonical layout: the tensors one after the other
    init = torch.from_numpy(np.concatenate([p.reshape(-1) for p in synth.init_cnn_np(w)]).astype(np.float32)).to(dev)
    stream = torch.cuda.current_stream(dev)

    def make(flags=0):
        return P.OscarsContext(num_workers=w.num_workers, dims=w.cnn_dims, model=P.MODEL_CNN, blocks=w.blocks,
                               batch=w.batch, lr=w.lr, speed=synth.speeds(w).tolist(), M=w.M, shards=shards,
                               init_params=init, stream=stream.cuda_stream, flags=flags)
    ctx = make()
    flush = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    for _ in range(args.warmup):
        P.oscars_local_steps(ctx.handle, want_tau=False, want_loss=False)
        P.oscars_push_merge(ctx.handle)
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(0) as clk:
        for i in range(args.steps):
            flush.fill_(float(i))
            evs[i][0].record(stream)
            P.oscars_local_steps(ctx.handle, want_tau=False, want_loss=False)
            P.oscars_push_merge(ctx.handle)
            evs[i][1].record(stream)
        torch.cuda.synchronize()
    total_ms = sum(a.elapsed_time(b) for a, b in evs)
    _, loss = P.oscars_local_steps(ctx.handle, want_tau=False, want_loss=True)
    P.oscars_push_merge(ctx.handle)
    ctx.close()
    # per-kernel-class device time
    pctx = make(flags=P.FLAG_PROFILE)
    P.oscars_local_steps(pctx.handle, want_tau=False, want_loss=False)
    P.oscars_push_merge(pctx.handle)
    torch.cuda.synchronize()
    pctx.profile_reset()
    prof_rounds = 3
    for i in range(prof_rounds):
        flush.fill_(float(i))
        P.oscars_local_steps(pctx.handle, want_tau=False, want_loss=False)
        P.oscars_push_merge(pctx.handle)
    prof = pctx.profile()
    torch.cuda.synchronize()
    pctx.close()
    work = cnn_work(w, tau)
    kernels = {}
    for name, (ms, cnt) in prof.items():
        per_round = ms / prof_rounds
        k = {"ms_per_round": per_round, "launches_per_round": cnt / prof_rounds}
        if name in work:
            k["tflops"] = work[name] / (per_round / 1e3) / 1e12
            k["frac"] = k["tflops"] / tf_sus
        kernels[name] = k
    conv_ms = sum(kernels[k]["ms_per_round"] for k in ("conv_fwd", "conv_dgrad", "conv_wgrad") if k in kernels)
    conv_fl = sum(work[k] for k in ("conv_fwd", "conv_dgrad", "conv_wgrad"))
    ach = conv_fl / (conv_ms / 1e3) / 1e12
    line = {"metric": "simulated-worker samples/s (Oscars rounds, convolutional worker)",
            "value": samples_per_round * args.steps / (total_ms / 1e3), "unit": "samples/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16 (fp32 master, fp32 accumulate)", "data": "synthetic (seeded CIFAR-shaped Gaussian mixture)",
            "config": {"workload": f"{w.name} (W={w.num_workers}, 32x32x3 images, stem + {w.blocks} residual block(s) "
                                   f"of 64 channels, batch={w.batch}, M={w.M})", "l2": "flushed between timed rounds"},
            "roofline": {"kernel": "conv_fwd + conv_dgrad + conv_wgrad", "bound": "tensor", "achieved": ach,
                         "peak": tf_sus, "unit": "TFLOP/s", "frac": ach / tf_sus,
                         "peak_kind": f"{peak_kind} bf16 dense (sustained)", "flops_per_round": conv_fl,
                         "traffic": None},
            "kernels": kernels, "samples_per_round": samples_per_round, "T_star": int(T_star),
            "tau": [int(v) for v in tau], "clocks": clk.summary(), "last_loss": [float(v) for v in loss]}
    print(json.dumps(line))


def run_reference(args):
    w = WORKLOADS[args.workload]
    oracle_rounds(w, max(1, min(args.warmup, 2)), 30.0)          # warm-up (imports, caches)
    samples, dt, done = oracle_rounds(w, args.steps, 120.0)
    value = samples / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": done, "warmup": args.warmup, "ms_per_step": dt / done * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64 (bf16 operand emulation)", "data": "synthetic",
            "config": workload_config(w),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
                             "sample": f"{done} Oscars rounds of {w.name} (numpy fp64, BLAS threads = all cores)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def training_cpu_baseline(w, rounds, budget_s):
    samples, dt, done = oracle_rounds(w, rounds, budget_s)
    return {"value": samples / dt, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
            "sample": f"{done} Oscars rounds of {w.name} (numpy fp64" +
                      (" with bf16 operand emulation)" if w.bf16 else ")")}


ROOF_KEYS = ("kernel", "bound", "achieved", "peak", "unit", "frac", "traffic", "ms_per_launch", "tensor_frac",
             "hbm_frac")


def config_records(res, cpus):
    """Every workload of the run by name: its throughput, the roofline of its
    dominant kernel, its oracle baseline and (training) its end-to-end rate."""
    roof, cpu, e2e = {}, {}, {}
    for name, r in (res.get("workloads") or {}).items():
        roof[name] = {k: r["roofline"].get(k) for k in ROOF_KEYS if r["roofline"].get(k) is not None}
        roof[name]["samples_per_s"] = r["value"]
        if r.get("e2e"):
            e2e[name] = {k: r["e2e"][k] for k in ("value", "unit", "h2d_bytes_per_step", "d2h_bytes_per_step")}
    for name, m in (res.get("merge") or {}).items():
        roof[name] = {"kernel": "merge_vec4", "bound": "hbm", "achieved": m["GB/s"], "peak": m["peak"],
                      "unit": "GB/s", "frac": m["frac"], "traffic": m["traffic"], "ms_per_launch": m["ms_median"]}
    for name, c in cpus.items():
        cpu[name] = c
    return roof, cpu, e2e


def result_line(args, world, w, res, cpu, cpus):
    roof, cpu_cfg, e2e_cfg = config_records(res, cpus)
    top_roof = dict(res["roofline"])
    head = {k: top_roof.get(k) for k in ROOF_KEYS if top_roof.get(k) is not None}
    head["samples_per_s"] = res["value"]
    top_roof["configs"] = {w.name: head, **roof}
    cpu_line = dict(cpu) if cpu else None
    if cpu_line is not None:
        cpu_line["configs"] = {w.name: dict(cpu), **cpu_cfg}
    e2e_line = dict(res["e2e"]) if res["e2e"] else None
    if e2e_line is not None:
        e2e_line["configs"] = {w.name: {k: res["e2e"][k] for k in ("value", "unit", "h2d_bytes_per_step",
                                                                  "d2h_bytes_per_step")}, **e2e_cfg}
    return {"metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16 (fp32 master, fp32 accumulate)",
            "data": "synthetic (seeded Gaussian-mixture shards, random-init MLP)",
            "config": workload_config(w), "roofline": top_roof, "cpu_baseline": cpu_line, "e2e": e2e_line,
            "gpu_launches": res["gpu_launches"], "clocks": res["clocks"], "merge": res["merge"],
            "kernels": res["kernels"], "samples_per_round": res["samples_per_round"],
            "T_star": res["T_star"], "tau": res["tau"], "workloads": res["workloads"]}


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            run_reference(args)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
    if args.cnn:
        import torch
        from paper_2102_08550_gb300 import _build
        _build.build()
        dev = torch.device(f"cuda:{local_rank}")
        torch.cuda.set_device(dev)
        if rank == 0:
            run_cnn(args, dev)
        return
    if args.compare:
        import torch
        from paper_2102_08550_gb300 import _build
        _build.build()
        dev = torch.device(f"cuda:{local_rank}")
        torch.cuda.set_device(dev)
        if rank == 0:
            run_compare(args, dev)
            for key in [k for k in args.compare_configs.split(",") if k in ("cfg1", "cfg2")]:
                run_compare_drift(args, dev, key)
        return
    if args.only == "merge":
        import torch
        from paper_2102_08550_gb300 import _build
        _build.build()
        dev = torch.device(f"cuda:{local_rank}")
        torch.cuda.set_device(dev)
        hbm, _, _, kind = peaks()
        print(json.dumps({"merge": run_merge(args, dev, torch.cuda.current_stream(dev), hbm, kind)}))
        return
    if args.only == "round" or args.workload != WORKLOAD.name:
        args.no_merge = True
    res = run_gpu(args, rank, world, local_rank)
    w = WORKLOADS[args.workload]
    if args.samples_per_worker:
        w = dataclasses.replace(w, samples_per_worker=args.samples_per_worker)
    cpu, cpus = None, {}
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = training_cpu_baseline(w, 6, 10.0)
        if res["workloads"]:
            cpus[synth.CFG1.name] = training_cpu_baseline(synth.CFG1, 20, 4.0)
            cpus[synth.CFG3.name] = training_cpu_baseline(synth.CFG3, 1, 30.0)
        if res["merge"]:
            import torch
            dev = torch.device(f"cuda:{local_rank}")
            for m in merge_workloads(args):
                cpus[m.name] = merge_cpu_baseline(m, dev)
    if rank == 0:
        print(json.dumps(result_line(args, world, w, res, cpu, cpus)))
    if world > 1:
        import torch
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
