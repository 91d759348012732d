"""Helpers for the GPU parity tests: build a context from a synthetic
workload, run rounds through the C ABI, and compare with the oracle."""
from __future__ import annotations

import numpy as np
import torch

import paper_2102_08550_gb300 as P
import synth
from oracle import run as orun
from oracle import schedule as osched

# tolerances of the parity contract
PARAM_RTOL = 1e-5     # merged parameters: max-abs error / max-abs value, per tensor
LOSS_RTOL = 1e-3      # losses: relative


def rel_maxabs(got: np.ndarray, ref: np.ndarray) -> float:
    ref = np.asarray(ref, np.float64)
    den = np.abs(ref).max()
    return float(np.abs(np.asarray(got, np.float64) - ref).max() / (den if den > 0 else 1.0))


def per_tensor_errors(flat_got, flat_ref, dims):
    out = []
    for (Wg, bg), (Wr, br) in zip(orun.unflatten(flat_got, dims), orun.unflatten(flat_ref, dims)):
        out.append(rel_maxabs(Wg, Wr))
        out.append(rel_maxabs(bg, br))
    return out


def device_shards(w: synth.TrainWorkload, device, n=None):
    return [synth.shard_t(w, k, device, n=n) for k in range(w.num_workers)]


def make_context(w: synth.TrainWorkload, shards, device, flags=0, layers0=None, **kw):
    layers0 = layers0 if layers0 is not None else synth.init_layers_np(w)
    init = torch.from_numpy(synth.flatten_layers(layers0)).to(device)
    ctx = P.OscarsContext(num_workers=w.num_workers, dims=w.dims, batch=w.batch, lr=w.lr,
                          server_lr=w.server_lr, bf16=w.bf16, speed=synth.speeds(w).tolist(),
                          ticks_per_unit=w.ticks_per_unit, M=w.M, shards=shards, init_params=init,
                          stream=torch.cuda.current_stream().cuda_stream, flags=flags, **kw)
    return ctx, layers0


def oracle_inputs(w: synth.TrainWorkload, rows: int):
    """First ``rows`` rows of every worker's shard (enough for the rounds run)."""
    return [synth.shard_np(w, k, n=rows) for k in range(w.num_workers)]


def pull_flat(ctx, device):
    out = torch.empty(ctx.P, dtype=torch.float32, device=device)
    ctx.pull(out)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def replica_flat(ctx, k, device):
    out = torch.empty(ctx.P, dtype=torch.float32, device=device)
    ctx.read_replica(k, out)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def oracle_schedule(w: synth.TrainWorkload):
    t = osched.iteration_ticks(synth.speeds(w), w.ticks_per_unit)
    T, mw, tau = osched.schedule(t, w.M)
    return t, T, mw, tau
