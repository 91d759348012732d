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


# ---------------------------------------------------------------- conditioning envelope
class perturbed_gemms:
    """Context manager: every GEMM (and convolution) output of the oracle is multiplied by
    (1 + rel * N(0, 1)), the size of the difference a different fp32
    summation order makes.  Used to measure how far the oracle moves from
    itself, i.e. how well conditioned a run is (test infrastructure only)."""

    def __init__(self, rel: float, seed: int):
        self.rel, self.rng = rel, np.random.default_rng(seed)

    def __enter__(self):
        from oracle import conv as oc
        from oracle import model as om
        self.om, self.nt, self.nn = om, om.gemm_nt, om.gemm_nn
        self.oc, self.convs = oc, (oc.conv3x3, oc.conv3x3_transposed, oc.conv3x3_weight_grad)
        rel, rng = self.rel, self.rng

        def wrap(f):
            def g(a, b, rnd):
                out = f(a, b, rnd)
                return (out * (1.0 + rel * rng.standard_normal(out.shape))).astype(np.float32)
            return g
        om.gemm_nt, om.gemm_nn = wrap(self.nt), wrap(self.nn)
        oc.conv3x3, oc.conv3x3_transposed, oc.conv3x3_weight_grad = (wrap(f) for f in self.convs)
        return self

    def __exit__(self, *a):
        self.om.gemm_nt, self.om.gemm_nn = self.nt, self.nn
        self.oc.conv3x3, self.oc.conv3x3_transposed, self.oc.conv3x3_weight_grad = self.convs


ENV_REL = 2e-6       # relative GEMM-output perturbation (about 30 fp32 ulps)
ENV_SEEDS = (11, 12)
ENV_FACTOR = 4.0


def envelope(run_fn, dims, ref_flats, errors=None):
    """Per-round, per-tensor max divergence of perturbed oracle runs from the
    unperturbed ones; ``run_fn()`` returns a list of flat parameter vectors.
    ``errors(flat, ref)`` gives the per-tensor errors (default: the MLP
    layout of ``dims``)."""
    errors = errors or (lambda f, ref: per_tensor_errors(f, ref, dims))
    env = [None for _ in ref_flats]
    for s in ENV_SEEDS:
        with perturbed_gemms(ENV_REL, s):
            flats = run_fn()
        for r, (f, ref) in enumerate(zip(flats, ref_flats)):
            e = np.asarray(errors(f, ref))
            env[r] = e if env[r] is None else np.maximum(env[r], e)
    return env


def assert_within(errs, env, what):
    """Every tensor within 1e-5, or within ENV_FACTOR times the oracle's own
    divergence under fp32-sized perturbations (bf16 rounding and ReLU masks
    amplify those; the envelope is measured, not assumed)."""
    bound = np.maximum(PARAM_RTOL, ENV_FACTOR * np.asarray(env))
    assert np.all(np.asarray(errs) <= bound), (what, list(np.round(errs, 9)), list(np.round(bound, 9)))
