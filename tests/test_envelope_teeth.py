"""The bound of the multi-step bf16 parity tests has teeth (CPU only).

Those tests accept, per tensor, max(1e-5, ENV_FACTOR x envelope), where the
envelope is how far the oracle moves from itself when every GEMM output is
perturbed by ENV_REL relative noise (a different fp32 summation order).
Here the oracle stands in for the GPU path:

* a correct implementation with yet another summation order (the oracle
  under a third perturbation seed) stays inside the bound;
* each planted mistake of ``tests.oracle_mutants`` (stale bf16 operand after
  step 0, bias update skipped, one sample dropped per mini-batch, cursor one
  batch ahead) lands outside it by at least a factor 2, on the 784-512-10
  workload with 16 workers
  and on a small 3-layer shape, in every round checked.
"""
import numpy as np
import pytest

import synth
from oracle import run as orun
from oracle import schedule as osched
from tests import oracle_mutants as OM
from tests.gpu_util import ENV_FACTOR, PARAM_RTOL, envelope, per_tensor_errors, perturbed_gemms

CASES = {
    # name: (workload, rounds, rows per shard)
    "mlp-784-512-10-W16": (synth.CFG2, 2, 2 * 6 * 64 + 64),
    "small-3layer": (synth.TrainWorkload("small-3layer", 3, [200, 256, 128, 10], 32, 0.05, 512, 6, 3), 3, 512),
}


def _runner(w, rounds, rows):
    t = osched.iteration_ticks(synth.speeds(w), w.ticks_per_unit)
    shards = [synth.shard_np(w, k, n=rows) for k in range(w.num_workers)]
    layers0 = synth.init_layers_np(w)

    def run():
        _, recs = orun.run(w.dims, layers0, shards, t_iter=t, M=w.M, rounds=rounds, batch=w.batch, lr=w.lr,
                           bf16=w.bf16)
        return [r.x_g for r in recs]
    return run


@pytest.fixture(scope="module", params=sorted(CASES))
def case(request):
    w, rounds, rows = CASES[request.param]
    _, _, tau = osched.schedule(osched.iteration_ticks(synth.speeds(w), w.ticks_per_unit), w.M)
    assert rounds * int(tau.max()) * w.batch <= rows          # no wrap within the rows generated
    run = _runner(w, rounds, rows)
    ref = run()
    env = envelope(run, w.dims, ref)
    bound = [np.maximum(PARAM_RTOL, ENV_FACTOR * np.asarray(e)) for e in env]
    return request.param, w, run, ref, bound


def test_another_summation_order_stays_inside(case):
    name, w, run, ref, bound = case
    with perturbed_gemms(2e-6, 13):
        got = run()
    for r, (g, x, b) in enumerate(zip(got, ref, bound)):
        e = np.asarray(per_tensor_errors(g, x, w.dims))
        assert np.all(e <= b), (name, r, e.tolist(), b.tolist())


@pytest.mark.parametrize("mutant", sorted(OM.MUTANTS))
def test_planted_mistake_lands_outside(case, mutant):
    name, w, run, ref, bound = case
    with OM.MUTANTS[mutant]():
        got = run()
    for r, (g, x, b) in enumerate(zip(got, ref, bound)):
        e = np.asarray(per_tensor_errors(g, x, w.dims))
        assert np.any(e > 2.0 * b), (name, mutant, r, (e / b).tolist())
