"""How well conditioned is a local-SGD round?  The oracle is run twice on
the same inputs, once with every GEMM output perturbed by 1e-7 relative noise
(the size of a different fp32 summation order).  With fp32 operands the two
runs stay within about 1e-6; with bf16 operand rounding the rounding and
ReLU-mask decisions amplify the perturbation by orders of magnitude.  This
is a property of the arithmetic: it fixes what tolerance a GPU path with a
different summation order can meet on multi-step bf16 runs."""
import dataclasses

import numpy as np

import synth
from oracle import run as orun
from oracle import schedule as osched
from tests.gpu_util import per_tensor_errors, perturbed_gemms

W = synth.TrainWorkload("cond", 4, [784, 512, 10], 64, 0.05, 512, 8, 1)


def one_round(w, noise=None):
    t = osched.iteration_ticks(synth.speeds(w))
    shards = [synth.shard_np(w, k, n=512) for k in range(w.num_workers)]
    layers = synth.init_layers_np(w)
    if noise is None:
        return orun.run(w.dims, layers, shards, t_iter=t, M=w.M, rounds=1, batch=w.batch, lr=w.lr, bf16=w.bf16)[1][0].x_g
    with perturbed_gemms(noise, 1):
        return orun.run(w.dims, layers, shards, t_iter=t, M=w.M, rounds=1, batch=w.batch, lr=w.lr, bf16=w.bf16)[1][0].x_g


def test_fp32_operands_are_well_conditioned():
    w = dataclasses.replace(W, bf16=False)
    errs = per_tensor_errors(one_round(w, 1e-7), one_round(w), w.dims)
    assert max(errs) < 2e-6, errs


def test_bf16_operands_amplify_rounding_differences():
    errs = per_tensor_errors(one_round(W, 1e-7), one_round(W), W.dims)
    assert max(errs) > 1e-4, errs
