"""Plausible implementation mistakes planted in the oracle (CPU, test
infrastructure only), to show that the parity bounds of the multi-step bf16
tests would catch them.  Each mutant is a context manager that swaps one
oracle function for a wrong variant and restores it on exit:

* ``stale_operand``: within a worker's round the GEMMs keep seeing the
  weights of the pull (the bf16 operand copy is not refreshed after step 0),
  while the fp32 master is updated;
* ``bias_frozen``: the SGD step updates the weights but not the biases;
* ``sample_dropped``: the last row of every mini-batch is left out;
* ``cursor_ahead``: every mini-batch starts one batch after the cursor.
"""
from __future__ import annotations

import contextlib

import numpy as np

from oracle import model as omodel
from oracle import run as orun


@contextlib.contextmanager
def _swap(module, name, fn):
    real = getattr(module, name)
    setattr(module, name, fn)
    try:
        yield
    finally:
        setattr(module, name, real)


def _loop(state, worker, shard, batch, lr, rnd, rows, step):
    """A worker's round with the mini-batch rows chosen by ``rows(cursor)``
    and each step done by ``step(layers, X, y, s)``."""
    X, y = shard
    layers = [(W.copy(), b.copy()) for W, b in state.x_g]
    losses = []
    for s in range(int(state.tau[worker])):
        idx = rows(int(state.cursor[worker]), X.shape[0])
        state.cursor[worker] = (state.cursor[worker] + batch) % X.shape[0]
        layers, loss = step(layers, X[idx], y[idx], s)
        losses.append(loss)
    return layers, float(np.mean(losses))


def stale_operand():
    def local_steps(state, worker, shard, batch, lr, rnd):
        pulled = [W.copy() for W, _ in state.x_g]

        def step(layers, Xb, yb, s):
            seen = [(Wp, b) for Wp, (_, b) in zip(pulled, layers)]
            loss, grads = omodel.gradients(seen, Xb, yb, rnd)
            return omodel.sgd_update(layers, grads, lr), loss
        return _loop(state, worker, shard, batch, lr, rnd, lambda c, n: orun.batch_indices(c, batch, n), step)
    return _swap(orun, "local_steps", local_steps)


def bias_frozen():
    real = omodel.sgd_update

    def sgd_update(layers, grads, lr):
        return [(Wn, b) for (Wn, _), (_, b) in zip(real(layers, grads, lr), layers)]
    return _swap(omodel, "sgd_update", sgd_update)


def sample_dropped():
    def local_steps(state, worker, shard, batch, lr, rnd):
        def step(layers, Xb, yb, s):
            return omodel.sgd_step(layers, Xb, yb, lr, rnd)
        return _loop(state, worker, shard, batch, lr, rnd,
                     lambda c, n: orun.batch_indices(c, batch, n)[:-1], step)
    return _swap(orun, "local_steps", local_steps)


def cursor_ahead():
    def local_steps(state, worker, shard, batch, lr, rnd):
        def step(layers, Xb, yb, s):
            return omodel.sgd_step(layers, Xb, yb, lr, rnd)
        return _loop(state, worker, shard, batch, lr, rnd,
                     lambda c, n: orun.batch_indices(c + batch, batch, n), step)
    return _swap(orun, "local_steps", local_steps)


MUTANTS = {"stale_operand": stale_operand, "bias_frozen": bias_frozen, "sample_dropped": sample_dropped,
           "cursor_ahead": cursor_ahead}
