"""The Oscars round loop, CPU oracle (test infrastructure only).

Reading of Eq. 4 (its condition ``t mod tau_i = 0`` is per worker while its
average is global): training proceeds in rounds.  In every round each worker
i starts from the global model (pull), runs exactly tau_i local SGD steps on
its own data ("otherwise" branch), pushes its model, and at the barrier T*
the server replaces the global model with the merge of the pushed models
(first branch).  Speeds are steady (Section "Problem Formulation"), so T* and
tau are computed once; synchronisation time is ignored, so the simulated
clock of worker i advances by tau_i * t_i of compute and mod(T*, t_i) of idle
time (Eq. 1) per round.  Under the comparison schemes (BSP, local SGD with a
fixed period, or any tau given by the caller) the round ends at the last
push, max_i tau_i * t_i, which for Algorithm 1's tau is T* itself.

Mini-batches (a reading; the data-partition section of the paper is empty):
worker i reads its shard sequentially from a cursor that persists across
rounds and wraps modulo the shard size.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable, List, Optional, Sequence, Tuple

import numpy as np

from . import bf16 as _bf16
from . import merge as _merge
from . import model as _model
from . import schedule as _sched


def flatten(layers) -> np.ndarray:
    """Canonical flat vector W_0, b_0, W_1, b_1, ... (fp32)."""
    return np.concatenate([np.concatenate([W.reshape(-1), b.reshape(-1)]) for W, b in layers]).astype(np.float32)


def unflatten(flat: np.ndarray, dims: Sequence[int]):
    out, off = [], 0
    for i, o in zip(dims[:-1], dims[1:]):
        W = np.asarray(flat[off:off + o * i], dtype=np.float32).reshape(o, i); off += o * i
        b = np.asarray(flat[off:off + o], dtype=np.float32); off += o
        out.append((W, b))
    return out


class MLPModel:
    """The MLP of ``oracle.model`` behind the interface the round loop uses
    (flatten, unflatten, sgd_step, loss_of); ``oracle.conv.CNN`` offers the
    same interface for the convolutional worker."""

    def __init__(self, dims: Sequence[int]):
        self.dims = list(dims)

    def flatten(self, layers):
        return flatten(layers)

    def unflatten(self, flat):
        return unflatten(flat, self.dims)

    def sgd_step(self, layers, X, y, lr, rnd):
        return _model.sgd_step(layers, X, y, lr, rnd)

    def loss_of(self, layers, X, y, rnd):
        return _model.loss_of(layers, X, y, rnd)


def _copy(params):
    return [tuple(a.copy() for a in p) if isinstance(p, tuple) else p.copy() for p in params]


def batch_indices(cursor: int, batch: int, n: int) -> np.ndarray:
    return (cursor + np.arange(batch, dtype=np.int64)) % n


@dataclass
class RoundRecord:
    tau: np.ndarray
    T_star: int
    worker_loss: np.ndarray          # mean mini-batch loss of each worker this round
    idle: np.ndarray                 # idle ticks of each worker this round (Eq. 1)
    x_g: Optional[np.ndarray] = None # global model after the merge (flat, fp32)
    eval_loss: Optional[float] = None
    replicas: Optional[list] = None  # the pushed models (flat), when asked for


@dataclass
class OscarsState:
    dims: List[int]
    x_g: list                # the global model's parameters (the model's own structure)
    cursor: np.ndarray
    clock: np.ndarray
    idle: np.ndarray
    t_iter: np.ndarray
    T_star: int          # the round's barrier: T* of Algorithm 1, else max_i tau_i t_i
    max_wait: int
    tau: np.ndarray
    model: object = None


def init_state(dims, layers0, t_iter, M: int, mode: int = _sched.CAPPED, tau_override=None,
               model=None) -> OscarsState:
    T_star, mw, tau = _sched.schedule(t_iter, M, mode)
    if tau_override is not None:
        tau = np.asarray(tau_override, dtype=np.int32)
        T_star = _sched.round_barrier(t_iter, tau)
        mw = int(np.max(T_star - tau.astype(np.int64) * np.asarray(t_iter, np.int64)))
    W = len(t_iter)
    return OscarsState(list(dims) if dims is not None else [], _copy(layers0),
                       np.zeros(W, np.int64), np.zeros(W, np.int64), np.zeros(W, np.int64),
                       np.asarray(t_iter, np.int64), T_star, mw, tau,
                       model if model is not None else MLPModel(dims))


def reschedule(state: OscarsState, t_iter, M: int, mode: int = _sched.CAPPED) -> None:
    """New iteration times (drifting speeds): Algorithm 1 again for the
    following rounds; the clocks keep what they have accumulated."""
    T_star, mw, tau = _sched.schedule(t_iter, M, mode)
    state.t_iter = np.asarray(t_iter, np.int64)
    state.T_star, state.max_wait, state.tau = T_star, mw, tau


def local_steps(state: OscarsState, worker: int, shard, batch: int, lr: float, rnd: Callable):
    """Worker ``worker`` pulls the global model and runs tau_i local SGD steps."""
    X, y = shard
    layers = _copy(state.x_g)                                      # pull
    losses = []
    for _ in range(int(state.tau[worker])):
        idx = batch_indices(int(state.cursor[worker]), batch, X.shape[0])
        state.cursor[worker] = (state.cursor[worker] + batch) % X.shape[0]
        layers, loss = state.model.sgd_step(layers, X[idx], y[idx], lr, rnd)
        losses.append(loss)
    return layers, float(np.mean(losses))


def run_round(state: OscarsState, shards, batch: int, lr: float, rnd: Callable,
              weight_rule: str = "uniform", server_lr: float = 1.0, weights=None,
              keep_replicas: bool = False) -> RoundRecord:
    W = len(shards)
    models, wl = [], np.zeros(W)
    for i in range(W):
        layers, wl[i] = local_steps(state, i, shards[i], batch, lr, rnd)
        models.append(state.model.flatten(layers))                 # push
    w = _sched.merge_weights(weight_rule, state.tau, weights)
    x_new = _merge.merge_models(state.model.flatten(state.x_g), models, w, server_lr)
    state.x_g = state.model.unflatten(x_new)
    idle = state.T_star - state.tau.astype(np.int64) * state.t_iter     # = mod(T*, t_i) under Algorithm 1
    state.clock += state.tau.astype(np.int64) * state.t_iter + idle
    state.idle += idle
    return RoundRecord(state.tau.copy(), state.T_star, wl, idle, x_new,
                       replicas=models if keep_replicas else None)


def run(dims, layers0, shards, speeds=None, t_iter=None, M: int = 8, rounds: int = 1,
        batch: int = 32, lr: float = 0.05, bf16: bool = True, weight_rule: str = "uniform",
        server_lr: float = 1.0, mode: int = _sched.CAPPED, tau_override=None,
        eval_set=None, ticks_per_unit: int = 1000, target_loss=None, t_per_round=None, model=None,
        keep_replicas: bool = False):
    """Run ``rounds`` rounds; returns (final state, [RoundRecord]).  With an
    eval set and a target loss, stop after the first round whose eval loss
    is at or below the target.  ``t_per_round[r]`` (optional): iteration
    times in force from round r on (drifting speeds), re-solved with
    Algorithm 1 before that round.  ``keep_replicas``: every record also
    holds the W pushed models of its round."""
    if t_iter is None:
        t_iter = t_per_round[0] if t_per_round is not None else _sched.iteration_ticks(speeds, ticks_per_unit)
    rnd = _bf16.round_bf16 if bf16 else _bf16.identity
    state = init_state(dims, layers0, t_iter, M, mode, tau_override, model)
    records = []
    for r in range(rounds):
        if t_per_round is not None and r > 0:
            reschedule(state, t_per_round[r], M, mode)
        rec = run_round(state, shards, batch, lr, rnd, weight_rule, server_lr, keep_replicas=keep_replicas)
        if eval_set is not None:
            rec.eval_loss = state.model.loss_of(state.x_g, eval_set[0], eval_set[1], rnd)
        records.append(rec)
        if target_loss is not None and rec.eval_loss is not None and rec.eval_loss <= target_loss:
            break
    return state, records


def time_to_loss(records, target: float):
    """Simulated ticks until the global model's eval loss first reaches
    ``target`` (None if it never does): every round lasts its barrier."""
    ticks = 0
    for rec in records:
        ticks += int(rec.T_star)
        if rec.eval_loss is not None and rec.eval_loss <= target:
            return ticks
    return None
