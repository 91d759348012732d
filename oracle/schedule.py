"""Oscars scheduler, CPU oracle (test infrastructure only).

Follows the paper's Problem Formulation and Algorithm 1:

* t_i^iter, the time of one local iteration of worker i (notation table).
* Eq. 1: the idle time of worker i before a barrier T is t_i^w = mod(T, t_i^iter).
* Eq. 2: the maximum wait max_i mod(T, t_i^iter).
* Eq. 3: T* = argmin_T max_i mod(T, t_i) subject to
  floor(T / min t) - floor(T / max t) < M.
* tau_i = floor(T* / t_i^iter): the number of local steps of worker i
  (the sentence after Eq. 3; Section "Local-SGD load balancing").
* Algorithm 1: start at T = max(t), evaluate Eq. 2 for T, T+1, ... while the
  constraint of Eq. 3 holds, keep the T with the smallest maximum wait.

Readings where the paper is silent or ambiguous:

* Speed factors map to integer ticks as t_i = max(1, floor(Q / s_i + 0.5)),
  Q ticks per unit-speed step (Q = 1000 by default); s_i is a relative
  throughput, larger is faster.  The paper's ``T++`` implies integer time.
* The initial T = max(t) is always a candidate (do-while): otherwise the
  candidate set can be empty.
* The constraint is strict (< M) in integer floor division.
* Ties keep the first (smallest) T.
* Termination: with all t_i equal the constraint never fails, so the default
  ("capped") search also stops once T > M * max(t).  The "literal" search has
  no cap and is only defined when min(t) < max(t).

The comparison schemes of the paper's Introduction and Motivation share the
round structure and differ only in the local-step counts:

* BSP: a barrier after every iteration, tau_i = 1;
* Local SGD with a fixed period I: every worker runs I iterations between
  averages, tau_i = I, and the fast workers wait for the slowest;
* Oscars: tau_i from Algorithm 1.

A round ends when the last worker has pushed, at B = max_i tau_i * t_i, and
worker i idles for B - tau_i * t_i.  For Algorithm 1's counts B equals T*:
with all waits mod(T*, t_i) > 0 the barrier max_i tau_i t_i would be an
earlier candidate with strictly smaller waits, so some worker has no wait.
"""
from __future__ import annotations

from typing import List, Tuple

import numpy as np

CAPPED = 0
LITERAL = 1


def iteration_ticks(speeds, ticks_per_unit: int = 1000) -> np.ndarray:
    """t_i^iter in integer ticks from speed factors (fp64 once, then int64)."""
    s = np.asarray(speeds, dtype=np.float64)
    if np.any(~(s > 0)):
        raise ValueError("speed factors must be > 0")
    t = np.floor(np.float64(ticks_per_unit) / s + 0.5)
    return np.maximum(t, 1.0).astype(np.int64)


def wait_times(t_iter, T: int) -> np.ndarray:
    """Eq. 1: t_i^w = mod(T, t_i^iter) for every worker."""
    return np.int64(T) % np.asarray(t_iter, dtype=np.int64)


def max_wait(t_iter, T: int) -> int:
    """Eq. 2: the maximum wait over workers at barrier T."""
    return int(np.max(wait_times(t_iter, T)))


def constraint_holds(t_iter, T: int, M: int) -> bool:
    """Constraint of Eq. 3: floor(T/min t) - floor(T/max t) < M."""
    t = np.asarray(t_iter, dtype=np.int64)
    return (T // int(t.min())) - (T // int(t.max())) < M


def load_balance_search(t_iter, M: int, mode: int = CAPPED) -> Tuple[int, int, List[Tuple[int, int]]]:
    """Algorithm 1.  Returns (T*, max wait at T*, [(T, max wait)] trace)."""
    t = np.asarray(t_iter, dtype=np.int64)
    if t.size == 0 or np.any(t < 1):
        raise ValueError("iteration times must be >= 1")
    if M < 1:
        raise ValueError("M must be >= 1")
    tmax = int(t.max())
    if mode == LITERAL and int(t.min()) == tmax:
        raise ValueError("literal search does not terminate when all t_i are equal")
    T = tmax                              # Initial: T = max(t_i^iter)
    T_set: List[int] = []
    max_wait_time: List[int] = []
    while True:
        tw = [int(T % int(tj)) for tj in t]        # t^w[j] = mod(T, t_j^iter)
        max_wait_time.append(max(tw))             # max_wait_time[i] = max(t^w)
        T_set.append(T)                           # T_set[i] = T
        T += 1                                    # T++
        if not constraint_holds(t, T, M):         # loop condition of Algorithm 1
            break
        if mode == CAPPED and T > M * tmax:
            break
    best = int(np.argmin(np.asarray(max_wait_time)))   # first minimum
    return T_set[best], max_wait_time[best], list(zip(T_set, max_wait_time))


def local_steps(t_iter, T_star: int) -> np.ndarray:
    """tau_i = floor(T* / t_i^iter), int32."""
    return (np.int64(T_star) // np.asarray(t_iter, dtype=np.int64)).astype(np.int32)


def schedule(t_iter, M: int, mode: int = CAPPED):
    """(T*, max wait, tau) of the load-balanced semi-synchronous round."""
    T_star, mw, _ = load_balance_search(t_iter, M, mode)
    return T_star, mw, local_steps(t_iter, T_star)


OSCARS = "oscars"
BSP = "bsp"
LOCAL_SGD = "local_sgd"


def round_barrier(t_iter, tau) -> int:
    """Length of a round in ticks: the time of the last push, max_i tau_i t_i."""
    return int(np.max(np.asarray(tau, dtype=np.int64) * np.asarray(t_iter, dtype=np.int64)))


def policy_local_steps(policy: str, t_iter, M: int = 1, period: int = 1, mode: int = CAPPED):
    """(tau, barrier) of one round under a synchronisation scheme: "oscars"
    (Algorithm 1), "bsp" (tau_i = 1) or "local_sgd" (tau_i = period)."""
    t = np.asarray(t_iter, dtype=np.int64)
    if t.size == 0 or np.any(t < 1):
        raise ValueError("iteration times must be >= 1")
    if policy == OSCARS:
        T_star, _, tau = schedule(t, M, mode)
        return tau, int(T_star)
    if policy == BSP:
        tau = np.ones(t.size, dtype=np.int32)
    elif policy == LOCAL_SGD:
        if period < 1:
            raise ValueError("the local-SGD period must be >= 1")
        tau = np.full(t.size, period, dtype=np.int32)
    else:
        raise ValueError(policy)
    return tau, round_barrier(t, tau)


def merge_weights(rule: str, tau, explicit=None) -> np.ndarray:
    """Per-worker merge weights as fp32.

    * "uniform": w_k = 1/N, the average of Eq. 4 (first branch).
    * "localsteps": w_k = tau_k / sum_j tau_j.  NOT in the paper; a
      non-uniform rule used by the merge microbench.
    * "explicit": the caller's weights.
    Computed in fp64 and rounded once to fp32.
    """
    tau = np.asarray(tau, dtype=np.int64)
    n = tau.size
    if rule == "uniform":
        return np.full(n, np.float32(1.0 / n), dtype=np.float32)
    if rule == "localsteps":
        return (tau.astype(np.float64) / float(tau.sum())).astype(np.float32)
    if rule == "explicit":
        return np.asarray(explicit, dtype=np.float32)
    raise ValueError(rule)
