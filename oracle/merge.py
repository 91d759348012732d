"""Server merge and global update, CPU oracle (test infrastructure only).

Eq. 4, first branch: at the barrier the new model is the average of the
workers' models after their last local step, (1/N) sum_k (x^k - eta g(x^k)).
The parameter-server description (Section "Introduction") has the workers
push, the server combine and update, and the workers pull the result.

Delta form (a reading): x_g' = x_g + eta_s * sum_k w_k * (x^k - x_g).  With
w_k = 1/N and eta_s = 1 this equals the average of Eq. 4 in exact arithmetic.
The sum runs in fp64 in worker order k = 0..W-1 and is rounded once to fp32.
"""
from __future__ import annotations

from typing import Sequence

import numpy as np


def merge_deltas(x_g: np.ndarray, deltas: Sequence[np.ndarray], weights, server_lr: float = 1.0) -> np.ndarray:
    """x_g' = fp32(x_g + eta_s * sum_k w_k * delta_k), fp64 sum in order k."""
    acc = np.zeros(np.shape(x_g), dtype=np.float64)
    for k, d in enumerate(deltas):
        acc += np.float64(np.float32(weights[k])) * np.asarray(d, dtype=np.float64)
    eta = np.float64(np.float32(server_lr))
    return (np.asarray(x_g, dtype=np.float64) + eta * acc).astype(np.float32)


def merge_models(x_g: np.ndarray, models: Sequence[np.ndarray], weights, server_lr: float = 1.0) -> np.ndarray:
    """Same update with pushed models: delta_k = x^k - x_g, formed in fp64."""
    xg64 = np.asarray(x_g, dtype=np.float64)
    return merge_deltas(x_g, [np.asarray(m, dtype=np.float64) - xg64 for m in models], weights, server_lr)


def average(models: Sequence[np.ndarray]) -> np.ndarray:
    """Eq. 4 as printed: (1/N) sum_k x^k, fp64, rounded once to fp32."""
    acc = np.zeros(np.shape(models[0]), dtype=np.float64)
    for m in models:
        acc += np.asarray(m, dtype=np.float64)
    return (acc / len(models)).astype(np.float32)
