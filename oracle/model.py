"""One worker's mini-batch SGD step, CPU oracle (test infrastructure only).

Eq. 4, "otherwise" branch: x_{t+1}^i = x_t^i - eta * g(x_t^i), where g is the
mean mini-batch gradient (Section "Motivation": mini-batch SGD; the paper
names plain SGD and no momentum, weight decay or schedule).  The model is a
ReLU MLP ending in a softmax cross-entropy; with one layer it is softmax
regression.

Arithmetic (readings; the paper fixes no precision):

* every GEMM operand (activation, weight, output gradient) passes through
  ``rnd`` first: ``bf16.round_bf16`` for the bf16-GEMM models, identity for
  the fp32 model;
* products are accumulated in fp64 and each GEMM output is rounded once to
  fp32;
* bias add, ReLU and the ReLU mask are fp32; softmax, log and the loss are
  fp64; dlogits = (p - onehot) / B is rounded to fp32;
* the bias gradient is the fp64 column sum of the fp32 output gradient,
  rounded to fp32;
* the update W <- fp32(W - eta * dW) is evaluated in fp64 and rounded once;
  all parameters (weights and biases) are updated.

Layout: ``layers`` is a list of (W [out, in], b [out]) fp32 arrays.
"""
from __future__ import annotations

from typing import Callable, List, Tuple

import numpy as np

f32, f64 = np.float32, np.float64


def gemm_nt(a: np.ndarray, b: np.ndarray, rnd: Callable) -> np.ndarray:
    """fp32( rnd(a) @ rnd(b).T ), products summed in fp64."""
    return (rnd(a).astype(f64) @ rnd(b).astype(f64).T).astype(f32)


def gemm_nn(a: np.ndarray, b: np.ndarray, rnd: Callable) -> np.ndarray:
    """fp32( rnd(a) @ rnd(b) ), products summed in fp64."""
    return (rnd(a).astype(f64) @ rnd(b).astype(f64)).astype(f32)


def forward(layers, X: np.ndarray, rnd: Callable):
    """Returns (list of layer inputs, list of pre-activations z_l)."""
    inputs, zs = [], []
    h = np.asarray(X, dtype=f32)
    for l, (W, b) in enumerate(layers):
        inputs.append(h)
        z = (gemm_nt(h, W, rnd) + b).astype(f32)
        zs.append(z)
        if l < len(layers) - 1:
            h = np.maximum(z, f32(0.0)).astype(f32)          # ReLU
    return inputs, zs


def softmax_xent(logits: np.ndarray, y: np.ndarray):
    """Per-sample loss -log softmax(logits)[y] and dlogits = (p - onehot)/B."""
    z = logits.astype(f64)
    B = z.shape[0]
    m = z.max(axis=1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(z - m).sum(axis=1))
    loss = lse - z[np.arange(B), y]
    p = np.exp(z - lse[:, None])
    onehot = np.zeros_like(p)
    onehot[np.arange(B), y] = 1.0
    dlogits = ((p - onehot) / B).astype(f32)
    return loss, dlogits


def gradients(layers, X, y, rnd: Callable):
    """Mean mini-batch loss and per-layer (dW, db) by backpropagation."""
    inputs, zs = forward(layers, X, rnd)
    loss, dz = softmax_xent(zs[-1], y)
    grads: List[Tuple[np.ndarray, np.ndarray]] = [None] * len(layers)
    for l in range(len(layers) - 1, -1, -1):
        W, _ = layers[l]
        dW = gemm_nt(dz.T, inputs[l].T, rnd)                 # dz^T @ h_l
        db = dz.astype(f64).sum(axis=0).astype(f32)
        grads[l] = (dW, db)
        if l > 0:
            dh = gemm_nn(dz, W, rnd)                                     # dz @ W
            dz = np.where(zs[l - 1] > 0, dh, f32(0.0)).astype(f32)      # ReLU mask
    return float(loss.mean()), grads


def sgd_update(layers, grads, lr: float):
    """W <- fp32(W - eta * dW) for every weight and bias."""
    eta = f64(f32(lr))
    return [((W.astype(f64) - eta * dW.astype(f64)).astype(f32),
             (b.astype(f64) - eta * db.astype(f64)).astype(f32))
            for (W, b), (dW, db) in zip(layers, grads)]


def sgd_step(layers, X, y, lr: float, rnd: Callable):
    """One local iteration of one worker.  Returns (new layers, batch loss)."""
    loss, grads = gradients(layers, X, y, rnd)
    return sgd_update(layers, grads, lr), loss


def loss_of(layers, X, y, rnd: Callable, chunk: int = 1024) -> float:
    """Mean cross-entropy of a model on a data set (forward only)."""
    total, n = 0.0, X.shape[0]
    for s in range(0, n, chunk):
        _, zs = forward(layers, X[s:s + chunk], rnd)
        loss, _ = softmax_xent(zs[-1], y[s:s + chunk])
        total += float(loss.sum())
    return total / n
