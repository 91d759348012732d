"""A convolutional worker model, CPU oracle (test infrastructure only).

The paper's workload is ResNet101 on CIFAR-10 (Section "Dataset and DL
Models").  Neither network weights nor the data set are available here, so
the convolutional worker is a small network of the same kind on CIFAR-shaped
inputs, and it is used for throughput and parity, not accuracy:

  s     = relu(conv3x3(x) + b0)                          stem
  u     = relu(conv3x3(s) + b_a)                         residual block
  v     = relu(conv3x3(u) + b_b + s)                     (repeated n_blocks times)
  g     = mean over the H x W positions of v
  logit = g W_f^T + b_f,  softmax cross-entropy.

Every convolution is 3x3 with stride 1 and zero padding 1:
out[b, y, x, o] = sum_{dy, dx, i} W[o, dy, dx, i] * in[b, y + dy - 1, x + dx - 1, i].
Images are NHWC.  The worker's local step is the same plain SGD as for the
MLP (Eq. 4, "otherwise" branch).

Arithmetic (readings, the same rules as the MLP oracle):
* every GEMM operand (weights, stored activations, output gradients, the
  pooled features) passes through ``rnd`` (bf16 rounding for the bf16
  model); activations are stored rounded: s = rnd(relu(.)), likewise u, v;
* products are summed in fp64 and each output rounded once to fp32;
* bias add, the residual add (of the stored s), ReLU and its mask (taken
  from the stored activation) are fp32; pooling sums in fp64 and rounds to
  fp32; softmax and the loss are fp64 (the MLP oracle's softmax_xent);
* backward: dv = (dg / (H W)) broadcast, masked by v > 0; a block's input
  gradient is the transposed convolution of its masked output gradient plus,
  on the skip path, that output gradient as the stored operand rnd(dz_b);
* weight gradients are the fp64 sums over batch and positions of
  rnd(dz) x rnd(input), rounded to fp32; bias gradients the fp64 sums of the
  fp32 dz; the update W <- fp32(W - eta dW) as in the MLP oracle.

Parameters are a flat list in canonical order: W_0 [C, 3, 3, Cin], b_0 [C],
then per block W_a, b_a, W_b, b_b ([C, 3, 3, C], [C]), then W_f [K, C],
b_f [K].
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Callable, List

import numpy as np

from . import model as _mlp

f32, f64 = np.float32, np.float64


def conv3x3(h: np.ndarray, W: np.ndarray, rnd: Callable) -> np.ndarray:
    """fp32( sum over taps of rnd(h shifted) @ rnd(W[:, tap, :]).T ), fp64 sums.
    h [B, H, W, I], W [O, 3, 3, I] -> [B, H, W, O]."""
    B, H, Wd, I = h.shape
    p = np.zeros((B, H + 2, Wd + 2, I), dtype=f64)
    p[:, 1:H + 1, 1:Wd + 1, :] = rnd(h).astype(f64)
    Wr = rnd(W).astype(f64)
    out = np.zeros((B, H, Wd, W.shape[0]), dtype=f64)
    for dy in range(3):
        for dx in range(3):
            out += p[:, dy:dy + H, dx:dx + Wd, :] @ Wr[:, dy, dx, :].T
    return out.astype(f32)


def conv3x3_transposed(dz: np.ndarray, W: np.ndarray, rnd: Callable) -> np.ndarray:
    """Gradient of conv3x3 with respect to its input: dz [B, H, W, O],
    W [O, 3, 3, I] -> [B, H, W, I], fp64 sums rounded to fp32."""
    B, H, Wd, O = dz.shape
    p = np.zeros((B, H + 2, Wd + 2, O), dtype=f64)
    p[:, 1:H + 1, 1:Wd + 1, :] = rnd(dz).astype(f64)
    Wr = rnd(W).astype(f64)
    out = np.zeros((B, H, Wd, W.shape[3]), dtype=f64)
    for dy in range(3):
        for dx in range(3):
            # in[y + dy - 1] received W[., dy, dx, .] * ... from out[y]: out position y = in - dy + 1
            out += p[:, 2 - dy:2 - dy + H, 2 - dx:2 - dx + Wd, :] @ Wr[:, dy, dx, :]
    return out.astype(f32)


def conv3x3_weight_grad(dz: np.ndarray, h: np.ndarray, rnd: Callable) -> np.ndarray:
    """dW[o, dy, dx, i] = sum_{b,y,x} rnd(dz)[b,y,x,o] rnd(h)[b,y+dy-1,x+dx-1,i],
    fp64 sums rounded to fp32."""
    B, H, Wd, I = h.shape
    O = dz.shape[3]
    p = np.zeros((B, H + 2, Wd + 2, I), dtype=f64)
    p[:, 1:H + 1, 1:Wd + 1, :] = rnd(h).astype(f64)
    d = rnd(dz).astype(f64).reshape(-1, O)
    dW = np.zeros((O, 3, 3, I), dtype=f64)
    for dy in range(3):
        for dx in range(3):
            dW[:, dy, dx, :] = d.T @ p[:, dy:dy + H, dx:dx + Wd, :].reshape(-1, I)
    return dW.astype(f32)


@dataclass
class CNN:
    """Shape of the convolutional worker model."""
    height: int = 32
    width: int = 32
    in_ch: int = 3
    ch: int = 64
    blocks: int = 1
    classes: int = 10

    # ------------------------------------------------------------------ layout
    def shapes(self):
        C, K = self.ch, self.classes
        out = [(C, 3, 3, self.in_ch), (C,)]
        for _ in range(self.blocks):
            out += [(C, 3, 3, C), (C,), (C, 3, 3, C), (C,)]
        return out + [(K, C), (K,)]

    def num_params(self) -> int:
        return int(sum(np.prod(s) for s in self.shapes()))

    def flatten(self, params) -> np.ndarray:
        return np.concatenate([np.asarray(p, f32).reshape(-1) for p in params]).astype(f32)

    def unflatten(self, flat) -> List[np.ndarray]:
        out, off = [], 0
        for s in self.shapes():
            n = int(np.prod(s))
            out.append(np.asarray(flat[off:off + n], dtype=f32).reshape(s))
            off += n
        return out

    # ------------------------------------------------------------------ model
    def forward(self, params, X, rnd: Callable):
        """Stored activations (stem output s, per block u and v) and the logits."""
        x = np.asarray(X, f32).reshape(-1, self.height, self.width, self.in_ch)
        W0, b0 = params[0], params[1]
        s = rnd(np.maximum(conv3x3(x, W0, rnd) + b0, f32(0.0)).astype(f32)).astype(f32)
        acts = {"x": x, "s": [s], "u": [], "v": []}
        h = s
        for k in range(self.blocks):
            Wa, ba, Wb, bb = params[2 + 4 * k: 6 + 4 * k]
            u = rnd(np.maximum(conv3x3(h, Wa, rnd) + ba, f32(0.0)).astype(f32)).astype(f32)
            v = rnd(np.maximum((conv3x3(u, Wb, rnd) + bb) + h, f32(0.0)).astype(f32)).astype(f32)
            acts["u"].append(u)
            acts["v"].append(v)
            h = v
        g = (h.astype(f64).sum(axis=(1, 2)) / (self.height * self.width)).astype(f32)
        Wf, bf = params[-2], params[-1]
        logits = (_mlp.gemm_nt(g, Wf, rnd) + bf).astype(f32)
        acts["g"] = g
        return acts, logits

    def gradients(self, params, X, y, rnd: Callable):
        acts, logits = self.forward(params, X, rnd)
        loss, dlog = _mlp.softmax_xent(logits, y)
        grads = [None] * len(params)
        Wf = params[-2]
        grads[-2] = _mlp.gemm_nt(dlog.T, acts["g"].T, rnd)
        grads[-1] = dlog.astype(f64).sum(axis=0).astype(f32)
        dg = _mlp.gemm_nn(dlog, Wf, rnd)                                   # [B, C]
        hw = self.height * self.width
        dh = np.broadcast_to((dg / f32(hw)).astype(f32)[:, None, None, :],
                             acts["s"][0].shape).astype(f32)               # d(pooled map)
        for k in range(self.blocks - 1, -1, -1):
            Wa, ba, Wb, bb = params[2 + 4 * k: 6 + 4 * k]
            h_in = acts["s"][0] if k == 0 else acts["v"][k - 1]
            u, v = acts["u"][k], acts["v"][k]
            dzb = np.where(v > 0, dh, f32(0.0)).astype(f32)
            grads[4 + 4 * k] = conv3x3_weight_grad(dzb, u, rnd)
            grads[5 + 4 * k] = dzb.astype(f64).sum(axis=(0, 1, 2)).astype(f32)
            du = conv3x3_transposed(dzb, Wb, rnd)
            dza = np.where(u > 0, du, f32(0.0)).astype(f32)
            grads[2 + 4 * k] = conv3x3_weight_grad(dza, h_in, rnd)
            grads[3 + 4 * k] = dza.astype(f64).sum(axis=(0, 1, 2)).astype(f32)
            # the block input's gradient: the transposed convolution of dza plus
            # the skip path, which carries dzb as its stored operand
            dh = (conv3x3_transposed(dza, Wa, rnd) + rnd(dzb)).astype(f32)
        dz0 = np.where(acts["s"][0] > 0, dh, f32(0.0)).astype(f32)
        grads[0] = conv3x3_weight_grad(dz0, acts["x"], rnd)
        grads[1] = dz0.astype(f64).sum(axis=(0, 1, 2)).astype(f32)
        return float(loss.mean()), grads

    def sgd_step(self, params, X, y, lr: float, rnd: Callable):
        loss, grads = self.gradients(params, X, y, rnd)
        eta = f64(f32(lr))
        new = [(p.astype(f64) - eta * g.astype(f64)).astype(f32) for p, g in zip(params, grads)]
        return new, loss

    def loss_of(self, params, X, y, rnd: Callable, chunk: int = 256) -> float:
        total, n = 0.0, X.shape[0]
        for s in range(0, n, chunk):
            _, logits = self.forward(params, X[s:s + chunk], rnd)
            loss, _ = _mlp.softmax_xent(logits, y[s:s + chunk])
            total += float(loss.sum())
        return total / n
