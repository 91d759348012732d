"""Pins for the oracle worker step (Eq. 4, "otherwise" branch): bf16 rounding
against torch's conversion, the softmax-cross-entropy gradient and full MLP
backpropagation against fp64 finite differences, and the SGD direction."""
import math

import numpy as np
import pytest
import torch

from oracle import bf16, model


def test_bf16_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-30).astype(np.float32),
        (rng.standard_normal(2000) * 1e30).astype(np.float32),
        np.array([0.0, -0.0, 1.0, -1.0, 1.00390625, 1.01171875, 3.0e38], dtype=np.float32),
    ])
    # exact ties: low half == 0x8000 with both parities of the kept LSB
    ties = (np.arange(1000, dtype=np.uint32) << 16 | 0x8000).view(np.float32)
    x = np.concatenate([x, ties, -ties])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(bf16.round_bf16(x), ref)


def ce_loss64(logits, y):
    z = logits.astype(np.float64)
    m = z.max(1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(z - m).sum(1))
    return float((lse - z[np.arange(len(y)), y]).mean())


def test_softmax_xent_gradient_finite_difference():
    rng = np.random.default_rng(1)
    B, C = 6, 10
    z = rng.standard_normal((B, C)) * 3
    y = rng.integers(0, C, B)
    loss, d = model.softmax_xent(z.astype(np.float32), y)
    assert abs(loss.mean() - ce_loss64(z.astype(np.float32), y)) < 1e-12
    h = 1e-6
    num = np.zeros_like(z)
    for i in range(B):
        for j in range(C):
            zp, zm = z.copy(), z.copy()
            zp[i, j] += h
            zm[i, j] -= h
            num[i, j] = (ce_loss64(zp, y) - ce_loss64(zm, y)) / (2 * h)
    np.testing.assert_allclose(d, num, rtol=2e-5, atol=1e-8)


def mlp_loss64(layers, X, y):
    """fp64 forward without any rounding (for finite differences)."""
    h = X.astype(np.float64)
    for l, (W, b) in enumerate(layers):
        z = h @ W.T + b
        h = np.maximum(z, 0) if l < len(layers) - 1 else z
    return ce_loss64(h, y)


@pytest.mark.parametrize("dims", [[7, 10], [5, 6, 10], [6, 9, 7, 10]])
def test_mlp_gradients_finite_difference(dims):
    rng = np.random.default_rng(len(dims))
    layers = [((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32),
               (rng.standard_normal(o) * 0.1).astype(np.float32))
              for i, o in zip(dims[:-1], dims[1:])]
    X = rng.standard_normal((5, dims[0])).astype(np.float32)
    y = rng.integers(0, 10, 5)
    _, grads = model.gradients(layers, X, y, bf16.identity)
    h = 1e-3
    for l, (W, b) in enumerate(layers):
        for P, G in ((W, grads[l][0]), (b, grads[l][1])):
            num = np.zeros(P.shape)
            for idx in np.ndindex(P.shape):
                base = [(w.astype(np.float64), c.astype(np.float64)) for w, c in layers]
                plus = [(w.copy(), c.copy()) for w, c in base]
                minus = [(w.copy(), c.copy()) for w, c in base]
                tgt_p = plus[l][0] if P is W else plus[l][1]
                tgt_m = minus[l][0] if P is W else minus[l][1]
                tgt_p[idx] += h
                tgt_m[idx] -= h
                num[idx] = (mlp_loss64(plus, X, y) - mlp_loss64(minus, X, y)) / (2 * h)
            np.testing.assert_allclose(G, num, rtol=2e-3, atol=2e-5)


def test_bf16_step_close_to_fp32_step():
    rng = np.random.default_rng(3)
    dims = [32, 48, 10]
    layers = [((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32), np.zeros(o, np.float32))
              for i, o in zip(dims[:-1], dims[1:])]
    X = rng.standard_normal((16, 32)).astype(np.float32)
    y = rng.integers(0, 10, 16)
    l32, g32 = model.gradients(layers, X, y, bf16.identity)
    l16, g16 = model.gradients(layers, X, y, bf16.round_bf16)
    assert abs(l32 - l16) < 2e-2 * abs(l32)
    # a ReLU mask may flip for pre-activations near zero (one flip moves a
    # whole row of the first layer's gradient), so compare norms loosely
    (a0, _), (a1, _) = g32
    (b0, _), (b1, _) = g16
    assert np.linalg.norm(a1 - b1) < 1e-2 * np.linalg.norm(a1)
    assert np.linalg.norm(a0 - b0) < 0.15 * np.linalg.norm(a0)


def test_sgd_step_decreases_loss():
    rng = np.random.default_rng(4)
    dims = [20, 16, 10]
    layers = [((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32), np.zeros(o, np.float32))
              for i, o in zip(dims[:-1], dims[1:])]
    X = rng.standard_normal((32, 20)).astype(np.float32)
    y = rng.integers(0, 10, 32)
    before = mlp_loss64(layers, X, y)
    new, loss = model.sgd_step(layers, X, y, 0.05, bf16.identity)
    assert abs(loss - before) < 1e-5
    assert mlp_loss64(new, X, y) < before


# ---------------------------------------------------------------- bf16 operand placement (reading R12)
# Every GEMM operand (input X, each weight W_l, each output gradient dz_l) is
# rounded to bf16 before its product; the bias gradient sums the fp32 output
# gradient.  Moving an operand's fp32 values inside their bf16 rounding
# intervals must therefore leave every product, and so the loss and the
# weight gradients, bit for bit unchanged; moving them across a boundary
# must change them.  A rounding dropped from any operand of any product, or
# added to the bias gradient, fails one of these.

PIN_DIMS = [24, 40, 32, 10]   # two hidden layers: two hidden output gradients


def _pin_setup(seed=7):
    rng = np.random.default_rng(seed)
    layers = [((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32),
               (rng.standard_normal(o) * 0.1).astype(np.float32))
              for i, o in zip(PIN_DIMS[:-1], PIN_DIMS[1:])]
    X = rng.standard_normal((16, PIN_DIMS[0])).astype(np.float32)
    y = rng.integers(0, 10, 16)
    return layers, X, y


def _bf16_step(r):
    """Distance from the bf16 value r to its upper neighbour (the fp32 spacing
    scaled by the 16 dropped mantissa bits); the lower neighbour is at least
    half as far."""
    return np.spacing(np.abs(r).astype(np.float32)) * np.float32(65536.0)


def inside_bf16(x, seed=0):
    """fp32 values that round to the same bf16 values as x, almost all of
    them different from x (moved by up to a fifth of the bf16 step)."""
    r = bf16.round_bf16(x)
    u = np.random.default_rng(seed).uniform(-1.0, 1.0, np.shape(x))
    out = (r + np.float32(0.2) * _bf16_step(r) * u).astype(np.float32)
    assert np.array_equal(bf16.round_bf16(out), r)
    assert np.mean(out != np.asarray(x, np.float32)) > 0.9
    return out


def across_bf16(x):
    """x scaled by 1 + 2^-6: every non-zero value lands on another bf16 value."""
    out = (np.asarray(x, np.float32) * np.float32(1.015625)).astype(np.float32)
    nz = np.asarray(x) != 0
    assert np.all(bf16.round_bf16(out)[nz] != bf16.round_bf16(x)[nz])
    return out


def _same(a, b):
    la, ga = a
    lb, gb = b
    return la == lb and all(np.array_equal(p, q) for g, h in zip(ga, gb) for p, q in zip(g, h))


def test_gradients_see_the_input_only_as_bf16():
    layers, X, y = _pin_setup()
    base = model.gradients(layers, X, y, bf16.round_bf16)
    assert _same(model.gradients(layers, inside_bf16(X), y, bf16.round_bf16), base)
    moved = model.gradients(layers, across_bf16(X), y, bf16.round_bf16)
    assert not np.array_equal(moved[1][0][0], base[1][0][0])        # dW_0 = dz_0^T X changes


@pytest.mark.parametrize("l", [0, 1, 2])
def test_gradients_see_each_weight_only_as_bf16(l):
    """W_l enters the forward product and the input-gradient product."""
    layers, X, y = _pin_setup()
    base = model.gradients(layers, X, y, bf16.round_bf16)
    inside = [(W.copy(), b.copy()) for W, b in layers]
    inside[l] = (inside_bf16(layers[l][0], seed=l), layers[l][1])
    assert _same(model.gradients(inside, X, y, bf16.round_bf16), base)
    across = [(W.copy(), b.copy()) for W, b in layers]
    across[l] = (across_bf16(layers[l][0]), layers[l][1])
    moved = model.gradients(across, X, y, bf16.round_bf16)
    assert moved[0] != base[0]                                        # the forward product moved
    if l > 0:                                                         # and the input-gradient product
        assert not np.array_equal(moved[1][l - 1][0], base[1][l - 1][0])


def test_output_gradients_enter_both_products_as_bf16_and_the_bias_sum_as_fp32(monkeypatch):
    """dz of the last layer (softmax output) and of each hidden layer (the
    masked input-gradient product) moved inside their bf16 intervals: every
    weight gradient is unchanged, the bias gradient of that layer changes.
    Moved across: the weight gradient of that layer changes."""
    layers, X, y = _pin_setup()
    base = model.gradients(layers, X, y, bf16.round_bf16)
    L = len(layers)
    real_xent, real_nn = model.softmax_xent, model.gemm_nn

    def run(move_last=None, move_hidden=None):
        def xent(z, yy):
            loss, d = real_xent(z, yy)
            return loss, (move_last(d) if move_last else d)
        calls = []

        def nn(a, b, rnd):                     # dh_{l-1} = dz_l @ W_l, from the top layer down
            out = real_nn(a, b, rnd)
            calls.append(out.shape)
            layer_below = L - 1 - len(calls)
            return move_hidden(out) if move_hidden and move_hidden.layer == layer_below else out
        monkeypatch.setattr(model, "softmax_xent", xent)
        monkeypatch.setattr(model, "gemm_nn", nn)
        try:
            return model.gradients(layers, X, y, bf16.round_bf16)
        finally:
            monkeypatch.setattr(model, "softmax_xent", real_xent)
            monkeypatch.setattr(model, "gemm_nn", real_nn)

    got = run(move_last=lambda d: inside_bf16(d, seed=3))
    for l in range(L):
        assert np.array_equal(got[1][l][0], base[1][l][0]), l
    assert not np.array_equal(got[1][L - 1][1], base[1][L - 1][1])
    for l in range(L - 1):
        assert np.array_equal(got[1][l][1], base[1][l][1]), l
    got = run(move_last=across_bf16)
    assert not np.array_equal(got[1][L - 1][0], base[1][L - 1][0])

    for layer in range(L - 1):
        def inside(d, layer=layer):
            return inside_bf16(d, seed=10 + layer)
        inside.layer = layer
        got = run(move_hidden=inside)
        for l in range(L):
            assert np.array_equal(got[1][l][0], base[1][l][0]), (layer, l)
        assert not np.array_equal(got[1][layer][1], base[1][layer][1]), layer
        across = lambda d: across_bf16(d)  # noqa: E731
        across.layer = layer
        got = run(move_hidden=across)
        assert not np.array_equal(got[1][layer][0], base[1][layer][0]), layer


# ---------------------------------------------------------------- the SGD update (reading R10)
def test_sgd_step_by_hand_zero_model():
    """2 classes, 2 inputs, one sample, zero model: p = (1/2, 1/2), so
    dz = p - onehot(0) = (-1/2, 1/2), dW = dz x^T, db = dz, and with
    eta = fp32(0.05) the new weights are -eta * dW, the new biases -eta * db
    (every product exact in fp64, one rounding to fp32)."""
    X = np.array([[1.0, 2.0]], np.float32)
    layers = [(np.zeros((2, 2), np.float32), np.zeros(2, np.float32))]
    new, loss = model.sgd_step(layers, X, np.array([0]), 0.05, bf16.identity)
    eta = float(np.float32(0.05))
    assert loss == math.log(2.0)
    np.testing.assert_array_equal(new[0][0], np.float32([[0.5 * eta, 1.0 * eta], [-0.5 * eta, -1.0 * eta]]))
    np.testing.assert_array_equal(new[0][1], np.float32([0.5 * eta, -0.5 * eta]))


def test_sgd_step_by_hand_closed_form():
    """W = [[1, 0], [0, 0]], b = (0, 1/2), x = (1, 3), label 1: logits
    (1, 1/2), so p_0 = s = 1 / (1 + e^{-1/2}), dz = (s, -s),
    loss = log(1 + e^{1/2}), dW = dz x^T, db = dz; W' = W - eta dW and
    b' = b - eta db, each rounded once to fp32 (dz rounded to fp32 first)."""
    X = np.array([[1.0, 3.0]], np.float32)
    layers = [(np.array([[1.0, 0.0], [0.0, 0.0]], np.float32), np.array([0.0, 0.5], np.float32))]
    new, loss = model.sgd_step(layers, X, np.array([1]), 0.05, bf16.identity)
    s = 1.0 / (1.0 + math.exp(-0.5))
    dz = [float(np.float32(s)), float(np.float32(-s))]
    eta = float(np.float32(0.05))
    W0 = [[1.0, 0.0], [0.0, 0.0]]
    xs = [1.0, 3.0]
    dW = [[float(np.float32(dz[c] * xs[k])) for k in range(2)] for c in range(2)]
    W_new = np.float32([[W0[c][k] - eta * dW[c][k] for k in range(2)] for c in range(2)])
    b_new = np.float32([0.0 - eta * dz[0], 0.5 - eta * dz[1]])
    assert abs(loss - math.log1p(math.exp(0.5))) <= 4e-16
    np.testing.assert_array_equal(new[0][0], W_new)
    np.testing.assert_array_equal(new[0][1], b_new)


# ---------------------------------------------------------------- eval loss in chunks (reading R14)
@pytest.mark.parametrize("chunk", [1024, 7, 5000])
def test_loss_of_closed_form_across_chunk_boundaries(chunk):
    """Softmax regression with logits (a_i, 0), label 0: the per-sample loss is
    log(1 + e^{-a_i}).  The first 1024 samples have a = 0 (loss log 2), the
    remaining 1476 (two chunk boundaries and a ragged tail at chunk 1024) have
    a = 3, so a dropped chunk, a lost tail or a wrong divisor shows."""
    n, head = 2500, 1024
    X = np.zeros((n, 4), np.float32)
    X[head:, 0] = 3.0
    y = np.zeros(n, np.int64)
    layers = [(np.array([[1.0, 0, 0, 0], [0, 0, 0, 0]], np.float32), np.zeros(2, np.float32))]
    want = (head * math.log(2.0) + (n - head) * math.log1p(math.exp(-3.0))) / n
    got = model.loss_of(layers, X, y, bf16.identity, chunk=chunk)
    assert abs(got - want) <= 1e-12 * want
    logits = X @ layers[0][0].T
    assert abs(model.loss_of(layers, X, y, bf16.round_bf16, chunk=chunk) - ce_loss64(logits, y)) <= 1e-12 * want
