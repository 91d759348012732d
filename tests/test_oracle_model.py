"""Pins for the oracle worker step (Eq. 4, "otherwise" branch): bf16 rounding
against torch's conversion, the softmax-cross-entropy gradient and full MLP
backpropagation against fp64 finite differences, and the SGD direction."""
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
