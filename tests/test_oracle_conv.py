"""Pins for the convolutional worker oracle (oracle/conv.py): the 3x3
convolution against a brute-force loop, a delta kernel, the adjoint
identities that tie the transposed convolution and the weight gradient to
the forward, finite differences of the whole network's loss, the residual
block with zero weights, the parameter layout, and the round loop (one
worker = sequential SGD; BSP = one step on the concatenated batch)."""
import numpy as np
import pytest

from oracle import bf16, conv, run

ident = bf16.identity


def brute_conv(h, W):
    B, H, Wd, I = h.shape
    O = W.shape[0]
    out = np.zeros((B, H, Wd, O))
    for b in range(B):
        for y in range(H):
            for x in range(Wd):
                for o in range(O):
                    acc = 0.0
                    for dy in range(3):
                        for dx in range(3):
                            yy, xx = y + dy - 1, x + dx - 1
                            if 0 <= yy < H and 0 <= xx < Wd:
                                for i in range(I):
                                    acc += float(W[o, dy, dx, i]) * float(h[b, yy, xx, i])
                    out[b, y, x, o] = acc
    return out


def test_conv_matches_brute_force():
    rng = np.random.default_rng(0)
    h = rng.standard_normal((2, 4, 5, 3)).astype(np.float32)
    W = rng.standard_normal((4, 3, 3, 3)).astype(np.float32)
    np.testing.assert_allclose(conv.conv3x3(h, W, ident), brute_conv(h, W), rtol=1e-5, atol=1e-5)


def test_delta_kernel_is_identity():
    rng = np.random.default_rng(1)
    h = rng.standard_normal((1, 5, 5, 3)).astype(np.float32)
    W = np.zeros((3, 3, 3, 3), np.float32)
    W[:, 1, 1, :] = np.eye(3)
    np.testing.assert_array_equal(conv.conv3x3(h, W, ident), h)
    W2 = np.zeros_like(W)
    W2[:, 0, 0, :] = np.eye(3)            # tap (dy, dx) = (0, 0) reads (y - 1, x - 1)
    out = conv.conv3x3(h, W2, ident)
    np.testing.assert_array_equal(out[:, 1:, 1:, :], h[:, :-1, :-1, :])
    assert np.all(out[:, 0, :, :] == 0) and np.all(out[:, :, 0, :] == 0)


def test_adjoint_identities():
    """<conv(h, W), dz> = <h, conv^T(dz, W)> = <W, dW(dz, h)> exactly in the
    real numbers; here within fp64-summed, fp32-rounded accuracy."""
    rng = np.random.default_rng(2)
    h = rng.standard_normal((2, 6, 5, 4)).astype(np.float32)
    W = rng.standard_normal((3, 3, 3, 4)).astype(np.float32)
    dz = rng.standard_normal((2, 6, 5, 3)).astype(np.float32)
    a = float((conv.conv3x3(h, W, ident).astype(np.float64) * dz).sum())
    b = float((h.astype(np.float64) * conv.conv3x3_transposed(dz, W, ident)).sum())
    c = float((W.astype(np.float64) * conv.conv3x3_weight_grad(dz, h, ident)).sum())
    assert abs(a - b) <= 1e-5 * abs(a) and abs(a - c) <= 1e-5 * abs(a)


def tiny_model(seed=3, blocks=1):
    m = conv.CNN(height=4, width=4, in_ch=3, ch=4, blocks=blocks, classes=3)
    rng = np.random.default_rng(seed)
    params = []
    for shp in m.shapes():
        if len(shp) == 1:
            params.append(np.full(shp, 0.5, np.float32))        # biases keep every ReLU open
        else:
            params.append((rng.standard_normal(shp) * 0.3).astype(np.float32))
    X = (np.abs(rng.standard_normal((2, 4 * 4 * 3))) + 0.5).astype(np.float32)
    y = np.array([0, 2], np.int32)
    return m, params, X, y


def test_gradients_match_finite_differences():
    m, params, X, y = tiny_model()
    _, grads = m.gradients(params, X, y, ident)
    rng = np.random.default_rng(4)
    for t, (p, g) in enumerate(zip(params, grads)):
        for _ in range(3):
            idx = tuple(int(rng.integers(0, n)) for n in p.shape)
            eps = 1e-2
            plus = [q.copy() for q in params]
            minus = [q.copy() for q in params]
            plus[t][idx] += eps
            minus[t][idx] -= eps
            lp = m.loss_of(plus, X, y, ident)
            lm = m.loss_of(minus, X, y, ident)
            fd = (lp - lm) / (2 * eps)
            assert abs(fd - float(g[idx])) <= 2e-3 + 2e-2 * abs(fd), (t, idx, fd, float(g[idx]))


def test_zero_block_is_identity():
    m, params, X, y = tiny_model(seed=5)
    for t in (2, 3, 4, 5):
        params[t] = np.zeros_like(params[t])
    acts, logits = m.forward(params, X, bf16.round_bf16)
    np.testing.assert_array_equal(acts["v"][0], acts["s"][0])
    m0 = conv.CNN(height=4, width=4, in_ch=3, ch=4, blocks=0, classes=3)
    _, logits0 = m0.forward(params[:2] + params[-2:], X, bf16.round_bf16)
    np.testing.assert_array_equal(logits, logits0)


def test_layout():
    m = conv.CNN()
    assert m.num_params() == 64 * 9 * 3 + 64 + 2 * (64 * 9 * 64 + 64) + 10 * 64 + 10
    rng = np.random.default_rng(6)
    flat = rng.standard_normal(m.num_params()).astype(np.float32)
    np.testing.assert_array_equal(m.flatten(m.unflatten(flat)), flat)


def test_round_loop_single_worker_and_bsp():
    m, params, X, y = tiny_model(seed=7)
    n = 4
    rng = np.random.default_rng(8)
    Xs = [(np.abs(rng.standard_normal((n, 48))) + 0.5).astype(np.float32) for _ in range(2)]
    ys = [rng.integers(0, 3, n).astype(np.int32) for _ in range(2)]
    # one worker, tau = 3: three sequential SGD steps
    state, _ = run.run([48, 3], params, [(Xs[0], ys[0])], t_iter=[5], M=4, rounds=1, batch=2, lr=0.1,
                       bf16=True, tau_override=[3], model=m)
    seq = params
    for s in range(3):
        idx = (2 * s + np.arange(2)) % n
        seq, _ = m.sgd_step(seq, Xs[0][idx], ys[0][idx], 0.1, bf16.round_bf16)
    np.testing.assert_array_equal(m.flatten(state.x_g), m.flatten(seq))
    # BSP over two workers = one step on the concatenated batch (fp32 model)
    state, _ = run.run([48, 3], params, [(Xs[0], ys[0]), (Xs[1], ys[1])], t_iter=[5, 5], M=4, rounds=1,
                       batch=n, lr=0.1, bf16=False, model=m)
    big, _ = m.sgd_step(params, np.concatenate(Xs), np.concatenate(ys), 0.1, ident)
    a, b = m.flatten(state.x_g), m.flatten(big)
    assert np.abs(a - b).max() <= 1e-6 * np.abs(b).max()
