"""Pins for the oracle round loop: W=1 reduces to sequential SGD, the BSP
special case (tau = 1, uniform weights) equals one SGD step on the
concatenated batch, the barrier makes every simulated clock equal R*T*, and
the data cursor wraps."""
import numpy as np

from oracle import bf16, model, run, schedule


def make(dims, W, n, seed=0):
    rng = np.random.default_rng(seed)
    layers = [((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32),
               (rng.standard_normal(o) * 0.01).astype(np.float32))
              for i, o in zip(dims[:-1], dims[1:])]
    shards = [(rng.standard_normal((n, dims[0])).astype(np.float32), rng.integers(0, 10, n).astype(np.int32))
              for _ in range(W)]
    return layers, shards


def test_single_worker_is_sequential_sgd():
    dims = [12, 16, 10]
    layers, shards = make(dims, 1, 40)
    for tau in (1, 3):
        state, recs = run.run(dims, layers, shards, t_iter=[7], M=4, rounds=4, batch=8, lr=0.1,
                              bf16=True, tau_override=[tau])
        seq = layers
        X, y = shards[0]
        cur = 0
        for _ in range(4 * tau):
            idx = (cur + np.arange(8)) % 40
            cur = (cur + 8) % 40
            seq, _ = model.sgd_step(seq, X[idx], y[idx], 0.1, bf16.round_bf16)
        np.testing.assert_array_equal(run.flatten(state.x_g), run.flatten(seq))


def test_bsp_equals_large_batch_sgd():
    dims = [10, 14, 10]
    W, B = 4, 8
    layers, shards = make(dims, W, B, seed=3)
    state, _ = run.run(dims, layers, shards, t_iter=[5] * W, M=4, rounds=1, batch=B, lr=0.2,
                       bf16=False)
    assert state.tau.tolist() == [1] * W
    Xc = np.concatenate([s[0] for s in shards])
    yc = np.concatenate([s[1] for s in shards])
    big, _ = model.sgd_step(layers, Xc, yc, 0.2, bf16.identity)
    a, b = run.flatten(state.x_g), run.flatten(big)
    assert np.abs(a - b).max() <= 1e-6 * np.abs(b).max()


def test_barrier_clocks_and_idle():
    dims = [6, 10]
    layers, shards = make(dims, 4, 64)
    t = [1000, 1000, 500, 250]
    state, recs = run.run(dims, layers, shards, t_iter=t, M=8, rounds=3, batch=4, lr=0.05, bf16=False)
    T, _, tau = schedule.schedule(t, 8)
    assert np.all(state.clock == 3 * T)
    assert np.all(state.idle == 3 * (T % np.asarray(t)))
    for r in recs:
        assert r.tau.tolist() == tau.tolist() and r.T_star == T


def test_cursor_wraps():
    dims = [4, 10]
    layers, shards = make(dims, 1, 12)
    state, _ = run.run(dims, layers, shards, t_iter=[3], M=2, rounds=2, batch=5, lr=0.05, bf16=False,
                       tau_override=[2])
    assert state.cursor.tolist() == [(4 * 5) % 12]
    assert run.batch_indices(10, 5, 12).tolist() == [10, 11, 0, 1, 2]


def test_flatten_roundtrip():
    dims = [5, 4, 3]
    layers, _ = make(dims, 1, 2)
    flat = run.flatten(layers)
    assert flat.size == 5 * 4 + 4 + 4 * 3 + 3
    back = run.unflatten(flat, dims)
    for (a, b), (c, d) in zip(layers, back):
        np.testing.assert_array_equal(a, c)
        np.testing.assert_array_equal(b, d)
