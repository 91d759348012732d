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


def test_policy_counts_and_barriers():
    t = np.array([1000, 1000, 500, 250])
    tau, B = schedule.policy_local_steps("bsp", t)
    assert tau.tolist() == [1, 1, 1, 1] and B == 1000
    tau, B = schedule.policy_local_steps("local_sgd", t, period=3)
    assert tau.tolist() == [3, 3, 3, 3] and B == 3000
    tau, B = schedule.policy_local_steps("oscars", t, M=8)
    assert tau.tolist() == [1, 1, 2, 4] and B == 1000


def test_alg1_barrier_is_last_push_brute_force():
    """T* of Algorithm 1 equals max_i tau_i t_i: some worker never waits."""
    rng = np.random.default_rng(5)
    for _ in range(300):
        t = rng.integers(1, 40, size=rng.integers(1, 6))
        M = int(rng.integers(1, 6))
        T, mw, tau = schedule.schedule(t, M)
        assert schedule.round_barrier(t, tau) == T
        assert (T % t).min() == 0


def test_override_clock_is_last_push():
    dims = [6, 10]
    layers, shards = make(dims, 3, 64)
    t = [700, 300, 200]
    for tau in ([1, 1, 1], [2, 2, 2], [1, 3, 4]):
        state, recs = run.run(dims, layers, shards, t_iter=t, M=8, rounds=2, batch=4, lr=0.05,
                              bf16=False, tau_override=tau)
        B = max(a * b for a, b in zip(tau, t))
        assert all(r.T_star == B for r in recs)
        assert state.clock.tolist() == [2 * B] * 3
        idle = [B - a * b for a, b in zip(tau, t)]
        assert state.idle.tolist() == [2 * i for i in idle] and min(idle) == 0


def test_local_sgd_period_one_is_bsp():
    dims = [8, 12, 10]
    layers, shards = make(dims, 3, 32, seed=7)
    t = [900, 400, 250]
    a, ra = run.run(dims, layers, shards, t_iter=t, M=8, rounds=3, batch=4, lr=0.1, bf16=True,
                    tau_override=schedule.policy_local_steps("local_sgd", t, period=1)[0])
    b, rb = run.run(dims, layers, shards, t_iter=t, M=8, rounds=3, batch=4, lr=0.1, bf16=True,
                    tau_override=schedule.policy_local_steps("bsp", t)[0])
    np.testing.assert_array_equal(run.flatten(a.x_g), run.flatten(b.x_g))
    assert [r.T_star for r in ra] == [900] * 3


def test_oscars_uses_idle_time_of_bsp():
    """Under Algorithm 1 the workers of the 4-worker example are never idle;
    under BSP the fast ones idle, so per simulated tick Oscars runs twice as
    many mini-batches (8 vs 4 per 1000 ticks)."""
    t = np.array([1000, 1000, 500, 250])
    tau_o, B_o = schedule.policy_local_steps("oscars", t, M=8)
    tau_b, B_b = schedule.policy_local_steps("bsp", t)
    assert (B_o - tau_o * t).sum() == 0
    assert (B_b - tau_b * t).tolist() == [0, 0, 500, 750]
    assert tau_o.sum() / B_o == 2 * tau_b.sum() / B_b


def test_time_to_loss_and_early_stop():
    recs = [run.RoundRecord(np.ones(2, np.int32), 100, np.zeros(2), np.zeros(2), eval_loss=v)
            for v in (2.0, 1.5, 1.2, 0.9)]
    assert run.time_to_loss(recs, 1.5) == 200
    assert run.time_to_loss(recs, 0.95) == 400
    assert run.time_to_loss(recs, 0.5) is None
    dims = [6, 10]
    layers, shards = make(dims, 2, 64, seed=9)
    ev = (shards[0][0][:32], shards[0][1][:32])
    _, full = run.run(dims, layers, shards, t_iter=[300, 100], M=8, rounds=6, batch=8, lr=0.2,
                      bf16=False, eval_set=ev)
    target = full[2].eval_loss
    _, part = run.run(dims, layers, shards, t_iter=[300, 100], M=8, rounds=6, batch=8, lr=0.2,
                      bf16=False, eval_set=ev, target_loss=target)
    k = next(i for i, r in enumerate(full) if r.eval_loss <= target)
    assert len(part) == k + 1
    assert run.time_to_loss(part, target) == (k + 1) * 300


def test_reschedule_follows_each_rounds_times():
    """Drifting speeds: every round runs Algorithm 1's counts for the times
    in force, and the clocks add up the rounds' barriers."""
    dims = [6, 10]
    layers, shards = make(dims, 3, 64, seed=11)
    ts = [[700, 300, 200], [700, 300, 200], [300, 600, 250], [410, 410, 990]]
    state, recs = run.run(dims, layers, shards, M=6, rounds=4, batch=4, lr=0.05, bf16=False, t_per_round=ts)
    total = 0
    for r, rec in enumerate(recs):
        T, mw, tau = schedule.schedule(ts[r], 6)
        assert rec.T_star == T and rec.tau.tolist() == tau.tolist()
        assert rec.idle.tolist() == (T - tau * np.asarray(ts[r])).tolist()
        total += T
    assert state.clock.tolist() == [total] * 3
    # constant times: the same run as without rescheduling
    a, _ = run.run(dims, layers, shards, M=6, rounds=3, batch=4, lr=0.05, bf16=False, t_per_round=[ts[0]] * 3)
    b, _ = run.run(dims, layers, shards, t_iter=ts[0], M=6, rounds=3, batch=4, lr=0.05, bf16=False)
    np.testing.assert_array_equal(run.flatten(a.x_g), run.flatten(b.x_g))
    assert a.clock.tolist() == b.clock.tolist()
