"""Pins for the data-partition oracle: a hand-worked case, the sum and quota
properties, brute-force optimality of the largest-remainder rule on tiny
inputs (it minimises the total deviation from the exact shares), refusals, and the
point of the rule: with shards sized by tau every worker's cursor wraps in
the same round.  The C ABI's helper is then compared with it bit for bit."""
import itertools
from fractions import Fraction

import numpy as np
import pytest

from oracle import partition, run, schedule


def test_hand_worked():
    # 16384 samples, batch 32: Q = 512 units by tau = 1,1,2,4 -> exact shares
    # 64, 64, 128, 256
    assert partition.partition_sizes([1, 1, 2, 4], 16384, 32) == [64 * 32, 64 * 32, 128 * 32, 256 * 32]
    # 16400 samples: still 512 whole units, the 16 leftover samples unused
    assert partition.partition_sizes([1, 1, 2, 4], 16400, 32) == [64 * 32, 64 * 32, 128 * 32, 256 * 32]
    # Q = 10 by 3,3,3: shares 3.33 each, the spare unit to the first
    assert partition.partition_sizes([3, 3, 3], 10, 1) == [4, 3, 3]
    # Q = 14 by 1,5: shares 2.33, 11.67 -> 2 + 12
    assert partition.partition_sizes([1, 5], 100, 7) == [2 * 7, 12 * 7]
    # Q = 7 by 1,2,4 -> exact 1, 2, 4
    assert partition.partition_sizes([1, 2, 4], 7, 1) == [1, 2, 4]


def test_sum_and_quota():
    rng = np.random.default_rng(4)
    for _ in range(500):
        n = int(rng.integers(1, 12))
        w = [int(v) for v in rng.integers(1, 20, n)]
        unit = int(rng.integers(1, 70))
        total = int(rng.integers(20 * n * unit, 50 * 20 * n * unit + 1))
        s = partition.partition_sizes(w, total, unit)
        Q = total // unit
        assert sum(s) == Q * unit and all(v % unit == 0 and v >= unit for v in s)
        for v, wi in zip(s, w):
            exact = Fraction(Q * wi, sum(w))
            assert abs(v // unit - exact) < 1


def test_minimises_total_deviation_brute_force():
    rng = np.random.default_rng(8)
    for _ in range(150):
        n = int(rng.integers(1, 5))
        w = [int(v) for v in rng.integers(1, 9, n)]
        Q = int(rng.integers(1, 10))
        exact = [Fraction(Q * wi, sum(w)) for wi in w]
        best = min(sum(abs(a - e) for a, e in zip(alloc, exact))
                   for alloc in itertools.product(range(Q + 1), repeat=n) if sum(alloc) == Q)
        try:
            got = partition.partition_sizes(w, Q, 1)
        except ValueError:          # only possible when some exact share is below one unit
            assert min(exact) < 1
            continue
        assert sum(abs(a - e) for a, e in zip(got, exact)) == best


def test_errors():
    for args in (([], 10, 1), ([1, 0], 10, 1), ([1, 1], 1, 1), ([1], 10, 0), ([1, 100], 50, 1)):
        with pytest.raises(ValueError):
            partition.partition_sizes(*args)


def test_shards_sized_by_tau_wrap_together():
    t = [1000, 1000, 500, 250]
    _, _, tau = schedule.schedule(t, 8)
    B, epochs = 4, 3
    sizes = partition.partition_sizes(tau.tolist(), epochs * int(tau.sum()) * B, B)
    assert sizes == [epochs * int(v) * B for v in tau]
    dims = [5, 10]
    rng = np.random.default_rng(0)
    shards = [(rng.standard_normal((n, 5)).astype(np.float32), rng.integers(0, 10, n).astype(np.int32))
              for n in sizes]
    layers = [(np.zeros((10, 5), np.float32), np.zeros(10, np.float32))]
    state, _ = run.run(dims, layers, shards, t_iter=t, M=8, rounds=epochs, batch=B, lr=0.05, bf16=False)
    assert state.cursor.tolist() == [0] * 4


def test_capi_matches_oracle(oscars_lib):
    import paper_2102_08550_gb300 as P
    rng = np.random.default_rng(21)
    for _ in range(300):
        n = int(rng.integers(1, 40))
        w = [int(v) for v in rng.integers(1, 1 << 20, n)]
        unit = int(rng.integers(1, 256))
        total = int(rng.integers(1 << 32, 1 << 40))
        assert P.oscars_partition_sizes(w, total, unit) == partition.partition_sizes(w, total, unit)
    for args in (([1, 0], 10, 1), ([1, 1], 1, 1), ([1], 10, 0), ([1, 100], 50, 1)):
        with pytest.raises(P.OscarsError):
            P.oscars_partition_sizes(*args)
