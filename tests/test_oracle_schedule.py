"""Pins for the oracle scheduler (Eq. 1-3, Algorithm 1): hand-derived worked
examples, an independent brute force, the least-common-multiple property the
paper names, and monotonicity invariants."""
import math
import os

import numpy as np
import pytest

from oracle import schedule as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "alg1_cases.txt")


def golden_cases():
    out = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        t, M, T, mw, tau, note = [f.strip() for f in line.split("|")]
        out.append(([int(v) for v in t.split(",")], int(M), int(T), int(mw),
                    [int(v) for v in tau.split(",")], note))
    return out


@pytest.mark.parametrize("case", golden_cases(), ids=lambda c: ",".join(map(str, c[0])))
def test_alg1_golden(case):
    t, M, T_exp, mw_exp, tau_exp, _ = case
    T, mw, tau = S.schedule(t, M)
    assert (T, mw) == (T_exp, mw_exp)
    assert tau.tolist() == tau_exp


def brute_force(t, M, capped=True):
    """Independent formulation: enumerate every integer T in the searched
    range, keep the candidates reachable from max(t) without violating the
    constraint, and take the lexicographic minimum of (max wait, T)."""
    tmin, tmax = min(t), max(t)
    hi = M * tmax if capped else tmax + 10 * M * tmax * tmax
    cands = [tmax]
    T = tmax + 1
    while T <= hi and (T // tmin - T // tmax) < M:
        cands.append(T)
        T += 1
    best = min(cands, key=lambda T: (max(T - (T // x) * x for x in t), T))
    return best, max(best - (best // x) * x for x in t)


def test_alg1_brute_force_random():
    rng = np.random.default_rng(123)
    for _ in range(400):
        n = int(rng.integers(1, 6))
        t = [int(v) for v in rng.integers(1, 13, n)]
        M = int(rng.integers(1, 7))
        T, mw, _ = S.load_balance_search(t, M)
        assert (T, mw) == brute_force(t, M), (t, M)


def test_alg1_literal_matches_uncapped_brute_force():
    rng = np.random.default_rng(7)
    for _ in range(200):
        t = [int(v) for v in rng.integers(1, 11, 3)]
        if min(t) == max(t):
            continue
        M = int(rng.integers(1, 6))
        T, mw, _ = S.load_balance_search(t, M, S.LITERAL)
        assert (T, mw) == brute_force(t, M, capped=False), (t, M)


def test_alg1_literal_rejects_homogeneous():
    with pytest.raises(ValueError):
        S.load_balance_search([5, 5], 4, S.LITERAL)


def test_lcm_principle():
    """If lcm(t) lies inside the searched range, T* = lcm(t) with zero wait."""
    rng = np.random.default_rng(5)
    hits = 0
    for _ in range(300):
        t = [int(v) for v in rng.integers(1, 9, int(rng.integers(1, 5)))]
        M = int(rng.integers(1, 9))
        L = math.lcm(*t)
        _, _, trace = S.load_balance_search(t, M)
        if L <= trace[-1][0]:
            hits += 1
            T, mw, _ = S.load_balance_search(t, M)
            assert (T, mw) == (L, 0)
    assert hits > 50


def test_schedule_invariants():
    rng = np.random.default_rng(11)
    for _ in range(200):
        t = np.asarray(rng.integers(1, 400, int(rng.integers(1, 9))), dtype=np.int64)
        M = int(rng.integers(1, 17))
        T, mw, tau = S.schedule(t, M)
        assert T >= t.max()
        assert np.all(tau >= 1)
        order = np.argsort(t, kind="stable")
        assert np.all(np.diff(tau[order]) <= 0)            # faster -> more steps
        assert mw <= S.max_wait(t, int(t.max()))          # never worse than T = max(t)
        assert np.array_equal(S.wait_times(t, T), T - tau.astype(np.int64) * t)


def test_iteration_ticks():
    assert S.iteration_ticks([1, 1, 2, 4]).tolist() == [1000, 1000, 500, 250]
    assert S.iteration_ticks([3.0]).tolist() == [333]        # 333.33 -> 333
    assert S.iteration_ticks([1.6]).tolist() == [625]
    assert S.iteration_ticks([2.5], 1).tolist() == [1]       # floor(0.4 + 0.5) = 0 -> max(1, .)
    assert S.iteration_ticks([0.8], 1).tolist() == [1]       # 1.25 + 0.5 -> 1
    assert S.iteration_ticks([0.4], 1).tolist() == [3]       # 2.5 + 0.5 -> 3 (half rounds up)
    with pytest.raises(ValueError):
        S.iteration_ticks([1.0, 0.0])


def test_merge_weights():
    w = S.merge_weights("uniform", [3, 1, 2])
    assert w.dtype == np.float32 and np.all(w == np.float32(1 / 3))
    w = S.merge_weights("localsteps", [3, 1, 4])
    assert w.tolist() == [np.float32(3 / 8), np.float32(1 / 8), np.float32(4 / 8)]
