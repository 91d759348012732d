"""Host logic of the one-launch round kernel: the worker lists when fewer
clusters fit on the device than there are workers (oscars_round_clusters,
longest processing time first).  CPU only: the library loads without a GPU."""
import itertools

import pytest

import paper_2102_08550_gb300 as P

# tau of the 784-512-10 workload with 16 workers (the schedule of its seeded speeds)
HEADLINE_TAU = [5, 6, 5, 2, 6, 5, 3, 5, 5, 5, 4, 5, 3, 4, 3, 5]


def loads(lists, tau):
    return [sum(tau[w] + 0.5 for w in l) for l in lists]


def test_one_cluster_per_worker_when_all_fit():
    tau = [3, 1, 4, 1, 5]
    for cap in (0, -1, 5, 8):
        lists = P.oscars_round_clusters(tau, cap)
        assert lists == [[4], [2], [0], [1], [3]]   # decreasing tau, ties by index


def test_headline_with_15_clusters():
    lists = P.oscars_round_clusters(HEADLINE_TAU, 15)
    assert len(lists) == 15
    assert sorted(w for l in lists for w in l) == list(range(16))
    shared = [l for l in lists if len(l) == 2]
    assert len(shared) == 1
    # the shortest worker (tau 2) follows the last tau-3 worker; that cluster
    # (3 + 2 steps) still ends before the tau-6 ones
    assert [HEADLINE_TAU[w] for w in shared[0]] == [3, 2]
    assert max(loads(lists, HEADLINE_TAU)) == 6.5


def greedy_reference(tau, cap):
    """The rule written out plainly: workers by decreasing tau (stable), each
    to the first cluster of least load, load += tau + 1/2."""
    order = sorted(range(len(tau)), key=lambda i: -tau[i])
    n = min(cap, len(tau)) if cap > 0 else len(tau)
    lists, load = [[] for _ in range(n)], [0.0] * n
    for w in order:
        k = min(range(n), key=lambda j: (load[j], j))
        lists[k].append(w)
        load[k] += tau[w] + 0.5
    return lists


@pytest.mark.parametrize("cap", [1, 2, 3, 7])
def test_matches_the_rule_and_is_near_optimal(cap):
    for tau in itertools.product([1, 2, 4, 7], repeat=5):
        tau = list(tau)
        lists = P.oscars_round_clusters(tau, cap)
        assert lists == greedy_reference(tau, cap)
        assert sorted(w for l in lists for w in l) == list(range(5))
        # LPT is within 4/3 of the best makespan (Graham); check against brute force
        n = min(cap, 5)
        best = min(max(sum(tau[w] + 0.5 for w in range(5) if a[w] == k) for k in range(n))
                   for a in itertools.product(range(n), repeat=5))
        assert max(loads(lists, tau)) <= 4 / 3 * best + 1e-9


def test_errors():
    with pytest.raises(P.OscarsError):
        P.oscars_round_clusters([], 4)
    with pytest.raises(P.OscarsError):
        P.oscars_round_clusters([3, 0, 2], 2)
