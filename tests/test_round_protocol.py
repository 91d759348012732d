"""A CPU model of the synchronisation in step D of the one-launch round
kernel (the weight gradient of the resident W0 block), run under random
interleavings.

Actors: the X^T producer, two MMA-issuing threads and two epilogue
warpgroups.  Tile c (the cluster's running tile index) belongs to chain
e = c % 2: its MMA is issued by chain e's thread into TMEM buffer e and
committed to accD[e] and xfreeD[c % K]; warpgroup e waits accD[e], reads the
buffer and hands it back by a named barrier that chain e's thread waits on
before the tile c + 2.  X^T tile c goes to ring slot c % K (fullD / xfreeD),
K = 4 in the kernel.  The ring depth must be even: with K = 3 a slot
alternates between the chains, and a chain can start its parity wait for a
slot's phase k while the other chain's phase k - 1 has not landed, which the
parity test would take for complete; the model catches that.

The checks: every mbarrier parity wait targets the phase in progress or the
one just completed (a barrier two phases ahead or behind would make the
parity test ambiguous), a buffer is never overwritten before its drain, a
named-barrier wait consumes exactly the drain it is paired with, nothing
deadlocks, and the last drains pair with the final waits.  A variant with
three buffers taken in turn and one accumulator barrier per buffer must
fail the parity check (the checker is not vacuous)."""
import random

import pytest

KNXD_KERNEL = 4


class _Bar:
    def __init__(self):
        self.n = 0          # completed phases


def _wait(bar, k):
    """Parity wait for phase k: only meaningful while k <= n <= k + 1."""
    assert k <= bar.n <= k + 1, ("parity wait out of range", bar.n, k)
    return bar.n == k + 1


def _run(nD, tau, seed, nbuf=2, acc_index=lambda c, nbuf: c % nbuf, KNXD=KNXD_KERNEL):
    rnd = random.Random(seed)
    fullD = [_Bar() for _ in range(KNXD)]
    xfree = [_Bar() for _ in range(KNXD)]
    acc = [_Bar() for _ in range(8)]
    pend = [[] for _ in range(nbuf)]          # drains not yet consumed, per buffer
    owner = [None] * nbuf
    for s in range(tau):
        tiles = [s * nD + tt for tt in range(nD)]
        prod = list(tiles)
        mma = {e: [c for c in tiles if c % 2 == e] for e in (0, 1)}
        epi = {e: [c for c in tiles if c % 2 == e] for e in (0, 1)}
        inflight, steps = [], 0
        while prod or mma[0] or mma[1] or epi[0] or epi[1] or inflight:
            steps += 1
            assert steps < 20000, "deadlock"
            acts = (["p"] if prod else []) + [("m", e) for e in (0, 1) if mma[e]] + \
                   [("e", e) for e in (0, 1) if epi[e]] + (["a"] if inflight else [])
            act = rnd.choice(acts)
            if act == "p":                                   # producer: tiles in order
                c = prod[0]
                if c >= KNXD and not _wait(xfree[c % KNXD], c // KNXD - 1):
                    continue
                prod.pop(0)
                inflight.append(("load", c))
            elif act == "a":                                 # an async completion lands
                kind, c = inflight.pop(rnd.randrange(len(inflight)))
                if kind == "load":
                    fullD[c % KNXD].n += 1
                else:
                    b = c % nbuf
                    assert owner[b] in (None, "drained"), ("buffer overwritten before its drain", c)
                    owner[b] = c
                    acc[acc_index(c, nbuf)].n += 1
                    xfree[c % KNXD].n += 1
            elif act[0] == "m":                              # chain e issues its next tile
                e = act[1]
                c = mma[e][0]
                b = c % nbuf
                if not _wait(fullD[c % KNXD], c // KNXD):
                    continue
                if c >= nbuf:                                # the buffer's previous use was drained
                    if not pend[b]:
                        continue
                    assert pend[b][0] == c - nbuf, ("wrong drain consumed", pend[b][0], c)
                    pend[b].pop(0)
                mma[e].pop(0)
                inflight.append(("mma", c))
            else:                                            # warpgroup e drains its next tile
                e = act[1]
                c = epi[e][0]
                b = c % nbuf
                if not _wait(acc[acc_index(c, nbuf)], c // nbuf):
                    continue
                assert owner[b] == c, ("epilogue reads another tile", owner[b], c)
                owner[b] = "drained"
                epi[e].pop(0)
                pend[b].append(c)
                assert len(pend[b]) <= 1, "two drains pending on one barrier"
    for b in range(nbuf):                                    # the final waits
        used = any(c % nbuf == b for c in range(tau * nD))
        assert len(pend[b]) == (1 if used else 0)


@pytest.mark.parametrize("knxd", [KNXD_KERNEL, 2, 6])
@pytest.mark.parametrize("nD", [1, 2, 3, 5, 8, 9, 12, 13])
@pytest.mark.parametrize("tau", [1, 2, 7])
def test_two_chain_step_d_protocol(nD, tau, knxd):
    for seed in range(40):
        _run(nD, tau, seed, KNXD=knxd)


def test_three_buffers_in_turn_with_one_barrier_per_buffer_is_caught():
    failures = 0
    for seed in range(40):
        try:
            _run(13, 7, seed, nbuf=3)
        except AssertionError:
            failures += 1
    assert failures > 0


def test_odd_ring_depth_is_caught():
    """Three X^T slots shared by two chains: some interleaving makes a parity
    wait two phases ahead of its barrier."""
    failures = 0
    for seed in range(40):
        try:
            _run(5, 2, seed, KNXD=3)
        except AssertionError:
            failures += 1
    assert failures > 0
