"""Data-partition load balancing, CPU oracle (test infrastructure only).

The paper names a subsection "Data partition load balancing" and leaves it
empty.  Reading: shard sizes follow the workers' per-round consumption
tau_i * B, so every worker sweeps its own shard in the same number of rounds
and every sample is visited equally often.  The data set is handed out in
whole units (normally one mini-batch): the Q units go in proportion to the
weights by largest remainder (Hamilton's apportionment), ties to the lower
index; a request that would leave a worker without data is refused.  Exact
rational arithmetic.
"""
from __future__ import annotations

from fractions import Fraction
from typing import List, Sequence


def partition_sizes(weight: Sequence[int], total: int, unit: int = 1) -> List[int]:
    w = [int(v) for v in weight]
    n = len(w)
    if n < 1 or unit < 1 or total < 0 or any(v < 1 for v in w):
        raise ValueError("bad partition request")
    Q = total // unit
    quota = [Fraction(Q * v, sum(w)) for v in w]          # exact shares
    units = [int(q) for q in quota]                       # floor
    left = Q - sum(units)
    by_remainder = sorted(range(n), key=lambda i: (-(quota[i] - units[i]), i))
    for i in by_remainder[:left]:
        units[i] += 1
    if min(units) < 1:
        raise ValueError("a worker would get no data")
    return [u * unit for u in units]
