"""CPU oracle for the Oscars hot path (semi-synchronous, load-balanced local SGD).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import, call or
link this package: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.

It is a plain, slow, obviously-correct restatement of what the paper's method
computes, in fp64 unless noted, and it shares no code with the CUDA library:

* ``schedule``  - iteration ticks, the wait time of Eq. 1, the max-wait
  objective of Eq. 2, Algorithm 1 (the load-balance search for the barrier
  T* of Eq. 3) and the local-step counts tau_i = floor(T*/t_i).
* ``model``     - one worker's mini-batch SGD step, Eq. 4 "otherwise" branch,
  for a ReLU MLP / softmax regression with softmax cross-entropy.
* ``merge``     - the server's merge and global update, Eq. 4 first branch,
  in the delta form x_g + eta_s * sum_k w_k (x^k - x_g).
* ``run``       - the round loop: local steps, push, merge, pull.

Each function cites the passage it follows.  Pins (tests that check the oracle
against something other than itself) live in ``tests/test_oracle_*.py``.
"""
