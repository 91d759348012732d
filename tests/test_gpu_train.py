"""Local steps + merge + pull (Eq. 4, both branches) on the GPU against the
oracle: schedules bit-exact, merged parameters within 1e-5 (max-abs,
normalised per tensor), losses within 1e-3 relative.

Cases: the fp32 softmax-regression workload at full size (all rounds), small
bf16 MLPs that span several tiles, ragged K tails and a middle layer (the
input-gradient GEMM), the 784-512-10 workload at full size for all 100
rounds, and every worker of the 3072-1024-1024-10 workload at full size for
two rounds."""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2102_08550_gb300 as P
import synth
from oracle import bf16 as obf16
from oracle import model as omodel
from oracle import run as orun
from tests.gpu_util import (LOSS_RTOL, PARAM_RTOL, assert_within, device_shards, envelope, make_context,
                            oracle_inputs, oracle_schedule, per_tensor_errors, pull_flat, replica_flat)

pytestmark = pytest.mark.gpu


def run_both(w, rounds, device, rows=None, flags=0, tau_override=None, eval_n=0, oracle_rows=None,
             exact_inputs=False, strict=None):
    """Run ``rounds`` rounds on the GPU and in the oracle on the same inputs.

    ``oracle_rows``: generate only the first rows of each shard for the
    oracle (enough when the cursor does not wrap within ``rounds``).
    ``exact_inputs``: integer samples and power-of-two weights, so that the
    first layer's products sum exactly in any order.  ``strict``: require
    1e-5 per tensor (default: for fp32 models and exact-input runs);
    otherwise the bound is the measured conditioning envelope."""
    rows = rows or w.samples_per_worker
    if exact_inputs:
        shards_d = [synth.shard_int_t(w, k, rows, device) for k in range(w.num_workers)]
        layers0 = synth.init_layers_int_np(w)
    else:
        shards_d = device_shards(w, device, n=rows)
        layers0 = None
    ctx, layers0 = make_context(w, shards_d, device, flags=flags, layers0=layers0)
    if tau_override is not None:
        ctx.set_local_steps(tau_override)
    gpu_losses, gpu_x = [], []
    for _ in range(rounds):
        tau, loss = ctx.local_steps()
        ctx.push_merge()
        gpu_losses.append(np.array(loss))
        gpu_x.append(pull_flat(ctx, device))
    orows = oracle_rows or rows
    shards_h = ([synth.shard_int_np(w, k, orows) for k in range(w.num_workers)] if exact_inputs
                else oracle_inputs(w, orows))
    t, T, mw, tau_o = oracle_schedule(w)

    def oracle_run():
        return orun.run(w.dims, layers0, shards_h, t_iter=t, M=w.M, rounds=rounds, batch=w.batch, lr=w.lr,
                        bf16=w.bf16, server_lr=w.server_lr, tau_override=tau_override)
    state, recs = oracle_run()
    sch = ctx.schedule()
    if tau_override is None:
        assert sch["tau"] == tau_o.tolist()
        assert sch["T_star"] == T and sch["max_wait"] == mw
    assert sch["t_iter"] == t.tolist()
    assert sch["clock"] == [rounds * sch["T_star"]] * w.num_workers
    for r in range(rounds):
        np.testing.assert_allclose(gpu_losses[r], recs[r].worker_loss, rtol=LOSS_RTOL)
    strict = (not w.bf16 or exact_inputs) if strict is None else strict
    if strict:
        env = [np.zeros(2 * (len(w.dims) - 1))] * rounds
    else:
        env = envelope(lambda: [rc.x_g for rc in oracle_run()[1]], w.dims, [rc.x_g for rc in recs])
    for r in range(rounds):
        assert_within(per_tensor_errors(gpu_x[r], recs[r].x_g, w.dims), env[r], f"round {r}")
    ev = None
    if eval_n:
        Xe, ye = synth.eval_np(w, n=eval_n)
        ge = ctx.eval_loss(torch.from_numpy(Xe).to(device), torch.from_numpy(ye).to(device))
        oe = omodel.loss_of(state.x_g, Xe, ye, obf16.round_bf16 if w.bf16 else obf16.identity)
        assert abs(ge - oe) <= LOSS_RTOL * abs(oe), (ge, oe)
        ev = (ge, oe)
    ctx.close()
    return ev


def test_softmax_regression_full(cuda_device):
    w = synth.CFG1
    run_both(w, w.rounds, cuda_device, eval_n=w.eval_n)


def test_softmax_regression_direct_launch(cuda_device):
    run_both(dataclasses.replace(synth.CFG1, samples_per_worker=200), 3, cuda_device, flags=P.FLAG_NO_GRAPH)


SMALL = [
    # name, dims, W, batch, rows, M
    ("2layer", [784, 512, 10], 4, 64, 512, 8),
    ("3layer", [200, 256, 128, 10], 3, 32, 256, 6),       # ragged K tail, middle layer (input-gradient GEMM)
    ("4layer", [96, 128, 256, 128, 10], 5, 128, 512, 4),
    # two workers, deep K: the forward and input-gradient GEMMs split K over clusters of 4 and 2 CTAs
    ("split-k", [1024, 512, 512, 10], 2, 64, 256, 4),
]


@pytest.mark.parametrize("name,dims,W,B,rows,M", SMALL, ids=[s[0] for s in SMALL])
def test_mlp_small(cuda_device, name, dims, W, B, rows, M):
    w = synth.TrainWorkload(f"small-{name}", W, dims, B, 0.05, rows, M, 3)
    run_both(w, 3, cuda_device, rows=rows, eval_n=4 * B)


EXACT = [
    ("2layer", [784, 512, 10], 4, 64),
    ("3layer", [384, 256, 128, 10], 3, 32),
]


@pytest.mark.parametrize("name,dims,W,B", EXACT, ids=[s[0] for s in EXACT])
def test_mlp_exact_inputs_one_step_strict(cuda_device, name, dims, W, B):
    """One local step per worker on integer inputs: the first layer's forward
    is exact in any summation order, so bf16 rounding and ReLU decisions agree
    and the merged model must match to 1e-5 per tensor."""
    w = synth.TrainWorkload(f"exact-{name}", W, dims, B, 0.05, 4 * B, 4, 1)
    run_both(w, 1, cuda_device, rows=4 * B, tau_override=[1] * W, exact_inputs=True, eval_n=2 * B)


def test_mlp_bsp_override(cuda_device):
    w = synth.TrainWorkload("small-bsp", 4, [128, 128, 10], 32, 0.1, 128, 4, 2)
    run_both(w, 2, cuda_device, tau_override=[1, 1, 1, 1])


def test_mlp_2layer_per_layer_kernels(cuda_device):
    """The per-layer kernel path for a 2-layer model (the default runs each
    round of such a model as one fused launch)."""
    w = synth.TrainWorkload("small-per-layer", 4, [784, 512, 10], 64, 0.05, 512, 8, 2)
    run_both(w, 2, cuda_device, rows=512, flags=P.FLAG_PER_LAYER)


def test_mlp_branches(cuda_device):
    w = synth.TrainWorkload("small-branches", 5, [256, 128, 128, 10], 32, 0.05, 256, 6, 2)
    run_both(w, 2, cuda_device, rows=256, flags=P.FLAG_BRANCHES)


def test_mlp_direct_launch_matches_graph(cuda_device):
    w = synth.TrainWorkload("small-direct", 3, [256, 128, 10], 64, 0.05, 256, 8, 2)
    run_both(w, 2, cuda_device, flags=P.FLAG_NO_GRAPH)


def test_mlp_784_512_10_w16_all_rounds(cuda_device):
    """The 784-512-10 workload (16 workers, batch 64) at full size for all its
    100 rounds (the cursors wrap): tau and T* bit-exact, every round's worker
    losses within 1e-3, the merged model after every round within the
    conditioning envelope, and the eval loss of the final global model on
    2048 held-out samples within 1e-3."""
    w = synth.CFG2
    _, _, _, tau = oracle_schedule(w)
    assert w.rounds * int(tau.max()) * w.batch > w.samples_per_worker      # the longest cursor wraps
    run_both(w, w.rounds, cuda_device, eval_n=2048)


def test_mlp_784_512_10_w16_exact_one_step_strict(cuda_device):
    """The headline shape with all 16 workers, one step each on integer
    inputs: only 15 clusters of the one-launch round fit on the device, so one
    cluster runs two workers back to back (its barriers, TMEM and rings carry
    over).  The merged model must match to 1e-5 per tensor."""
    w = dataclasses.replace(synth.CFG2, samples_per_worker=4 * synth.CFG2.batch)
    names = kernel_classes(w, cuda_device, w.samples_per_worker)
    assert "fused_round" in names, names
    run_both(w, 1, cuda_device, rows=w.samples_per_worker, tau_override=[1] * w.num_workers, exact_inputs=True,
             eval_n=2 * w.batch)


def test_mlp_3072_1024_1024_10_w32_every_worker(cuda_device):
    """The 3072-1024-1024-10 workload (32 workers, batch 128) at full size for
    two rounds: after each round's local steps every one of the 32 pushed
    replicas, and after each merge the global model, against the oracle
    (conditioning envelope per tensor), with the schedule bit-exact and the
    worker losses within 1e-3."""
    w = synth.CFG3
    rounds = 2
    t, T, mw, tau = oracle_schedule(w)
    rows = rounds * int(tau.max()) * w.batch
    shards_d = device_shards(w, cuda_device, n=rows)
    ctx, layers0 = make_context(w, shards_d, cuda_device)
    got_rep, got_x, got_loss = [], [], []
    for _ in range(rounds):
        tau_g, loss_g = ctx.local_steps()
        assert tau_g == tau.tolist()
        got_rep.append([replica_flat(ctx, k, cuda_device) for k in range(w.num_workers)])
        got_loss.append(np.array(loss_g))
        ctx.push_merge()
        got_x.append(pull_flat(ctx, cuda_device))
    sch = ctx.schedule()
    ctx.close()
    del shards_d
    assert sch["T_star"] == T and sch["max_wait"] == mw
    shards_h = oracle_inputs(w, rows)

    def oracle_run():
        _, recs = orun.run(w.dims, layers0, shards_h, t_iter=t, M=w.M, rounds=rounds, batch=w.batch, lr=w.lr,
                           bf16=True, keep_replicas=True)
        return recs

    def flats(recs):
        return [f for rc in recs for f in (*rc.replicas, rc.x_g)]
    recs = oracle_run()
    env = envelope(lambda: flats(oracle_run()), w.dims, flats(recs))
    i = 0
    for r in range(rounds):
        np.testing.assert_allclose(got_loss[r], recs[r].worker_loss, rtol=LOSS_RTOL)
        for k in range(w.num_workers):
            assert_within(per_tensor_errors(got_rep[r][k], recs[r].replicas[k], w.dims), env[i],
                          f"round {r} worker {k} (tau {int(tau[k])})")
            i += 1
        assert_within(per_tensor_errors(got_x[r], recs[r].x_g, w.dims), env[i], f"round {r} merged")
        i += 1


SOFTREG_SHAPES = [
    # name, D, C, B, rows: the cluster kernel's column split (8 CTAs per worker)
    ("d18-c10", 18, 10, 20, 100),      # some CTAs own no column, one owns 2
    ("d785-c10", 785, 10, 32, 128),    # D % 4 != 0: one float at a time
    ("d64-c32-b256", 64, 32, 256, 600),  # the largest batch and class count of the cluster kernel
]


@pytest.mark.parametrize("name,D,C,B,rows", SOFTREG_SHAPES, ids=[s[0] for s in SOFTREG_SHAPES])
def test_softmax_regression_shapes(cuda_device, name, D, C, B, rows):
    """fp32 softmax regression with each worker on a cluster that splits the
    input columns: ragged and empty column slices, scalar row loads, shards
    that wrap; three rounds, strict 1e-5 against the oracle."""
    w = synth.TrainWorkload(f"softreg-{name}", 3, [D, C], B, 0.05, rows, 4, 3, bf16=False,
                            speeds=[1.0, 2.0, 1.5])
    run_both(w, 3, cuda_device, rows=rows)


def test_softmax_regression_batch_512(cuda_device):
    """The largest batch of the fp32 round kernel (one thread per row): three
    rounds, shards that wrap, strict 1e-5 against the oracle."""
    w = synth.TrainWorkload("softreg-b512", 3, [64, 10], 512, 0.05, 1300, 4, 3, bf16=False)
    run_both(w, 3, cuda_device, rows=1300)


def test_bounded_wait_runs_out_and_context_stays_usable(cuda_device):
    """A kernel wait that runs out (an mbarrier that nothing completes, 1000
    polls) records its code in the context's error word: the host reports
    ETIMEOUT and clears the word, and the next rounds run and match those of
    a fresh context bit for bit (no fault, no hang, the GPU stays usable)."""
    w = synth.TrainWorkload("wait-check", 2, [128, 128, 10], 32, 0.05, 64, 4, 1)
    shards = device_shards(w, cuda_device, n=64)
    a, _ = make_context(w, shards, cuda_device)
    with pytest.raises(P.OscarsError) as e:
        P.oscars_check_wait_timeout(a.handle, 1000)
    assert e.value.status == P.OSCARS_ETIMEOUT
    with pytest.raises(P.OscarsError) as e:
        P.oscars_check_wait_timeout(a.handle, 0)
    assert e.value.status == P.OSCARS_EINVAL
    b, _ = make_context(w, shards, cuda_device)
    for ctx in (a, b):
        for _ in range(2):
            ctx.local_steps()          # reads the error word: it must be clear again
            ctx.push_merge()
    np.testing.assert_array_equal(pull_flat(a, cuda_device), pull_flat(b, cuda_device))
    a.close()
    b.close()


def test_create_out_of_device_memory(cuda_device):
    """A model whose W + 1 parameter slots cannot fit in device memory
    (65 x 8.6 GB): oscars_create returns ENOMEM, creates nothing, and leaves
    the device usable for the next context."""
    x = torch.zeros(64, 1048576, device=cuda_device)
    y = torch.zeros(64, dtype=torch.int32, device=cuda_device)
    with pytest.raises(P.OscarsError) as e:
        P.OscarsContext(num_workers=64, dims=[1048576, 2048, 10], batch=32, lr=0.05, t_ticks=[1] * 64, M=2,
                        shards=[(x, y)] * 64, init_params=torch.zeros(1, device=cuda_device),
                        stream=torch.cuda.current_stream().cuda_stream)
    assert e.value.status == P.OSCARS_ENOMEM
    del x, y
    torch.cuda.empty_cache()
    w = synth.TrainWorkload("after-enomem", 2, [128, 128, 10], 32, 0.05, 64, 4, 1)
    ctx, _ = make_context(w, device_shards(w, cuda_device, n=64), cuda_device)
    ctx.local_steps()
    ctx.push_merge()
    ctx.close()


def test_protocol_errors(cuda_device):
    w = synth.TrainWorkload("small-proto", 2, [128, 128, 10], 32, 0.05, 64, 4, 1)
    ctx, _ = make_context(w, device_shards(w, cuda_device, n=64), cuda_device)
    with pytest.raises(P.OscarsError) as e:
        ctx.push_merge()                         # nothing pushed yet
    assert e.value.status == P.OSCARS_ESTATE
    ctx.local_steps()
    with pytest.raises(P.OscarsError) as e:
        ctx.local_steps()                        # previous round not merged
    assert e.value.status == P.OSCARS_ESTATE
    with pytest.raises(P.OscarsError) as e:
        ctx.set_local_steps([1, 1])
    assert e.value.status == P.OSCARS_ESTATE
    ctx.push_merge()
    ctx.pull(None)                               # explicit broadcast pull
    x = pull_flat(ctx, cuda_device)
    for k in range(2):
        np.testing.assert_array_equal(replica_flat(ctx, k, cuda_device), x)
    ctx.close()


@pytest.mark.parametrize("dims,B", [([784, 512, 10], 64), ([256, 128, 128, 10], 64), ([1024, 256, 128, 10], 64),
                                    ([1000, 256, 128, 10], 32)],
                         ids=["fused", "per-layer", "per-layer-strided", "per-layer-strided-ragged"])
def test_pinned_host_shards_match_device_shards(cuda_device, dims, B):
    """Shards in pinned host memory (read over the host link by the staging
    kernel) give bit-identical rounds to the same shards in device memory.
    The per-layer path stages host rows from a fixed number of blocks
    striding over the tiles; at 1024 inputs a round has more tiles (8 feature
    blocks x 2 row blocks x every (step, worker) slot) than blocks, so each
    block stages several; at 1000 inputs the last feature block of every slot
    holds 104 of 128 columns (the batch of a bf16 MLP is a multiple of the
    32-row block, so row blocks are always whole)."""
    w = synth.TrainWorkload("host-shards", 3, dims, B, 0.05, 256, 6, 2)
    dev_shards = device_shards(w, cuda_device, n=256)
    host_shards = [(x.cpu().pin_memory(), y.cpu().pin_memory()) for x, y in dev_shards]
    outs = []
    for shards in (dev_shards, host_shards):
        ctx, _ = make_context(w, shards, cuda_device)
        for _ in range(2):
            _, loss = ctx.local_steps()
            ctx.push_merge()
        outs.append((pull_flat(ctx, cuda_device), np.array(loss)))
        ctx.close()
    np.testing.assert_array_equal(outs[0][0], outs[1][0])
    np.testing.assert_array_equal(outs[0][1], outs[1][1])


POLICIES = [("oscars", P.POLICY_OSCARS, 1), ("bsp", P.POLICY_BSP, 1), ("local_sgd_3", P.POLICY_LOCAL_SGD, 3)]


@pytest.mark.parametrize("name,policy,period", POLICIES, ids=[p[0] for p in POLICIES])
def test_policies_train_to_loss(cuda_device, name, policy, period):
    """The comparison schemes through the native round runner (oscars_train)
    on the fp32 softmax-regression workload: per-round barriers and clocks
    exact, eval losses within 1e-3, the merged model within 1e-5, and the
    early stop at the first round whose eval loss reaches the target."""
    w = dataclasses.replace(synth.CFG1, samples_per_worker=1024)
    rounds = 8
    t, _, _, _ = oracle_schedule(w)
    tau, barrier = P.oscars_policy_local_steps(policy, t.tolist(), w.M, P.SEARCH_CAPPED, period)
    ora_name = {P.POLICY_OSCARS: "oscars", P.POLICY_BSP: "bsp", P.POLICY_LOCAL_SGD: "local_sgd"}[policy]
    tau_o, barrier_o = orun._sched.policy_local_steps(ora_name, t, M=w.M, period=period)
    assert (tau, barrier) == (tau_o.tolist(), barrier_o)
    Xe, ye = synth.eval_np(w, n=2048)
    shards_h = oracle_inputs(w, w.samples_per_worker)
    layers0 = synth.init_layers_np(w)
    _, full = orun.run(w.dims, layers0, shards_h, t_iter=t, M=w.M, rounds=rounds, batch=w.batch, lr=w.lr,
                       bf16=False, tau_override=tau_o, eval_set=(Xe, ye))
    losses = np.array([r.eval_loss for r in full])
    # a target crossed at a round whose neighbours are far from it
    k = 4
    target = float(0.5 * (losses[k] + losses[k - 1]))
    assert np.all(np.abs(losses - target) > 1e-3 * target)
    k_exp = int(np.argmax(losses <= target))
    ex, ey = torch.from_numpy(Xe).to(cuda_device), torch.from_numpy(ye).to(cuda_device)
    for tgt in (0.0, target):
        ctx, _ = make_context(w, device_shards(w, cuda_device, n=w.samples_per_worker), cuda_device)
        ctx.set_local_steps(tau)
        log = ctx.train(rounds, ex, ey, target_loss=tgt)
        n = rounds if tgt == 0.0 else k_exp + 1
        assert len(log) == n
        for r in range(n):
            assert log[r]["barrier"] == barrier and log[r]["ticks"] == (r + 1) * barrier
            assert abs(log[r]["eval_loss"] - losses[r]) <= LOSS_RTOL * losses[r], (r, log[r], losses[r])
            assert abs(log[r]["worker_loss"] - full[r].worker_loss.mean()) <= LOSS_RTOL * full[r].worker_loss.mean()
        assert_within(per_tensor_errors(pull_flat(ctx, cuda_device), full[n - 1].x_g, w.dims),
                      np.zeros(2), f"{name} after {n} rounds")
        sch = ctx.schedule()
        idle = [barrier - a * b for a, b in zip(tau, t.tolist())]
        assert sch["clock"] == [n * barrier] * w.num_workers and sch["idle"] == [n * i for i in idle]
        ctx.close()
    assert orun.time_to_loss(full, target) == (k_exp + 1) * barrier


def test_drifting_speeds_rescheduled_each_round(cuda_device):
    """Speeds drift every round; oscars_set_iteration_ticks re-runs
    Algorithm 1 before each round.  Per-round tau and barrier exact, clocks
    and idle times exact, merged model within 1e-5 and losses within 1e-3
    (fp32 softmax regression)."""
    w = dataclasses.replace(synth.CFG1, samples_per_worker=1024)
    rounds = 6
    sp = synth.drifting_speeds(w, rounds, sigma=0.4)
    ts = [P.oscars_iteration_ticks(sp[r].tolist(), w.ticks_per_unit) for r in range(rounds)]
    assert len({tuple(t) for t in ts}) > 1
    ctx, layers0 = make_context(w, device_shards(w, cuda_device, n=w.samples_per_worker), cuda_device)
    ctx.set_iteration_ticks(ts[0])
    losses, flats, taus = [], [], []
    for r in range(rounds):
        if r > 0:
            ctx.set_iteration_ticks(ts[r])
        tau, loss = ctx.local_steps()
        ctx.push_merge()
        taus.append(list(tau))
        losses.append(np.array(loss))
        flats.append(pull_flat(ctx, cuda_device))
    sch = ctx.schedule()
    ctx.close()
    state, recs = orun.run(w.dims, layers0, oracle_inputs(w, w.samples_per_worker), M=w.M, rounds=rounds,
                           batch=w.batch, lr=w.lr, bf16=False, t_per_round=[np.asarray(t) for t in ts])
    for r in range(rounds):
        assert taus[r] == recs[r].tau.tolist(), r
        np.testing.assert_allclose(losses[r], recs[r].worker_loss, rtol=LOSS_RTOL)
        assert_within(per_tensor_errors(flats[r], recs[r].x_g, w.dims), np.zeros(2), f"round {r}")
    assert sch["clock"] == state.clock.tolist() and sch["idle"] == state.idle.tolist()
    assert sch["T_star"] == recs[-1].T_star


def test_shards_partitioned_by_tau(cuda_device):
    """Data-partition load balancing: one data set cut into contiguous shards
    sized by tau (oscars_partition_sizes), so the shards differ in size and
    every cursor wraps in the same round.  fp32 softmax regression, 4 rounds
    (the wrap falls inside), against the oracle on the same slices."""
    from oracle import partition as opart
    w = synth.CFG1
    _, _, _, tau = oracle_schedule(w)
    total = 3 * int(tau.sum()) * w.batch
    sizes = P.oscars_partition_sizes([int(v) for v in tau], total, w.batch)
    assert sizes == opart.partition_sizes(tau.tolist(), total, w.batch)
    assert len(set(sizes)) > 1
    X, y = synth.shard_np(w, 0, n=total)
    offs = np.concatenate([[0], np.cumsum(sizes)])
    Xd, yd = torch.from_numpy(X).to(cuda_device), torch.from_numpy(y).to(cuda_device)
    shards_d = [(Xd[a:b], yd[a:b]) for a, b in zip(offs[:-1], offs[1:])]
    shards_h = [(X[a:b], y[a:b]) for a, b in zip(offs[:-1], offs[1:])]
    ctx, layers0 = make_context(w, shards_d, cuda_device)
    flats, losses = [], []
    for _ in range(4):
        _, loss = ctx.local_steps()
        ctx.push_merge()
        losses.append(np.array(loss))
        flats.append(pull_flat(ctx, cuda_device))
    ctx.close()
    t, _, _, _ = oracle_schedule(w)
    state, recs = orun.run(w.dims, layers0, shards_h, t_iter=t, M=w.M, rounds=4, batch=w.batch, lr=w.lr,
                           bf16=False)
    for r in range(4):
        np.testing.assert_allclose(losses[r], recs[r].worker_loss, rtol=LOSS_RTOL)
        assert_within(per_tensor_errors(flats[r], recs[r].x_g, w.dims), np.zeros(2), f"round {r}")
    assert state.cursor.tolist() == (tau.astype(np.int64) * w.batch).tolist()   # wrapped after round 3


def kernel_classes(w, device, rows):
    """Kernel classes one round of a context runs (profiling context)."""
    ctx, _ = make_context(w, device_shards(w, device, n=rows), device, flags=P.FLAG_PROFILE)
    ctx.local_steps()
    ctx.push_merge()
    names = set(ctx.profile())
    ctx.close()
    return names


FUSED_VARIANTS = [
    # name, dims, W, B, one-launch round expected
    ("b32-pair", [784, 512, 10], 3, 32, True),       # two CTAs per unit group, batch 32
    ("b32-single", [384, 768, 10], 2, 32, True),     # one CTA per group (cluster of 6)
    ("ragged-d", [200, 256, 10], 3, 64, True),       # 200 inputs: partial K-block and weight-gradient tile
    ("b64-single", [384, 768, 10], 2, 64, False),    # too large for one CTA per group: per-layer path
]


@pytest.mark.parametrize("name,dims,W,B,fused", FUSED_VARIANTS, ids=[v[0] for v in FUSED_VARIANTS])
def test_round_kernel_variants(cuda_device, name, dims, W, B, fused):
    """Shapes of the one-launch round kernel beyond the headline one, and a
    shape it refuses: the path taken is checked, then one exact step on
    integer inputs (1e-5 per tensor) and three rounds on Gaussian inputs
    (conditioning envelope) against the oracle."""
    rows = 4 * B
    w = synth.TrainWorkload(f"variant-{name}", W, dims, B, 0.05, rows, 6, 3)
    names = kernel_classes(w, cuda_device, rows)
    assert ("fused_round" in names) == fused, names
    run_both(w, 1, cuda_device, rows=rows, tau_override=[1] * W, exact_inputs=True, eval_n=2 * B)
    run_both(w, 3, cuda_device, rows=rows, eval_n=2 * B)


def test_losses_async_matches_synchronous_read(cuda_device):
    w = synth.TrainWorkload("small-async", 3, [256, 128, 10], 32, 0.05, 128, 4, 2)
    ctx, _ = make_context(w, device_shards(w, cuda_device, n=128), cuda_device)
    buf = torch.empty(3, dtype=torch.float32).pin_memory()
    with pytest.raises(P.OscarsError) as e:
        ctx.losses_async(buf)                    # no round yet
    assert e.value.status == P.OSCARS_ESTATE
    for _ in range(2):
        _, loss = ctx.local_steps()
        buf.fill_(-1.0)
        ctx.losses_async(buf)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(buf.numpy(), np.asarray(loss, np.float32))
        ctx.push_merge()
    ctx.close()


@pytest.mark.parametrize("dims,bf16,B", [([784, 512, 10], True, 64), ([256, 256, 128, 10], True, 64),
                                         ([784, 10], False, 32)],
                         ids=["one-launch", "per-layer", "softmax-regression"])
def test_train_without_eval_matches_round_by_round(cuda_device, dims, bf16, B):
    """oscars_train without evaluation pipelines its rounds one deep; the
    models and per-round losses must be those of the same rounds run one
    call at a time (bit for bit: the same kernels in the same order)."""
    w = synth.TrainWorkload("train-pipe", 4, dims, B, 0.05, 512, 8, 5, bf16=bf16)
    shards = device_shards(w, cuda_device, n=512)
    a, _ = make_context(w, shards, cuda_device)
    log = a.train(5)
    assert len(log) == 5
    b, _ = make_context(w, shards, cuda_device)
    for r in range(5):
        _, loss = b.local_steps()
        b.push_merge()
        assert log[r]["worker_loss"] == pytest.approx(float(np.mean(np.asarray(loss, np.float64))), rel=1e-6)
        assert np.isnan(log[r]["eval_loss"])
        assert log[r]["ticks"] == b.schedule()["clock"][0]
    np.testing.assert_array_equal(pull_flat(a, cuda_device), pull_flat(b, cuda_device))
    a.close()
    b.close()


@pytest.mark.parametrize("ref_flags,flags", [(0, P.FLAG_NO_GRAPH), (0, P.FLAG_PROFILE),
                                             (P.FLAG_BRANCHES, P.FLAG_BRANCHES | P.FLAG_NO_GRAPH)],
                         ids=["no-graph", "profile", "branches"])
def test_train_matches_other_launch_modes(cuda_device, ref_flags, flags):
    """oscars_train with its rounds and merges launched as CUDA graphs must
    train the same model bit for bit as without graphs or while profiling
    (also with the workers' kernels on concurrent stream branches)."""
    w = synth.TrainWorkload("train-modes", 4, [256, 256, 128, 10], 64, 0.05, 512, 8, 5)
    shards = device_shards(w, cuda_device, n=512)
    a, _ = make_context(w, shards, cuda_device, flags=ref_flags)
    b, _ = make_context(w, shards, cuda_device, flags=flags)
    la, lb = a.train(4), b.train(4)
    assert [r["worker_loss"] for r in la] == [r["worker_loss"] for r in lb]
    np.testing.assert_array_equal(pull_flat(a, cuda_device), pull_flat(b, cuda_device))
    a.close()
    b.close()


@pytest.mark.parametrize("dims", [[784, 512, 10], [256, 256, 128, 10]], ids=["one-launch", "per-layer"])
def test_train_follows_schedule_changes(cuda_device, dims):
    """oscars_train pipelines its rounds through cached round and merge
    graphs; between calls a tau override, an evaluation (which reuses the
    first input buffer) and new iteration times (Algorithm 1 again, new merge
    weights) must reach the next call's rounds.  Against the same rounds run
    one call at a time, bit for bit."""
    w = synth.TrainWorkload("train-sched", 4, dims, 64, 0.05, 1024, 8, 1)
    shards = device_shards(w, cuda_device, n=w.samples_per_worker)
    Xe, ye = synth.eval_np(w, n=128)
    ex, ey = torch.from_numpy(Xe).to(cuda_device), torch.from_numpy(ye).to(cuda_device)
    t_new = (oracle_schedule(w)[0][::-1]).copy()
    a, _ = make_context(w, shards, cuda_device, weight_rule=P.W_LOCALSTEPS)
    b, _ = make_context(w, shards, cuda_device, weight_rule=P.W_LOCALSTEPS)
    logs = []
    plan = [("train", 2), ("tau", [2, 1, 3, 1]), ("train", 2), ("eval", None), ("ticks", t_new), ("train", 3)]
    for op, arg in plan:
        if op == "train":
            logs += a.train(arg)
            for k in range(arg):
                _, loss = b.local_steps()
                b.push_merge()
                assert logs[len(logs) - arg + k]["worker_loss"] == pytest.approx(
                    float(np.mean(np.asarray(loss, np.float64))), rel=1e-6)
        elif op == "tau":
            a.set_local_steps(arg)
            b.set_local_steps(arg)
        elif op == "eval":
            assert a.eval_loss(ex, ey) == b.eval_loss(ex, ey)
        else:
            a.set_iteration_ticks(arg.tolist())
            b.set_iteration_ticks(arg.tolist())
    np.testing.assert_array_equal(a.schedule()["clock"], b.schedule()["clock"])
    np.testing.assert_array_equal(pull_flat(a, cuda_device), pull_flat(b, cuda_device))
    a.close()
    b.close()


@pytest.mark.parametrize("dims,kernel,host", [([784, 512, 10], "fused_round", False),
                                              ([256, 256, 128, 10], "gemm_dw_sgd", False),
                                              ([512, 256, 128, 10], "gemm_dw_sgd", True)],
                         ids=["one-launch", "per-layer", "per-layer-host-shards"])
def test_round_kernel_restaging_between_rounds(cuda_device, dims, kernel, host):
    """Both round paths stage the next round's mini-batches while the current
    round runs (from host-resident shards, the per-layer path with a fixed
    number of blocks striding over the tiles).  Between rounds: an evaluation
    (which reuses the first input buffer), a tau override, new iteration
    times (Algorithm 1 again) and a plain round; the staged data must follow
    every change.  Against the oracle driven through the same changes."""
    from oracle import schedule as osched
    w = synth.TrainWorkload("restage", 4, dims, 64, 0.05, 1024, 8, 1)
    shards = device_shards(w, cuda_device, n=w.samples_per_worker)
    if host:
        shards = [(x.cpu().pin_memory(), y.cpu().pin_memory()) for x, y in shards]
    ctx, layers0 = make_context(w, shards, cuda_device, flags=P.FLAG_PROFILE)
    Xe, ye = synth.eval_np(w, n=128)
    ex, ey = torch.from_numpy(Xe).to(cuda_device), torch.from_numpy(ye).to(cuda_device)
    t0 = oracle_schedule(w)[0]
    t_new = (t0[::-1]).copy()                      # the speeds swap
    plan = ["round", "eval", "round", "tau", "round", "ticks", "round", "round"]
    gpu_flats, gpu_losses = [], []
    for op in plan:
        if op == "round":
            _, loss = ctx.local_steps()
            ctx.push_merge()
            gpu_losses.append(np.array(loss))
            gpu_flats.append(pull_flat(ctx, cuda_device))
        elif op == "eval":
            ctx.eval_loss(ex, ey)
        elif op == "tau":
            ctx.set_local_steps([2, 1, 3, 1])
        elif op == "ticks":
            ctx.set_iteration_ticks(t_new.tolist())
    assert kernel in ctx.profile()
    ctx.close()

    def oracle_run():
        state = orun.init_state(w.dims, layers0, t0, w.M)
        shards_h = oracle_inputs(w, w.samples_per_worker)
        flats, losses = [], []
        for op in plan:
            if op == "round":
                rec = orun.run_round(state, shards_h, w.batch, w.lr, obf16.round_bf16)
                flats.append(rec.x_g)
                losses.append(rec.worker_loss)
            elif op == "tau":
                state.tau = np.array([2, 1, 3, 1], np.int32)
                state.T_star = osched.round_barrier(state.t_iter, state.tau)
            elif op == "ticks":
                orun.reschedule(state, t_new, w.M)
        return flats, losses
    ref, ref_losses = oracle_run()
    env = envelope(lambda: oracle_run()[0], w.dims, ref)
    for r in range(len(ref)):
        np.testing.assert_allclose(gpu_losses[r], ref_losses[r], rtol=LOSS_RTOL)
        assert_within(per_tensor_errors(gpu_flats[r], ref[r], w.dims), env[r], f"round {r}")
