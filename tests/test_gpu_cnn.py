"""The convolutional worker on the GPU against the oracle (oracle/conv.py):
schedules exact, merged parameters per tensor within 1e-5 or the measured
conditioning envelope of the oracle (bf16 rounding and ReLU masks amplify
fp32 summation-order differences), worker losses and eval loss within 1e-3.

Cases: small runs of one and two residual blocks through two rounds (the
second round starts from the merged model; 3 input channels take the im2col
stem, 16 the nine-tap one), and the full-size workload (16 workers, batch
32) for one full round: every worker's replica and the merged model."""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2102_08550_gb300 as P
import synth
from oracle import bf16 as obf16
from oracle import conv as oconv
from oracle import run as orun
from tests.gpu_util import LOSS_RTOL, assert_within, envelope, oracle_schedule, per_tensor_errors

pytestmark = pytest.mark.gpu


def cnn_errors(m, got, ref):
    """Per-tensor max-abs error / max-abs value (canonical order)."""
    out = []
    for g, r in zip(m.unflatten(got), m.unflatten(ref)):
        den = np.abs(r).max()
        out.append(float(np.abs(g.astype(np.float64) - r).max() / (den if den > 0 else 1.0)))
    return out


def make_cnn_context(w, device, rows, flags=0):
    shards = [synth.shard_t(w, k, device, n=rows) for k in range(w.num_workers)]
    params0 = synth.init_cnn_np(w)
    m = oconv.CNN(w.height, w.width, w.in_ch, w.ch, w.blocks, w.dims[-1])
    init = torch.from_numpy(m.flatten(params0)).to(device)
    ctx = P.OscarsContext(num_workers=w.num_workers, dims=w.cnn_dims, model=P.MODEL_CNN, blocks=w.blocks,
                          batch=w.batch, lr=w.lr, speed=synth.speeds(w).tolist(), M=w.M, shards=shards,
                          init_params=init, stream=torch.cuda.current_stream().cuda_stream, flags=flags)
    return ctx, m, params0


def pull(ctx, device):
    out = torch.empty(ctx.P, dtype=torch.float32, device=device)
    ctx.pull(out)
    torch.cuda.synchronize()
    return out.cpu().numpy()


# (name, blocks, workers, batch, input channels): 3 channels take the im2col
# stem (9 x 3 <= 64 channels), 16 the nine-tap stem
SMALL = [("1block", 1, 3, 16, 3), ("2blocks", 2, 2, 16, 3), ("1block-cin16", 1, 2, 16, 16)]


@pytest.mark.parametrize("name,blocks,W,B,cin", SMALL, ids=[s[0] for s in SMALL])
def test_cnn_small_two_rounds(cuda_device, name, blocks, W, B, cin):
    rows = 4 * B
    w = synth.ConvWorkload(f"cnn-{name}", W, [32 * 32 * cin, 10], B, 0.05, rows, 4, 2, clip=3.0, blocks=blocks,
                           in_ch=cin)
    ctx, m, params0 = make_cnn_context(w, cuda_device, rows)
    rounds = 2
    losses, flats = [], []
    for _ in range(rounds):
        tau, loss = ctx.local_steps()
        ctx.push_merge()
        losses.append(np.array(loss))
        flats.append(pull(ctx, cuda_device))
    Xe, ye = synth.eval_np(w, n=2 * B)
    ge = ctx.eval_loss(torch.from_numpy(Xe).to(cuda_device), torch.from_numpy(ye).to(cuda_device))
    sch = ctx.schedule()
    ctx.close()
    t, T, mw, tau_o = oracle_schedule(w)
    assert sch["tau"] == tau_o.tolist() and sch["T_star"] == T
    shards_h = [synth.shard_np(w, k, n=rows) for k in range(W)]

    def oracle_run():
        return orun.run(None, params0, shards_h, t_iter=t, M=w.M, rounds=rounds, batch=B, lr=w.lr,
                        bf16=True, model=m)
    state, recs = oracle_run()
    env = envelope(lambda: [r.x_g for r in oracle_run()[1]], None, [r.x_g for r in recs],
                   errors=lambda f, ref: cnn_errors(m, f, ref))
    for r in range(rounds):
        np.testing.assert_allclose(losses[r], recs[r].worker_loss, rtol=LOSS_RTOL)
        errs = cnn_errors(m, flats[r], recs[r].x_g)
        assert_within(errs, env[r], f"{name} round {r}")
    oe = m.loss_of(state.x_g, Xe, ye, obf16.round_bf16)   # the model's own structure (state.x_g)
    assert abs(ge - oe) <= LOSS_RTOL * abs(oe), (ge, oe)


def test_cnn_full_size_one_round_every_worker(cuda_device):
    """The 16-worker, batch-32 workload for one full round of its schedule (71
    worker-steps, tau up to 6): every worker's pushed replica and the merged
    model against the oracle (conditioning envelope per tensor), the schedule
    exact and the worker losses within 1e-3."""
    w = synth.CFG6
    t, T, mw, tau = oracle_schedule(w)
    rows = int(tau.max()) * w.batch
    ctx, m, params0 = make_cnn_context(w, cuda_device, rows)
    tau_g, loss = ctx.local_steps()
    assert tau_g == tau.tolist()
    reps = []
    for k in range(w.num_workers):
        out = torch.empty(ctx.P, dtype=torch.float32, device=cuda_device)
        ctx.read_replica(k, out)
        torch.cuda.synchronize()
        reps.append(out.cpu().numpy())
    ctx.push_merge()
    merged = pull(ctx, cuda_device)
    sch = ctx.schedule()
    ctx.close()
    assert sch["T_star"] == T
    shards_h = [synth.shard_np(w, k, n=rows) for k in range(w.num_workers)]

    def oracle_run():
        _, recs = orun.run(None, params0, shards_h, t_iter=t, M=w.M, rounds=1, batch=w.batch, lr=w.lr,
                           bf16=True, model=m, keep_replicas=True)
        return recs[0]

    def flats(rec):
        return [*rec.replicas, rec.x_g]
    rec = oracle_run()
    env = envelope(lambda: flats(oracle_run()), None, flats(rec), errors=lambda f, r: cnn_errors(m, f, r))
    np.testing.assert_allclose(loss, rec.worker_loss, rtol=LOSS_RTOL)
    for k in range(w.num_workers):
        assert_within(cnn_errors(m, reps[k], rec.replicas[k]), env[k], f"worker {k} (tau {int(tau[k])})")
    assert_within(cnn_errors(m, merged, rec.x_g), env[-1], "merged")


def test_cnn_train_matches_round_by_round(cuda_device):
    """oscars_train pipelines the rounds of the convolutional worker and their
    merges (with the transposed-copy refresh); the models and per-round
    losses are those of the same rounds run one call at a time, bit for
    bit."""
    B = 16
    rows = 6 * B
    w = synth.ConvWorkload("cnn-train", 2, [32 * 32 * 3, 10], B, 0.05, rows, 4, 2, clip=3.0, blocks=1, in_ch=3)
    a, _, _ = make_cnn_context(w, cuda_device, rows)
    b, _, _ = make_cnn_context(w, cuda_device, rows)
    log = a.train(3)
    for r in range(3):
        _, loss = b.local_steps()
        b.push_merge()
        assert log[r]["worker_loss"] == pytest.approx(float(np.mean(np.asarray(loss, np.float64))), rel=1e-6)
    np.testing.assert_array_equal(pull(a, cuda_device), pull(b, cuda_device))
    a.close()
    b.close()
