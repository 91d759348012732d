"""The allocation-free entry point, oscars_softreg_steps_noalloc: one worker's
fp32 softmax-regression local steps for callers that cannot allocate device
memory at the call (code recording a CUDA graph in global capture mode, hosts
whose own pool owns the GPU, loops that cannot pay for cudaMalloc/cudaFree).

It is checked against the context path it mirrors and against the oracle on
two calls in a row, in place (params_in == params_out), on a shard that is
not 16-byte aligned, at the largest batch, and for every refusal it
documents.  Collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test."""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2102_08550_gb300 as P
import synth
from oracle import bf16 as obf16
from oracle import model as omodel
from tests.gpu_util import LOSS_RTOL, PARAM_RTOL, make_context, pull_flat, rel_maxabs, replica_flat

pytestmark = pytest.mark.gpu


def oracle_steps(flat, X, y, cursor, tau, D, C, B, lr):
    """tau local steps of the oracle on rows (cursor + s*B + b) mod n."""
    layers = [(flat[:C * D].reshape(C, D).copy(), flat[C * D:C * D + C].copy())]
    losses = []
    for s in range(tau):
        idx = (cursor + s * B + np.arange(B)) % X.shape[0]
        layers, loss = omodel.sgd_step(layers, X[idx], y[idx], lr, obf16.identity)
        losses.append(loss)
    return synth.flatten_layers(layers), float(np.mean(losses))


def check(got, loss, ref, ref_loss, C, D):
    assert rel_maxabs(got[:C * D], ref[:C * D]) <= PARAM_RTOL
    assert rel_maxabs(got[C * D:], ref[C * D:]) <= PARAM_RTOL
    assert abs(loss - ref_loss) <= LOSS_RTOL * abs(ref_loss)


def call(pin, pout, x, y, n, cursor, tau, D, C, B, lr, loss):
    P.oscars_softreg_steps_noalloc(pin.data_ptr(), pout.data_ptr(), x.data_ptr(), y.data_ptr(), n, cursor, tau,
                                   D, C, B, lr, loss.data_ptr(), torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()


def test_noalloc_matches_context_and_oracle_two_calls(cuda_device):
    w = dataclasses.replace(synth.CFG1, samples_per_worker=512)
    shards = [synth.shard_t(w, k, cuda_device, n=512) for k in range(w.num_workers)]
    ctx, layers0 = make_context(w, shards, cuda_device)
    k = 3                                          # the worker with the most local steps
    tau = ctx.schedule()["tau"][k]
    D, C, B = w.dims[0], w.dims[1], w.batch
    Xh, yh = synth.shard_np(w, k, n=512)
    x0 = torch.from_numpy(synth.flatten_layers(layers0)).to(cuda_device)
    out = torch.empty_like(x0)
    loss = torch.empty(1, device=cuda_device)
    start = x0
    for rnd in range(2):                           # two rounds: context, oracle and the no-alloc call
        cursor = rnd * tau * B
        _, ctx_loss = ctx.local_steps()
        ctx_rep = replica_flat(ctx, k, cuda_device)
        call(start, out, shards[k][0], shards[k][1], 512, cursor, tau, D, C, B, w.lr, loss)
        got = out.cpu().numpy()
        check(got, loss.item(), ctx_rep, ctx_loss[k], C, D)
        ref, ref_loss = oracle_steps(start.cpu().numpy(), Xh, yh, cursor, tau, D, C, B, w.lr)
        check(got, loss.item(), ref, ref_loss, C, D)
        ctx.push_merge()
        start = torch.from_numpy(pull_flat(ctx, cuda_device)).to(cuda_device)   # the next round's global model
    ctx.close()


def test_noalloc_in_place_unaligned_and_largest_batch(cuda_device):
    """params_in == params_out gives the out-of-place result bit for bit; a
    shard starting 4 bytes past a 16-byte boundary (scalar row loads) gives
    the aligned result bit for bit; batch 512 (the largest) and a shard that
    wraps within the call match the oracle."""
    D, C, B, n, tau, lr = 64, 10, 512, 1300, 5, 0.05
    w = synth.TrainWorkload("noalloc-b512", 1, [D, C], B, lr, n, 4, 1, bf16=False)
    Xh, yh = synth.shard_np(w, 0, n=n)
    flat0 = synth.flatten_layers(synth.init_layers_np(w))
    dev = cuda_device
    x = torch.from_numpy(Xh).to(dev)
    y = torch.from_numpy(yh).to(dev)
    xu_buf = torch.zeros(n * D + 4, device=dev)    # the same rows one float past an aligned start
    xu_buf[1:1 + n * D] = x.reshape(-1)
    xu = xu_buf[1:]
    assert xu.data_ptr() % 16 == 4
    x0 = torch.from_numpy(flat0).to(dev)
    loss = torch.empty(1, device=dev)
    out = torch.empty_like(x0)
    call(x0, out, x, y, n, 300, tau, D, C, B, lr, loss)
    ref, ref_loss = oracle_steps(flat0, Xh, yh, 300, tau, D, C, B, lr)
    check(out.cpu().numpy(), loss.item(), ref, ref_loss, C, D)
    inplace = x0.clone()
    loss2 = torch.empty(1, device=dev)
    call(inplace, inplace, x, y, n, 300, tau, D, C, B, lr, loss2)
    torch.testing.assert_close(inplace, out, rtol=0, atol=0)
    assert loss2.item() == loss.item()
    un = torch.empty_like(x0)
    call(x0, un, xu, y, n, 300, tau, D, C, B, lr, loss2)
    torch.testing.assert_close(un, out, rtol=0, atol=0)
    assert loss2.item() == loss.item()


@pytest.mark.parametrize("tau,D,C,B,status", [
    (16321, 784, 10, 32, P.OSCARS_EINVAL),         # one step more than the scratch holds
    (1, 784, 1, 32, P.OSCARS_EINVAL),              # classes below 2
    (1, 784, 33, 32, P.OSCARS_EINVAL),             # classes above 32
    (1, 64, 10, 513, P.OSCARS_ENOTSUP),            # batch above 512
    (1, 4096, 10, 32, P.OSCARS_ENOTSUP),           # weights plus one batch beyond shared memory
], ids=["tau", "classes-1", "classes-33", "batch-513", "smem"])
def test_noalloc_refusals(cuda_device, tau, D, C, B, status):
    buf = torch.zeros(C * D + C, device=cuda_device)
    x = torch.zeros(B, D, device=cuda_device)
    y = torch.zeros(B, dtype=torch.int32, device=cuda_device)
    loss = torch.zeros(1, device=cuda_device)
    with pytest.raises(P.OscarsError) as e:
        P.oscars_softreg_steps_noalloc(buf.data_ptr(), buf.data_ptr(), x.data_ptr(), y.data_ptr(), B, 0,
                                       tau, D, C, B, 0.05, loss.data_ptr())
    assert e.value.status == status


def test_noalloc_largest_tau(cuda_device):
    """tau = 16320, the most the scratch holds: the per-step loss partials fill
    it; the mean loss over all steps matches the oracle's."""
    D, C, B, n, tau, lr = 16, 2, 4, 64, 16320, 0.01
    w = synth.TrainWorkload("noalloc-tau", 1, [D, C], B, lr, n, 4, 1, bf16=False)
    Xh, yh = synth.shard_np(w, 0, n=n)
    yh = (yh % C).astype(np.int32)
    flat0 = synth.flatten_layers(synth.init_layers_np(w))
    dev = cuda_device
    x0 = torch.from_numpy(flat0).to(dev)
    out = torch.empty_like(x0)
    loss = torch.empty(1, device=dev)
    call(x0, out, torch.from_numpy(Xh).to(dev), torch.from_numpy(yh).to(dev), n, 0, tau, D, C, B, lr, loss)
    ref, ref_loss = oracle_steps(flat0, Xh, yh, 0, tau, D, C, B, lr)
    assert abs(loss.item() - ref_loss) <= LOSS_RTOL * abs(ref_loss)
    assert rel_maxabs(out.cpu().numpy(), ref) <= 1e-3      # 16320 fp32 steps: summation order drifts
