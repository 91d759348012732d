"""The allocation-free entry point (for callers that cannot allocate device
memory at the call, e.g. while recording a CUDA graph) against the context
path it mirrors: one worker's fp32 softmax-regression local steps, two calls
in a row, within the parity tolerances of the other tests.  Collected last
on purpose."""
import dataclasses

import numpy as np
import pytest
import torch

import paper_2102_08550_gb300 as P
import synth
from tests.gpu_util import LOSS_RTOL, PARAM_RTOL, make_context, pull_flat, rel_maxabs, replica_flat

pytestmark = pytest.mark.gpu


def test_noalloc_matches_context_two_calls(cuda_device):
    w = dataclasses.replace(synth.CFG1, samples_per_worker=512)
    shards = [synth.shard_t(w, k, cuda_device, n=512) for k in range(w.num_workers)]
    ctx, layers0 = make_context(w, shards, cuda_device)
    k = 3                                          # the worker with the most local steps
    tau = ctx.schedule()["tau"][k]
    D, C, B = w.dims[0], w.dims[1], w.batch
    x0 = torch.from_numpy(synth.flatten_layers(layers0)).to(cuda_device)
    out = torch.empty_like(x0)
    loss = torch.empty(1, device=cuda_device)
    stream = torch.cuda.current_stream().cuda_stream
    start = x0
    for call in range(2):                          # two rounds: context vs the no-alloc call
        _, ctx_loss = ctx.local_steps()
        ref = replica_flat(ctx, k, cuda_device)
        P.oscars_softreg_steps_noalloc(start.data_ptr(), out.data_ptr(), shards[k][0].data_ptr(),
                                       shards[k][1].data_ptr(), 512, call * tau * B, tau, D, C, B, w.lr,
                                       loss.data_ptr(), stream)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert rel_maxabs(got[:C * D], ref[:C * D]) <= PARAM_RTOL
        assert rel_maxabs(got[C * D:], ref[C * D:]) <= PARAM_RTOL
        assert abs(loss.item() - ctx_loss[k]) <= LOSS_RTOL * abs(ctx_loss[k])
        ctx.push_merge()
        start = torch.from_numpy(pull_flat(ctx, cuda_device)).to(cuda_device)   # the next round's global model
    ctx.close()


def test_noalloc_rejects_oversized(cuda_device):
    buf = torch.zeros(7850, device=cuda_device)
    x = torch.zeros(64, 784, device=cuda_device)
    y = torch.zeros(64, dtype=torch.int32, device=cuda_device)
    loss = torch.zeros(1, device=cuda_device)
    with pytest.raises(P.OscarsError) as e:
        P.oscars_softreg_steps_noalloc(buf.data_ptr(), buf.data_ptr(), x.data_ptr(), y.data_ptr(), 64, 0,
                                       1_000_000, 784, 10, 32, 0.05, loss.data_ptr())
    assert e.value.status == P.OSCARS_EINVAL
