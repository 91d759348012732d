"""No kernel writes outside its tensors (the memory checker is closed on
this GPU pool, so the library checks its own layout): after rounds of every
round-kernel path, an evaluation and the merge, every padding value of the
fp32 slab and of its bf16 copy is still zero and the guard words after both
still hold the pattern written at creation (oscars_check_padding)."""
import numpy as np
import pytest
import torch

import paper_2102_08550_gb300 as P
import synth
from tests.gpu_util import device_shards, make_context

pytestmark = pytest.mark.gpu

CASES = [
    # name, dims, W, batch, rows, bf16, flags
    ("fused-b64-tensor-core-head", [784, 512, 10], 16, 64, 256, True, 0),
    ("fused-b32-pair", [784, 512, 10], 3, 32, 128, True, 0),
    ("fused-b32-single", [384, 768, 10], 2, 32, 128, True, 0),
    ("fused-ragged-d", [200, 256, 10], 3, 64, 256, True, 0),
    ("per-layer-3layer", [200, 256, 128, 10], 3, 32, 128, True, 0),
    ("per-layer-4layer", [96, 128, 256, 128, 10], 3, 128, 256, True, 0),
    ("per-layer-2layer", [784, 512, 10], 3, 64, 256, True, P.FLAG_PER_LAYER),
    ("softreg-cluster-ragged", [18, 10], 3, 20, 100, False, 0),
    ("softreg-cluster-scalar", [785, 10], 3, 32, 128, False, 0),
    ("softreg-one-cta", [64, 10], 2, 300, 600, False, 0),
]


@pytest.mark.parametrize("name,dims,W,B,rows,bf16,flags", CASES, ids=[c[0] for c in CASES])
def test_padding_and_guards_untouched(cuda_device, name, dims, W, B, rows, bf16, flags):
    w = synth.TrainWorkload(f"pad-{name}", W, dims, B, 0.05, rows, 6, 3, bf16=bf16)
    ctx, _ = make_context(w, device_shards(w, cuda_device, n=rows), cuda_device, flags=flags)
    assert P.oscars_check_padding(ctx.handle) == 0          # as created
    Xe, ye = synth.eval_np(w, n=2 * B)
    for _ in range(3):
        ctx.local_steps()
        ctx.push_merge()
    ctx.eval_loss(torch.from_numpy(Xe).to(cuda_device), torch.from_numpy(ye).to(cuda_device))
    out = torch.empty(ctx.P, device=cuda_device)
    ctx.read_replica(W - 1, out)
    ctx.pull(out)
    ctx.pull(None)                                          # broadcast into every replica
    assert P.oscars_check_padding(ctx.handle) == 0
    assert np.isfinite(out.cpu().numpy()).all()
    ctx.close()


def test_padding_check_sees_a_planted_write(cuda_device):
    """The check is not vacuous: one float added into the padding after b_1 of
    worker 1's slot (through the slab's device address and the context-free
    merge entry) is counted, and only that one."""
    w = synth.TrainWorkload("pad-planted", 2, [200, 256, 10], 64, 0.05, 128, 6, 1)
    ctx, _ = make_context(w, device_shards(w, cuda_device, n=128), cuda_device)
    ctx.local_steps()
    ctx.push_merge()
    assert P.oscars_check_padding(ctx.handle) == 0
    slab, stride = P.oscars_debug_slab(ctx.handle)
    # layout: W_0 (51200), b_0 (256), W_1 (2560), b_1 (10, padded to 64)
    off_b1 = 51200 + 256 + 2560
    assert stride == off_b1 + 64
    one = torch.ones(1, device=cuda_device)
    P.oscars_merge(slab + 4 * (stride + off_b1 + 20), [one.data_ptr()], [1.0], 1, 1.0,
                   torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert P.oscars_check_padding(ctx.handle) == 1
    ctx.close()
