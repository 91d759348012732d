"""Server merge and global update (Eq. 4, first branch) on the GPU against
the oracle: small exhaustive cases (odd P, tails, unaligned pointers, W=1)
and sampled elements of the two full-size microbench workloads."""
import numpy as np
import pytest
import torch

import paper_2102_08550_gb300 as P
import synth
from oracle import merge as omerge
from oracle import schedule as osched
from tests.gpu_util import PARAM_RTOL, rel_maxabs

pytestmark = pytest.mark.gpu


# offset: elements before every buffer.  With (Pn + offset) % 4 == 0 all the
# buffers share one misalignment (the vector kernel after a peeled scalar
# head: (5, 4099, 1), (17, 777, 3), (5, 7, 1), (9, 4095, 1) with no tail, and
# (5, 3, 1) where the head is all of P); otherwise the delta rows are
# misaligned differently and the scalar kernel takes the whole vector
# ((4, 1001, 1)).
@pytest.mark.parametrize("W,Pn,offset", [(1, 1, 0), (1, 7, 0), (3, 1023, 0), (8, 4096, 0), (5, 4099, 1),
                                           (64, 10001, 0), (17, 777, 3), (256, 513, 0), (5, 3, 1), (5, 7, 1),
                                           (9, 4095, 1), (4, 1001, 1)])
def test_merge_small(cuda_device, W, Pn, offset):
    rng = np.random.default_rng(W * 1000 + Pn)
    xg = rng.standard_normal(Pn).astype(np.float32)
    d = (rng.standard_normal((W, Pn)) * 1e-3).astype(np.float32)
    w = rng.random(W).astype(np.float32)
    eta = 0.75
    ref = omerge.merge_deltas(xg, list(d), w, eta)
    # allocate with an element offset to exercise unaligned pointers
    xg_t = torch.zeros(Pn + offset, device=cuda_device)
    xg_t[offset:] = torch.from_numpy(xg).to(cuda_device)
    d_t = torch.zeros(W, Pn + offset, device=cuda_device)
    d_t[:, offset:] = torch.from_numpy(d).to(cuda_device)
    P.oscars_merge(xg_t[offset:].data_ptr(), [d_t[k, offset:].data_ptr() for k in range(W)], w.tolist(), Pn, eta,
                   torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    got = xg_t[offset:].cpu().numpy()
    assert rel_maxabs(got, ref) <= PARAM_RTOL
    assert np.all(xg_t[:offset].cpu().numpy() == 0)


def test_merge_context_flat_rules(cuda_device):
    rng = np.random.default_rng(1)
    W, Pn = 6, 3333
    x0 = rng.standard_normal(Pn).astype(np.float32)
    d = (rng.standard_normal((W, Pn)) * 1e-3).astype(np.float32)
    tau = [3, 1, 4, 1, 5, 9]
    d_t = torch.from_numpy(d).to(cuda_device)
    for rule, name in ((P.W_UNIFORM, "uniform"), (P.W_LOCALSTEPS, "localsteps"), (P.W_EXPLICIT, "explicit")):
        ctx = P.OscarsContext(num_workers=W, dims=[Pn], model=P.MODEL_FLAT, weight_rule=rule,
                              t_ticks=[1] * W, M=2, init_params=torch.from_numpy(x0).to(cuda_device),
                              server_lr=1.0, stream=torch.cuda.current_stream().cuda_stream)
        ctx.set_local_steps(tau)
        ew = rng.random(W).astype(np.float32)
        ctx.push_merge(list(d_t), ew.tolist() if rule == P.W_EXPLICIT else None)
        # a second merge in a row: the update composes
        ctx.push_merge(list(d_t), ew.tolist() if rule == P.W_EXPLICIT else None)
        out = torch.empty(Pn, device=cuda_device)
        ctx.pull(out)
        torch.cuda.synchronize()
        w = osched.merge_weights(name, tau, ew)
        ref = omerge.merge_deltas(omerge.merge_deltas(x0, list(d), w), list(d), w)
        assert rel_maxabs(out.cpu().numpy(), ref) <= PARAM_RTOL, name
        ctx.close()


def test_merge_context_errors(cuda_device):
    ctx = P.OscarsContext(num_workers=2, dims=[16], model=P.MODEL_FLAT, t_ticks=[1, 1], M=2)
    with pytest.raises(P.OscarsError) as e:
        ctx.push_merge(None)               # FLAT: no replicas to merge
    assert e.value.status == P.OSCARS_ESTATE
    with pytest.raises(P.OscarsError) as e:
        P.oscars_local_steps(ctx.handle)
    assert e.value.status == P.OSCARS_ESTATE
    ctx.close()


def _full_size_merge(cuda_device, m: synth.MergeWorkload, rule_name: str):
    W, Pn = m.num_workers, m.num_params
    taus = synth.merge_taus(m)
    rule = P.W_LOCALSTEPS if rule_name == "localsteps" else P.W_UNIFORM
    xg0 = synth.merge_xg_t(m, 0, Pn, cuda_device)
    deltas = [synth.merge_delta_t(m, k, 0, Pn, cuda_device) for k in range(W)]
    ctx = P.OscarsContext(num_workers=W, dims=[Pn], model=P.MODEL_FLAT, weight_rule=rule, t_ticks=[1] * W, M=2,
                          init_params=xg0, server_lr=m.server_lr, stream=torch.cuda.current_stream().cuda_stream)
    del xg0
    ctx.set_local_steps(taus.tolist())
    ctx.push_merge(deltas)
    out = torch.empty(Pn, device=cuda_device)
    ctx.pull(out)
    torch.cuda.synchronize()
    idx = np.unique(np.concatenate([np.random.default_rng(5).integers(0, Pn, 20000), [0, 1, 2, Pn - 1]]))
    got = out[torch.from_numpy(idx).to(cuda_device)].cpu().numpy()
    w = osched.merge_weights(rule_name, taus)
    ref = omerge.merge_deltas(synth.merge_xg_np(m, idx), [synth.merge_delta_np(m, k, idx) for k in range(W)], w,
                              m.server_lr)
    ctx.close()
    del deltas, out
    torch.cuda.empty_cache()
    return rel_maxabs(got, ref)


def test_merge_full_size_p25m_w64(cuda_device):
    assert _full_size_merge(cuda_device, synth.CFG4, "localsteps") <= PARAM_RTOL


@pytest.mark.parametrize("rule", ["uniform", "localsteps"])
def test_merge_full_size_p340m_w8(cuda_device, rule):
    assert _full_size_merge(cuda_device, synth.CFG5, rule) <= PARAM_RTOL
