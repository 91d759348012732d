"""C-ABI checks that need no GPU: the library loads, exports every function
declared in include/oscars.h, its host scheduler matches the oracle bit for
bit (Algorithm 1, Eq. 1-3, iteration ticks, merge weights), and invalid
configurations are rejected before any device work."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2102_08550_gb300 as P
from oracle import schedule as S

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "oscars.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(oscars_\w+)\s*\(", text, flags=re.M)))


def test_exports_every_declared_function(oscars_lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(oscars_lib, n), n


def test_status_strings(oscars_lib):
    assert oscars_lib.oscars_status_string(0) == b"OSCARS_OK"
    assert oscars_lib.oscars_status_string(5) == b"OSCARS_ETIMEOUT"


def test_schedule_matches_oracle_golden(oscars_lib):
    from tests.test_oracle_schedule import golden_cases
    for t, M, T_exp, mw_exp, tau_exp, _ in golden_cases():
        assert P.oscars_schedule_solve(t, M) == (T_exp, mw_exp, tau_exp)


def test_schedule_matches_oracle_random(oscars_lib):
    rng = np.random.default_rng(99)
    for trial in range(300):
        n = int(rng.integers(1, 40))
        t = [int(v) for v in rng.integers(1, 3000 if trial % 3 else 20, n)]
        M = int(rng.integers(1, 20))
        T, mw, tau = S.schedule(t, M)
        assert P.oscars_schedule_solve(t, M) == (T, mw, tau.tolist()), (t, M)
        if min(t) < max(t) and trial % 5 == 0:
            Tl, mwl, taul = S.schedule(t, M, S.LITERAL)
            assert P.oscars_schedule_solve(t, M, P.SEARCH_LITERAL) == (Tl, mwl, taul.tolist())


def test_workload_schedules_match_oracle(oscars_lib):
    import synth
    for w in (synth.CFG1, synth.CFG2, synth.CFG3):
        s = synth.speeds(w)
        t = S.iteration_ticks(s, w.ticks_per_unit)
        assert P.oscars_iteration_ticks(s.tolist(), w.ticks_per_unit) == t.tolist()
        T, mw, tau = S.schedule(t, w.M)
        assert P.oscars_schedule_solve(t.tolist(), w.M) == (T, mw, tau.tolist())


def test_iteration_ticks_matches_oracle(oscars_lib):
    rng = np.random.default_rng(3)
    s = np.concatenate([rng.lognormal(0, 1.5, 2000), [0.4, 2.5, 1.6, 3.0, 1e-3, 1e3, 2000.0]])
    for Q in (1, 7, 1000, 12345):
        assert P.oscars_iteration_ticks(s.tolist(), Q) == S.iteration_ticks(s, Q).tolist()


def test_merge_weights_match_oracle(oscars_lib):
    rng = np.random.default_rng(4)
    for _ in range(50):
        tau = rng.integers(1, 17, int(rng.integers(1, 70)))
        got = np.array(P.oscars_merge_weights(P.W_LOCALSTEPS, tau.tolist()), np.float32)
        np.testing.assert_array_equal(got, S.merge_weights("localsteps", tau))
        got = np.array(P.oscars_merge_weights(P.W_UNIFORM, tau.tolist()), np.float32)
        np.testing.assert_array_equal(got, S.merge_weights("uniform", tau))


def test_host_errors(oscars_lib):
    with pytest.raises(P.OscarsError) as e:
        P.oscars_schedule_solve([5, 5], 4, P.SEARCH_LITERAL)
    assert e.value.status == P.OSCARS_EINVAL
    with pytest.raises(P.OscarsError):
        P.oscars_schedule_solve([0, 3], 4)
    with pytest.raises(P.OscarsError):
        P.oscars_schedule_solve([3, 4], 0)
    with pytest.raises(P.OscarsError):
        P.oscars_iteration_ticks([1.0, -2.0])
    with pytest.raises(P.OscarsError):
        P.oscars_schedule_solve([1, 10**15], 8)     # search range too large: refused, not run


def _cfg(**kw):
    cfg = P.OscarsConfig()
    dims = kw.pop("dims", [8, 128, 10])
    arr = (ctypes.c_int32 * len(dims))(*dims)
    cfg.dims = arr
    cfg.num_workers = kw.pop("W", 2)
    cfg.model = kw.pop("model", P.MODEL_MLP)
    cfg.num_layers = len(dims) - 1
    cfg.batch = kw.pop("batch", 32)
    cfg.lr = 0.05
    cfg.server_lr = 1.0
    cfg.bf16_gemm = kw.pop("bf16", 1)
    cfg.M = kw.pop("M", 4)
    t = kw.pop("t", [3, 5])
    tt = (ctypes.c_int64 * len(t))(*t)
    cfg.t_ticks = tt
    cfg.search_mode = kw.pop("mode", 0)
    return cfg, (arr, tt)


@pytest.mark.parametrize("change, status", [
    (dict(W=0), P.OSCARS_EINVAL),
    (dict(M=0), P.OSCARS_EINVAL),
    (dict(t=[0, 5]), P.OSCARS_EINVAL),
    (dict(t=[4, 4], mode=1), P.OSCARS_EINVAL),
    (dict(dims=[8, 100, 10]), P.OSCARS_ENOTSUP),      # hidden dim not a multiple of 128
    (dict(dims=[8, 128, 40]), P.OSCARS_ENOTSUP),      # more than 32 classes
    (dict(batch=48), P.OSCARS_ENOTSUP),
    (dict(), P.OSCARS_EINVAL),                        # valid shape but NULL shards
    (dict(dims=[64, 10], bf16=0, batch=513), P.OSCARS_ENOTSUP),    # fp32 softmax regression: batch > 512
    (dict(dims=[64, 10], bf16=0, batch=512), P.OSCARS_EINVAL),     # batch 512 passes; NULL shards
    (dict(dims=[4096, 10], bf16=0, batch=32), P.OSCARS_ENOTSUP),   # weights + batch beyond shared memory
])
def test_create_rejects_before_device_work(oscars_lib, change, status):
    cfg, keep = _cfg(**change)
    h = ctypes.c_void_p()
    assert oscars_lib.oscars_create(ctypes.byref(cfg), ctypes.byref(h)) == status
    assert h.value is None


def test_destroy_null_is_ok(oscars_lib):
    assert oscars_lib.oscars_destroy(None) == 0


def test_policy_local_steps_match_oracle(oscars_lib):
    rng = np.random.default_rng(17)
    names = {P.POLICY_OSCARS: S.OSCARS, P.POLICY_BSP: S.BSP, P.POLICY_LOCAL_SGD: S.LOCAL_SGD}
    for trial in range(200):
        t = [int(v) for v in rng.integers(1, 2000, int(rng.integers(1, 20)))]
        M = int(rng.integers(1, 12))
        I = int(rng.integers(1, 9))
        for pol, name in names.items():
            tau, B = S.policy_local_steps(name, t, M=M, period=I)
            assert P.oscars_policy_local_steps(pol, t, M, P.SEARCH_CAPPED, I) == (tau.tolist(), B), (pol, t, M, I)


def test_policy_errors(oscars_lib):
    for pol, I in ((3, 1), (P.POLICY_LOCAL_SGD, 0), (-1, 1)):
        with pytest.raises(P.OscarsError):
            P.oscars_policy_local_steps(pol, [3, 5], 4, P.SEARCH_CAPPED, I)
    with pytest.raises(P.OscarsError):
        P.oscars_policy_local_steps(P.POLICY_BSP, [0, 5])


def test_train_rejects_null_context(oscars_lib):
    done = ctypes.c_int32(7)
    assert oscars_lib.oscars_train(None, 1, None, None, 0, 0.0, None, ctypes.byref(done)) == P.OSCARS_EINVAL
    assert done.value == 0


def test_set_iteration_ticks_null_context(oscars_lib):
    t = (ctypes.c_int64 * 2)(3, 5)
    assert oscars_lib.oscars_set_iteration_ticks(None, t) == P.OSCARS_EINVAL


def _cnn_cfg(**kw):
    cfg = P.OscarsConfig()
    dims = kw.pop("dims", [32, 32, 3, 64, 10])
    arr = (ctypes.c_int32 * len(dims))(*dims)
    cfg.dims = arr
    cfg.num_workers = kw.pop("W", 2)
    cfg.model = P.MODEL_CNN
    cfg.num_layers = kw.pop("blocks", 1)
    cfg.batch = kw.pop("batch", 16)
    cfg.lr = 0.05
    cfg.server_lr = 1.0
    cfg.bf16_gemm = kw.pop("bf16", 1)
    cfg.M = 4
    t = (ctypes.c_int64 * 2)(3, 5)
    cfg.t_ticks = t
    return cfg, (arr, t)


@pytest.mark.parametrize("change, status", [
    (dict(dims=[28, 28, 1, 64, 10]), P.OSCARS_ENOTSUP),    # image size
    (dict(dims=[32, 32, 3, 32, 10]), P.OSCARS_ENOTSUP),    # channels
    (dict(dims=[32, 32, 65, 64, 10]), P.OSCARS_ENOTSUP),   # input channels
    (dict(dims=[32, 32, 3, 64, 40]), P.OSCARS_ENOTSUP),    # classes
    (dict(blocks=0), P.OSCARS_ENOTSUP),
    (dict(blocks=5), P.OSCARS_ENOTSUP),
    (dict(batch=24), P.OSCARS_ENOTSUP),                     # not a multiple of 16
    (dict(bf16=0), P.OSCARS_ENOTSUP),
    (dict(dims=[32, 32, 0, 64, 10]), P.OSCARS_EINVAL),
    (dict(), P.OSCARS_EINVAL),                              # valid shape but NULL shards
])
def test_cnn_create_rejects_before_device_work(oscars_lib, change, status):
    cfg, keep = _cnn_cfg(**change)
    h = ctypes.c_void_p()
    assert oscars_lib.oscars_create(ctypes.byref(cfg), ctypes.byref(h)) == status
    assert h.value is None
