"""Python binding of liboscars (the C ABI in include/oscars.h).

Argument marshalling only: every step of the hot path runs in the CUDA
library.  The functions below keep the C names; ``OscarsContext`` is a small
convenience wrapper over them for torch tensors.  There is no fallback: if
the shared library is missing, loading raises.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int32, c_int64, c_void_p
from typing import Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_lib", "liboscars.so")

OSCARS_OK, OSCARS_EINVAL, OSCARS_ENOMEM, OSCARS_ECUDA, OSCARS_ESTATE, OSCARS_ETIMEOUT, OSCARS_ENOTSUP = range(7)
MODEL_FLAT, MODEL_MLP, MODEL_CNN = 0, 1, 2
W_UNIFORM, W_LOCALSTEPS, W_EXPLICIT = 0, 1, 2
SEARCH_CAPPED, SEARCH_LITERAL = 0, 1
POLICY_OSCARS, POLICY_BSP, POLICY_LOCAL_SGD = 0, 1, 2
FLAG_NO_GRAPH = 1
FLAG_PROFILE = 2
FLAG_BRANCHES = 4
FLAG_PER_LAYER = 8
FLAG_PHASE_TIMES = 16


class OscarsError(RuntimeError):
    def __init__(self, status: int, msg: str = ""):
        self.status = status
        super().__init__(f"{_status_name(status)}: {msg}")


class OscarsConfig(ctypes.Structure):
    _fields_ = [
        ("num_workers", c_int32), ("model", c_int32), ("num_layers", c_int32), ("dims", POINTER(c_int32)),
        ("batch", c_int32), ("lr", c_float), ("server_lr", c_float), ("weight_rule", c_int32),
        ("bf16_gemm", c_int32), ("speed", POINTER(c_double)), ("t_ticks", POINTER(c_int64)),
        ("ticks_per_unit", c_int64), ("M", c_int64), ("search_mode", c_int32),
        ("shard_x", POINTER(c_void_p)), ("shard_y", POINTER(c_void_p)), ("shard_n", POINTER(c_int64)),
        ("init_params", c_void_p), ("cuda_stream", c_void_p), ("flags", c_int32),
    ]


class OscarsRoundLog(ctypes.Structure):
    _fields_ = [("ticks", c_int64), ("barrier", c_int64), ("eval_loss", c_float), ("worker_loss", c_float)]


_lib = None

_SIGS = {
    "oscars_create": (c_int32, [POINTER(OscarsConfig), POINTER(c_void_p)]),
    "oscars_destroy": (c_int32, [c_void_p]),
    "oscars_local_steps": (c_int32, [c_void_p, POINTER(c_int32), POINTER(c_float)]),
    "oscars_losses_async": (c_int32, [c_void_p, c_void_p]),
    "oscars_push_merge": (c_int32, [c_void_p, POINTER(c_void_p), POINTER(c_float)]),
    "oscars_pull": (c_int32, [c_void_p, c_void_p]),
    "oscars_get_schedule": (c_int32, [c_void_p, POINTER(c_int64), POINTER(c_int64), POINTER(c_int64),
                                      POINTER(c_int32), POINTER(c_int64), POINTER(c_int64), POINTER(c_int64)]),
    "oscars_set_local_steps": (c_int32, [c_void_p, POINTER(c_int32)]),
    "oscars_set_iteration_ticks": (c_int32, [c_void_p, POINTER(c_int64)]),
    "oscars_eval_loss": (c_int32, [c_void_p, c_void_p, c_void_p, c_int64, POINTER(c_float)]),
    "oscars_num_params": (c_int32, [c_void_p, POINTER(c_int64)]),
    "oscars_last_error": (ctypes.c_char_p, [c_void_p]),
    "oscars_status_string": (ctypes.c_char_p, [c_int32]),
    "oscars_iteration_ticks": (c_int32, [POINTER(c_double), c_int32, c_int64, POINTER(c_int64)]),
    "oscars_schedule_solve": (c_int32, [POINTER(c_int64), c_int32, c_int64, c_int32, POINTER(c_int64),
                                        POINTER(c_int64), POINTER(c_int32)]),
    "oscars_merge_weights": (c_int32, [c_int32, POINTER(c_int32), c_int32, POINTER(c_float)]),
    "oscars_read_replica": (c_int32, [c_void_p, c_int32, c_void_p]),
    "oscars_check_wait_timeout": (c_int32, [c_void_p, c_int32]),
    "oscars_check_padding": (c_int32, [c_void_p, POINTER(c_int64)]),
    "oscars_debug_slab": (c_int32, [c_void_p, POINTER(c_void_p), POINTER(c_int64)]),
    "oscars_gemm_bf16_nt": (c_int32, [c_void_p, c_void_p, c_void_p, c_int32, c_int32, c_int32, c_void_p]),
    "oscars_profile_read": (c_int32, [c_void_p, c_int32, POINTER(ctypes.c_char_p), POINTER(c_double),
                                      POINTER(c_int32)]),
    "oscars_profile_reset": (c_int32, [c_void_p]),
    "oscars_phase_times": (c_int32, [c_void_p, c_int32, POINTER(c_double)]),
    "oscars_softreg_steps_noalloc": (c_int32, [c_void_p, c_void_p, c_void_p, c_void_p, c_int64, c_int64, c_int32,
                                               c_int32, c_int32, c_int32, c_float, c_void_p, c_void_p]),
    "oscars_policy_local_steps": (c_int32, [c_int32, POINTER(c_int64), c_int32, c_int64, c_int32, c_int32,
                                            POINTER(c_int32), POINTER(c_int64)]),
    "oscars_partition_sizes": (c_int32, [POINTER(c_int64), c_int32, c_int64, c_int64, POINTER(c_int64)]),
    "oscars_round_clusters": (c_int32, [POINTER(c_int32), c_int32, c_int32, POINTER(c_int32), POINTER(c_int32),
                                        POINTER(c_int32)]),
    "oscars_train": (c_int32, [c_void_p, c_int32, c_void_p, c_void_p, c_int64, c_float, POINTER(OscarsRoundLog),
                               POINTER(c_int32)]),
    "oscars_merge": (c_int32, [c_void_p, POINTER(c_void_p), POINTER(c_float), c_int32, c_int64, c_float, c_void_p]),
}


def lib():
    """Load liboscars.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"liboscars.so is not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _status_name(s: int) -> str:
    try:
        return lib().oscars_status_string(s).decode()
    except Exception:
        return f"status {s}"


def _check(status: int, ctx=None):
    if status != OSCARS_OK:
        msg = lib().oscars_last_error(ctx).decode() if ctx else ""
        raise OscarsError(status, msg)


def _arr(ctype, values):
    values = list(values)
    return (ctype * len(values))(*values)


# ---------------------------------------------------------------- C names
def oscars_iteration_ticks(speed: Sequence[float], ticks_per_unit: int = 1000):
    n = len(speed)
    out = (c_int64 * n)()
    _check(lib().oscars_iteration_ticks(_arr(c_double, speed), n, ticks_per_unit, out))
    return list(out)


def oscars_schedule_solve(t_iter: Sequence[int], M: int, search_mode: int = SEARCH_CAPPED):
    n = len(t_iter)
    T, mw, tau = c_int64(), c_int64(), (c_int32 * n)()
    _check(lib().oscars_schedule_solve(_arr(c_int64, t_iter), n, M, search_mode, ctypes.byref(T),
                                       ctypes.byref(mw), tau))
    return T.value, mw.value, list(tau)


def oscars_policy_local_steps(policy: int, t_iter: Sequence[int], M: int = 1, search_mode: int = SEARCH_CAPPED,
                              I: int = 1):
    """(tau, barrier) of one round under a synchronisation scheme."""
    n = len(t_iter)
    tau, B = (c_int32 * n)(), c_int64()
    _check(lib().oscars_policy_local_steps(policy, _arr(c_int64, t_iter), n, M, search_mode, I, tau,
                                           ctypes.byref(B)))
    return list(tau), B.value


def oscars_partition_sizes(weight: Sequence[int], total: int, unit: int = 1):
    n = len(weight)
    out = (c_int64 * n)()
    _check(lib().oscars_partition_sizes(_arr(c_int64, weight), n, total, unit, out))
    return list(out)


def oscars_round_clusters(tau: Sequence[int], max_clusters: int):
    """Worker lists of the one-launch round kernel: a list of workers per cluster."""
    n = len(tau)
    order, first, ncl = (c_int32 * n)(), (c_int32 * (n + 1))(), c_int32()
    _check(lib().oscars_round_clusters(_arr(c_int32, tau), n, max_clusters, order, first, ctypes.byref(ncl)))
    return [list(order[first[k]:first[k + 1]]) for k in range(ncl.value)]


def oscars_train(ctx: int, rounds: int, eval_x_ptr: Optional[int] = None, eval_y_ptr: Optional[int] = None,
                 eval_n: int = 0, target_loss: float = 0.0):
    """Rounds run natively; returns one dict per round run."""
    log, done = (OscarsRoundLog * rounds)(), c_int32()
    _check(lib().oscars_train(c_void_p(ctx), rounds, c_void_p(eval_x_ptr) if eval_x_ptr else None,
                              c_void_p(eval_y_ptr) if eval_y_ptr else None, eval_n, target_loss, log,
                              ctypes.byref(done)), c_void_p(ctx))
    return [{"ticks": log[r].ticks, "barrier": log[r].barrier, "eval_loss": log[r].eval_loss,
             "worker_loss": log[r].worker_loss} for r in range(done.value)]


def oscars_merge_weights(rule: int, tau: Sequence[int]):
    n = len(tau)
    w = (c_float * n)()
    _check(lib().oscars_merge_weights(rule, _arr(c_int32, tau), n, w))
    return list(w)


def oscars_merge(x_g_ptr: int, delta_ptrs: Sequence[int], w: Sequence[float], P: int, server_lr: float = 1.0,
                 stream: Optional[int] = None):
    W = len(delta_ptrs)
    _check(lib().oscars_merge(c_void_p(x_g_ptr), _arr(c_void_p, delta_ptrs), _arr(c_float, w), W, P,
                              server_lr, c_void_p(stream or 0)))


def oscars_softreg_steps_noalloc(params_in_ptr: int, params_out_ptr: int, x_ptr: int, y_ptr: int, n: int,
                                 cursor: int, tau: int, dim: int, classes: int, batch: int, lr: float,
                                 loss_out_ptr: int, stream: Optional[int] = None):
    _check(lib().oscars_softreg_steps_noalloc(c_void_p(params_in_ptr), c_void_p(params_out_ptr), c_void_p(x_ptr),
                                              c_void_p(y_ptr), n, cursor, tau, dim, classes, batch, lr,
                                              c_void_p(loss_out_ptr), c_void_p(stream or 0)))


def oscars_create(cfg: OscarsConfig) -> int:
    h = c_void_p()
    st = lib().oscars_create(ctypes.byref(cfg), ctypes.byref(h))
    if st != OSCARS_OK:
        raise OscarsError(st, "oscars_create")
    return h.value


def oscars_destroy(ctx: int):
    _check(lib().oscars_destroy(c_void_p(ctx)))


def oscars_local_steps(ctx: int, want_tau: bool = True, want_loss: bool = True):
    n = oscars_get_schedule(ctx)["W"]
    tau = (c_int32 * n)() if want_tau else None
    loss = (c_float * n)() if want_loss else None
    _check(lib().oscars_local_steps(c_void_p(ctx), tau, loss), c_void_p(ctx))
    return (list(tau) if tau is not None else None), (list(loss) if loss is not None else None)


def oscars_losses_async(ctx: int, dst_ptr: int):
    """Enqueue the copy of the last round's W losses into dst (no synchronisation)."""
    _check(lib().oscars_losses_async(c_void_p(ctx), c_void_p(dst_ptr)), c_void_p(ctx))


def oscars_push_merge(ctx: int, delta_ptrs: Optional[Sequence[int]] = None, weights: Optional[Sequence[float]] = None):
    d = _arr(c_void_p, delta_ptrs) if delta_ptrs is not None else None
    w = _arr(c_float, weights) if weights is not None else None
    _check(lib().oscars_push_merge(c_void_p(ctx), d, w), c_void_p(ctx))


def oscars_pull(ctx: int, dst_ptr: Optional[int] = None):
    _check(lib().oscars_pull(c_void_p(ctx), c_void_p(dst_ptr or 0) if dst_ptr else None), c_void_p(ctx))


_W_CACHE = {}


def oscars_get_schedule(ctx: int):
    W = _W_CACHE.get(ctx)
    if W is None:
        raise KeyError("unknown context")
    T, mw = c_int64(), c_int64()
    t, tau = (c_int64 * W)(), (c_int32 * W)()
    wait, clock, idle = (c_int64 * W)(), (c_int64 * W)(), (c_int64 * W)()
    _check(lib().oscars_get_schedule(c_void_p(ctx), ctypes.byref(T), ctypes.byref(mw), t, tau, wait, clock, idle))
    return {"W": W, "T_star": T.value, "max_wait": mw.value, "t_iter": list(t), "tau": list(tau),
            "wait": list(wait), "clock": list(clock), "idle": list(idle)}


def oscars_set_local_steps(ctx: int, tau: Sequence[int]):
    _check(lib().oscars_set_local_steps(c_void_p(ctx), _arr(c_int32, tau)), c_void_p(ctx))


def oscars_set_iteration_ticks(ctx: int, t_iter: Sequence[int]):
    _check(lib().oscars_set_iteration_ticks(c_void_p(ctx), _arr(c_int64, t_iter)), c_void_p(ctx))


def oscars_eval_loss(ctx: int, x_ptr: int, y_ptr: int, n: int) -> float:
    out = c_float()
    _check(lib().oscars_eval_loss(c_void_p(ctx), c_void_p(x_ptr), c_void_p(y_ptr), n, ctypes.byref(out)),
           c_void_p(ctx))
    return out.value


def oscars_read_replica(ctx: int, k: int, dst_ptr: int):
    _check(lib().oscars_read_replica(c_void_p(ctx), k, c_void_p(dst_ptr)), c_void_p(ctx))


def oscars_check_padding(ctx: int) -> int:
    """Padding values that are not zero plus changed guard words (0 when no
    kernel wrote outside its tensors)."""
    bad = c_int64()
    _check(lib().oscars_check_padding(c_void_p(ctx), ctypes.byref(bad)), c_void_p(ctx))
    return bad.value


def oscars_debug_slab(ctx: int):
    """(device address of the fp32 slab, slot stride in floats)."""
    p, st = c_void_p(), c_int64()
    _check(lib().oscars_debug_slab(c_void_p(ctx), ctypes.byref(p), ctypes.byref(st)))
    return p.value, st.value


def oscars_check_wait_timeout(ctx: int, polls: int):
    """Run the kernels' bounded-wait failure path once (raises OscarsError
    with OSCARS_ETIMEOUT when the path works)."""
    _check(lib().oscars_check_wait_timeout(c_void_p(ctx), polls), c_void_p(ctx))


def oscars_gemm_bf16_nt(a_ptr: int, b_ptr: int, c_ptr: int, M: int, N: int, K: int, stream: Optional[int] = None):
    _check(lib().oscars_gemm_bf16_nt(c_void_p(a_ptr), c_void_p(b_ptr), c_void_p(c_ptr), M, N, K,
                                     c_void_p(stream or 0)))


def oscars_profile_read(ctx: int):
    """{kernel class: (total ms, launches)} since the last reset."""
    cap = 64
    names, ms, cnt = (ctypes.c_char_p * cap)(), (c_double * cap)(), (c_int32 * cap)()
    n = lib().oscars_profile_read(c_void_p(ctx), cap, names, ms, cnt)
    if n < 0:
        raise OscarsError(OSCARS_EINVAL, "profile_read")
    return {names[i].decode(): (ms[i], cnt[i]) for i in range(min(n, cap))}


def oscars_phase_times(ctx: int):
    """[(forward, last layer, weight gradient) us per local step] of worker 0."""
    cap = 3 * 256
    buf = (c_double * cap)()
    n = lib().oscars_phase_times(c_void_p(ctx), cap, buf)
    if n < 0:
        raise OscarsError(OSCARS_ECUDA, "phase_times")
    return [tuple(buf[i:i + 3]) for i in range(0, n, 3)]


def oscars_profile_reset(ctx: int):
    _check(lib().oscars_profile_reset(c_void_p(ctx)))


def oscars_num_params(ctx: int) -> int:
    P = c_int64()
    _check(lib().oscars_num_params(c_void_p(ctx), ctypes.byref(P)))
    return P.value


# ---------------------------------------------------------------- convenience wrapper
class OscarsContext:
    """Owns one oscars_ctx; keeps the borrowed buffers alive.

    ``shards`` are (X, y) torch CUDA tensors (fp32 [n, d], int32 [n]);
    ``init_params`` a flat fp32 tensor (host or CUDA) in canonical layout.
    """

    def __init__(self, *, num_workers: int, dims: Sequence[int], model: int = MODEL_MLP, batch: int = 32,
                 lr: float = 0.05, server_lr: float = 1.0, weight_rule: int = W_UNIFORM, bf16: bool = True,
                 speed: Optional[Sequence[float]] = None, t_ticks: Optional[Sequence[int]] = None,
                 ticks_per_unit: int = 1000, M: int = 8, search_mode: int = SEARCH_CAPPED, shards=None,
                 init_params=None, stream: Optional[int] = None, flags: int = 0, blocks: int = 1):
        """dims: MLP [input, hidden..., classes]; CNN [H, W, Cin, C, classes]
        with ``blocks`` residual blocks; FLAT [P]."""
        W = num_workers
        self._keep = []
        cfg = OscarsConfig()
        cfg.num_workers = W
        cfg.model = model
        L = len(dims) - 1 if model == MODEL_MLP else (blocks if model == MODEL_CNN else 1)
        cfg.num_layers = L
        dims_arr = _arr(c_int32, dims)
        self._keep.append(dims_arr)
        cfg.dims = dims_arr
        cfg.batch = batch
        cfg.lr = lr
        cfg.server_lr = server_lr
        cfg.weight_rule = weight_rule
        cfg.bf16_gemm = 1 if bf16 else 0
        if speed is not None:
            sp = _arr(c_double, speed)
            self._keep.append(sp)
            cfg.speed = sp
        if t_ticks is not None:
            tt = _arr(c_int64, t_ticks)
            self._keep.append(tt)
            cfg.t_ticks = tt
        cfg.ticks_per_unit = ticks_per_unit
        cfg.M = M
        cfg.search_mode = search_mode
        if shards is not None:
            xs = _arr(c_void_p, [s[0].data_ptr() for s in shards])
            ys = _arr(c_void_p, [s[1].data_ptr() for s in shards])
            ns = _arr(c_int64, [s[0].shape[0] for s in shards])
            self._keep += [xs, ys, ns, shards]
            cfg.shard_x, cfg.shard_y, cfg.shard_n = xs, ys, ns
        if init_params is not None:
            self._keep.append(init_params)
            cfg.init_params = init_params.data_ptr()
        cfg.cuda_stream = stream or 0
        cfg.flags = flags
        self.W = W
        self.handle = oscars_create(cfg)
        _W_CACHE[self.handle] = W
        self.P = oscars_num_params(self.handle)

    def local_steps(self, want_loss: bool = True):
        return oscars_local_steps(self.handle, want_tau=True, want_loss=want_loss)

    def losses_async(self, dst):
        oscars_losses_async(self.handle, dst.data_ptr())

    def push_merge(self, deltas=None, weights=None):
        ptrs = [d.data_ptr() for d in deltas] if deltas is not None else None
        oscars_push_merge(self.handle, ptrs, weights)

    def pull(self, dst=None):
        oscars_pull(self.handle, dst.data_ptr() if dst is not None else None)

    def profile(self):
        return oscars_profile_read(self.handle)

    def profile_reset(self):
        oscars_profile_reset(self.handle)

    def read_replica(self, k: int, dst):
        oscars_read_replica(self.handle, k, dst.data_ptr())

    def schedule(self):
        return oscars_get_schedule(self.handle)

    def set_local_steps(self, tau):
        oscars_set_local_steps(self.handle, tau)

    def set_iteration_ticks(self, t_iter):
        oscars_set_iteration_ticks(self.handle, t_iter)

    def eval_loss(self, x, y) -> float:
        return oscars_eval_loss(self.handle, x.data_ptr(), y.data_ptr(), x.shape[0])

    def train(self, rounds: int, eval_x=None, eval_y=None, target_loss: float = 0.0):
        if eval_x is None:
            return oscars_train(self.handle, rounds)
        return oscars_train(self.handle, rounds, eval_x.data_ptr(), eval_y.data_ptr(), eval_x.shape[0], target_loss)

    def close(self):
        if getattr(self, "handle", None):
            oscars_destroy(self.handle)
            _W_CACHE.pop(self.handle, None)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
