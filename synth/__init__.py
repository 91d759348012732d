"""Seeded synthetic inputs shared by the oracle, the tests and the bench.

This module only *draws inputs*.  It holds none of the method's arithmetic
(no scheduling, no SGD, no merge): the oracle and the CUDA library both take
what is generated here as plain arrays.

Every random value is a pure function of ``(seed, stream, counter)`` so that
any element can be regenerated anywhere, bit for bit:

* ``lowbias32`` is the 32-bit integer hash published by C. Wellons
  ("hash prospector", constants 0x7feb352d / 0x846ca68b).
* a uniform in [0, 1) is the top 24 bits of one hash times 2**-24 (exact in
  fp32);
* a standard "normal" is the Irwin-Hall sum of four such uniforms, centred
  and scaled to unit variance, ``((u0 + u1) + u2) + u3 - 2`` times
  ``sqrt(3)``.  Every step is a single fp32 operation in a fixed order, so the
  numpy (host) and torch (host or device) versions below agree exactly.

The numpy and torch versions are written side by side; ``tests`` check that
they agree bit for bit.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Tuple

import numpy as np

M32 = 0xFFFFFFFF
NUM_CLASSES = 10

# stream identifiers (the high part of the stream word; the low 16 bits carry
# the worker index where there is one)
S_LABEL = 1
S_NOISE = 2
S_MEAN = 3
S_INIT = 4
S_EVAL_LABEL = 5
S_EVAL_NOISE = 6
S_MERGE_XG = 7
S_MERGE_DELTA = 8

# sub-seed offsets: data = seed, speeds = seed+1, init = seed+2, eval = seed+3
SEED_SPEED = 1
SEED_INIT = 2
SEED_EVAL = 3
SEED_DRIFT = 4


# --------------------------------------------------------------------------
# counter-based generator, numpy
# --------------------------------------------------------------------------
def _lowbias32_np(x: np.ndarray) -> np.ndarray:
    x = np.asarray(x, dtype=np.uint64) & M32
    x ^= x >> np.uint64(16)
    x = (x * np.uint64(0x7FEB352D)) & M32
    x ^= x >> np.uint64(15)
    x = (x * np.uint64(0x846CA68B)) & M32
    x ^= x >> np.uint64(16)
    return x


def stream_key(seed: int, stream: int) -> int:
    """32-bit key of one (seed, stream) pair."""
    k = int(_lowbias32_np(np.array([seed & M32], dtype=np.uint64))[0])
    return int(_lowbias32_np(np.array([k ^ (stream & M32)], dtype=np.uint64))[0])


def bits_np(seed: int, stream: int, ctr: np.ndarray) -> np.ndarray:
    ctr = np.asarray(ctr, dtype=np.uint64)
    assert ctr.size == 0 or int(ctr.max()) <= M32
    return _lowbias32_np(ctr ^ np.uint64(stream_key(seed, stream)))


def uniform_np(seed: int, stream: int, ctr: np.ndarray) -> np.ndarray:
    """Uniform in [0, 1): 24 random bits, exact in fp32."""
    b = bits_np(seed, stream, ctr) >> np.uint64(8)
    return (b.astype(np.float32) * np.float32(2.0 ** -24)).astype(np.float32)


def gauss_np(seed: int, stream: int, idx: np.ndarray, sd: float) -> np.ndarray:
    """Approximately N(0, sd^2): scaled Irwin-Hall(4) of counter uniforms."""
    idx = np.asarray(idx, dtype=np.uint64)
    assert idx.size == 0 or int(idx.max()) < (1 << 30)
    base = idx * np.uint64(4)
    s = uniform_np(seed, stream, base)
    s = s + uniform_np(seed, stream, base + np.uint64(1))
    s = s + uniform_np(seed, stream, base + np.uint64(2))
    s = s + uniform_np(seed, stream, base + np.uint64(3))
    c = np.float32(sd * math.sqrt(3.0))
    return ((s - np.float32(2.0)) * c).astype(np.float32)


def label_np(seed: int, stream: int, idx: np.ndarray) -> np.ndarray:
    return (bits_np(seed, stream, idx) % np.uint64(NUM_CLASSES)).astype(np.int32)


# --------------------------------------------------------------------------
# counter-based generator, torch (same bits; int64 tensors hold 32-bit words)
# --------------------------------------------------------------------------
def _mul32_t(x, c: int):
    lo = x & 0xFFFF
    hi = x >> 16
    return (lo * c + (((hi * c) & 0xFFFF) << 16)) & M32


def _lowbias32_t(x):
    x = x & M32
    x = x ^ (x >> 16)
    x = _mul32_t(x, 0x7FEB352D)
    x = x ^ (x >> 15)
    x = _mul32_t(x, 0x846CA68B)
    x = x ^ (x >> 16)
    return x


def uniform_t(seed: int, stream: int, ctr):
    import torch
    b = _lowbias32_t(ctr ^ stream_key(seed, stream)) >> 8
    return b.to(torch.float32) * (2.0 ** -24)


def gauss_t(seed: int, stream: int, idx, sd: float):
    import torch
    base = idx * 4
    s = uniform_t(seed, stream, base)
    s = s + uniform_t(seed, stream, base + 1)
    s = s + uniform_t(seed, stream, base + 2)
    s = s + uniform_t(seed, stream, base + 3)
    c = float(np.float32(sd * math.sqrt(3.0)))
    return (s - 2.0) * torch.tensor(c, dtype=torch.float32, device=s.device)


def label_t(seed: int, stream: int, idx):
    import torch
    return (_lowbias32_t(idx ^ stream_key(seed, stream)) % NUM_CLASSES).to(torch.int32)


# --------------------------------------------------------------------------
# workloads
# --------------------------------------------------------------------------
@dataclass
class TrainWorkload:
    """A local-SGD training workload (W workers, MLP or softmax regression)."""
    name: str
    num_workers: int
    dims: List[int]            # input, hidden..., classes
    batch: int
    lr: float
    samples_per_worker: int
    M: int
    rounds: int
    seed: int = 0
    speeds: Optional[List[float]] = None   # fixed speeds; None = lognormal(0, 0.5)
    clip: Optional[float] = None
    bf16: bool = True
    server_lr: float = 1.0
    eval_n: int = 8192
    ticks_per_unit: int = 1000

    @property
    def num_params(self) -> int:
        return sum(o * i + o for i, o in zip(self.dims[:-1], self.dims[1:]))

    def flops_per_sample(self) -> float:
        """Forward + backward multiply-adds x2 of the linear layers."""
        f = 0
        for l, (i, o) in enumerate(zip(self.dims[:-1], self.dims[1:])):
            f += 2 * i * o          # forward
            f += 2 * i * o          # weight gradient
            if l > 0:
                f += 2 * i * o      # input gradient
        return float(f)


@dataclass
class ConvWorkload(TrainWorkload):
    """A local-SGD workload with the convolutional worker: CIFAR-shaped
    images (height x width x in_ch, NHWC, flattened as the data vector),
    a stem, ``blocks`` residual blocks of ``ch`` channels, pooling and a
    linear head.  ``dims`` is [height * width * in_ch, classes] (the data
    generator's view)."""
    height: int = 32
    width: int = 32
    in_ch: int = 3
    ch: int = 64
    blocks: int = 1

    @property
    def cnn_dims(self) -> List[int]:
        return [self.height, self.width, self.in_ch, self.ch, self.dims[-1]]

    @property
    def num_params(self) -> int:
        C, K = self.ch, self.dims[-1]
        return C * 9 * self.in_ch + C + self.blocks * 2 * (C * 9 * C + C) + K * C + K

    def flops_per_sample(self) -> float:
        """Multiply-adds x2 of the convolutions (forward, weight gradient, and
        the input gradient of the block convolutions) and the head."""
        hw, C, K = self.height * self.width, self.ch, self.dims[-1]
        stem = 2 * hw * C * 9 * self.in_ch
        block = 2 * hw * C * 9 * C
        return float(2 * stem + self.blocks * 2 * 3 * block + 3 * 2 * C * K)


@dataclass
class MergeWorkload:
    """A server-merge microbench: W pushed deltas of P fp32 parameters."""
    name: str
    num_workers: int
    num_params: int
    delta_sd: float
    tau_max: int
    weight_rule: str          # "uniform" or "localsteps"
    seed: int = 0
    server_lr: float = 1.0


CFG1 = TrainWorkload("softmax-reg-784x10-W4", 4, [784, 10], 32, 0.05, 4096, 8, 20,
                     speeds=[1.0, 1.0, 2.0, 4.0], bf16=False)
CFG2 = TrainWorkload("mlp-784-512-10-W16", 16, [784, 512, 10], 64, 0.05, 16384, 16, 100)
CFG3 = TrainWorkload("mlp-3072-1024-1024-10-W32", 32, [3072, 1024, 1024, 10], 128, 0.05,
                     8192, 16, 50, clip=3.0)
CFG4 = MergeWorkload("merge-P25.6M-W64", 64, 25_600_000, 1e-3, 8, "localsteps")
CFG5 = MergeWorkload("merge-P340M-W8", 8, 340_000_000, 1e-3, 16, "uniform")

CFG6 = ConvWorkload("resnet-mini-c64-W16", 16, [32 * 32 * 3, 10], 32, 0.05, 2048, 16, 20, clip=3.0)

WORKLOADS = {"cfg1": CFG1, "cfg2": CFG2, "cfg3": CFG3, "cfg4": CFG4, "cfg5": CFG5, "cfg6": CFG6}


def speeds(w: TrainWorkload) -> np.ndarray:
    """Per-worker speed factors s_i (larger = faster), fp64."""
    if w.speeds is not None:
        return np.asarray(w.speeds, dtype=np.float64)
    rng = np.random.default_rng(w.seed + SEED_SPEED)
    return rng.lognormal(0.0, 0.5, w.num_workers).astype(np.float64)


def drifting_speeds(w: TrainWorkload, rounds: int, sigma: float = 0.3) -> np.ndarray:
    """[rounds][W] speed factors of a volatile cluster: round 0 has the
    workload's speeds, then each worker's log-speed takes a Gaussian step of
    sd ``sigma`` per round (seeded)."""
    rng = np.random.default_rng(w.seed + SEED_DRIFT)
    steps = rng.standard_normal((rounds, w.num_workers)) * sigma
    steps[0] = 0.0
    return speeds(w)[None, :] * np.exp(np.cumsum(steps, axis=0))


def class_means_np(seed: int, d: int) -> np.ndarray:
    idx = np.arange(NUM_CLASSES * d, dtype=np.uint64)
    return gauss_np(seed, S_MEAN << 16, idx, 1.0).reshape(NUM_CLASSES, d)


def _samples_np(seed, label_stream, noise_stream, n, d, clip, means):
    y = label_np(seed, label_stream, np.arange(n, dtype=np.uint64))
    noise = gauss_np(seed, noise_stream, np.arange(n * d, dtype=np.uint64), 1.0).reshape(n, d)
    x = (means[y] + noise).astype(np.float32)
    if clip is not None:
        x = np.clip(x, np.float32(-clip), np.float32(clip)).astype(np.float32)
    return x, y


def shard_np(w: TrainWorkload, worker: int, n: Optional[int] = None) -> Tuple[np.ndarray, np.ndarray]:
    """Worker ``worker``'s training shard: X [n, d] fp32, y [n] int32."""
    n = w.samples_per_worker if n is None else n
    d = w.dims[0]
    means = class_means_np(w.seed, d)
    return _samples_np(w.seed, (S_LABEL << 16) | worker, (S_NOISE << 16) | worker, n, d, w.clip, means)


def eval_np(w: TrainWorkload, n: Optional[int] = None) -> Tuple[np.ndarray, np.ndarray]:
    n = w.eval_n if n is None else n
    d = w.dims[0]
    means = class_means_np(w.seed, d)
    return _samples_np(w.seed + SEED_EVAL, S_EVAL_LABEL << 16, S_EVAL_NOISE << 16, n, d, w.clip, means)


def init_layers_np(w: TrainWorkload) -> List[Tuple[np.ndarray, np.ndarray]]:
    """Initial model: W_l ~ U(-1/sqrt(fan_in), 1/sqrt(fan_in)), b_l = 0."""
    out = []
    for l, (i, o) in enumerate(zip(w.dims[:-1], w.dims[1:])):
        u = uniform_np(w.seed + SEED_INIT, (S_INIT << 16) | l, np.arange(o * i, dtype=np.uint64))
        a = np.float32(1.0 / math.sqrt(i))
        W = ((u * np.float32(2.0) - np.float32(1.0)) * a).astype(np.float32).reshape(o, i)
        out.append((W, np.zeros(o, dtype=np.float32)))
    return out


def init_cnn_np(w: "ConvWorkload") -> List[np.ndarray]:
    """Initial convolutional model in canonical order: weights
    U(-1/sqrt(fan_in), 1/sqrt(fan_in)) (fan_in = 9 Cin for a 3x3 convolution,
    C for the head), biases 0."""
    rng = np.random.default_rng(w.seed + SEED_INIT)
    C, K = w.ch, w.dims[-1]
    shapes = [(C, 3, 3, w.in_ch), (C,)]
    for _ in range(w.blocks):
        shapes += [(C, 3, 3, C), (C,), (C, 3, 3, C), (C,)]
    shapes += [(K, C), (K,)]
    out = []
    for s in shapes:
        if len(s) == 1:
            out.append(np.zeros(s, np.float32))
        else:
            fan_in = int(np.prod(s[1:]))
            lim = 1.0 / np.sqrt(fan_in)
            out.append(rng.uniform(-lim, lim, size=s).astype(np.float32))
    return out


def flatten_layers(layers) -> np.ndarray:
    """Canonical flat parameter vector: W_0, b_0, W_1, b_1, ... (fp32)."""
    return np.concatenate([np.concatenate([W.reshape(-1), b.reshape(-1)]) for W, b in layers]).astype(np.float32)


def unflatten_layers(flat: np.ndarray, dims: Sequence[int]):
    out, off = [], 0
    for i, o in zip(dims[:-1], dims[1:]):
        W = flat[off:off + o * i].reshape(o, i); off += o * i
        b = flat[off:off + o]; off += o
        out.append((W, b))
    return out


# ---- torch versions (device generation for full-size runs) ----
def class_means_t(seed: int, d: int, device):
    import torch
    idx = torch.arange(NUM_CLASSES * d, dtype=torch.int64, device=device)
    return gauss_t(seed, S_MEAN << 16, idx, 1.0).reshape(NUM_CLASSES, d)


def _samples_t(seed, label_stream, noise_stream, n, d, clip, means):
    import torch
    dev = means.device
    y = label_t(seed, label_stream, torch.arange(n, dtype=torch.int64, device=dev))
    noise = gauss_t(seed, noise_stream, torch.arange(n * d, dtype=torch.int64, device=dev), 1.0).reshape(n, d)
    x = means[y.long()] + noise
    if clip is not None:
        x = torch.clamp(x, -clip, clip)
    return x.contiguous(), y


def shard_t(w: TrainWorkload, worker: int, device, n: Optional[int] = None):
    n = w.samples_per_worker if n is None else n
    d = w.dims[0]
    means = class_means_t(w.seed, d, device)
    return _samples_t(w.seed, (S_LABEL << 16) | worker, (S_NOISE << 16) | worker, n, d, w.clip, means)


def eval_t(w: TrainWorkload, device, n: Optional[int] = None):
    n = w.eval_n if n is None else n
    d = w.dims[0]
    means = class_means_t(w.seed, d, device)
    return _samples_t(w.seed + SEED_EVAL, S_EVAL_LABEL << 16, S_EVAL_NOISE << 16, n, d, w.clip, means)


# ---- integer-valued inputs: fp32 sums of their products are exact ----
S_INT_X = 9
S_INT_W = 10


def shard_int_np(w: TrainWorkload, worker: int, n: int, vmax: int = 3):
    """Integer samples in [-vmax, vmax] (fp32) with uniform labels."""
    d = w.dims[0]
    b = bits_np(w.seed, (S_INT_X << 16) | worker, np.arange(n * d, dtype=np.uint64))
    x = ((b % np.uint64(2 * vmax + 1)).astype(np.int64) - vmax).astype(np.float32).reshape(n, d)
    y = label_np(w.seed, (S_LABEL << 16) | worker, np.arange(n, dtype=np.uint64))
    return x, y


def shard_int_t(w: TrainWorkload, worker: int, n: int, device, vmax: int = 3):
    import torch
    d = w.dims[0]
    idx = torch.arange(n * d, dtype=torch.int64, device=device)
    b = _lowbias32_t(idx ^ stream_key(w.seed, (S_INT_X << 16) | worker))
    x = ((b % (2 * vmax + 1)) - vmax).to(torch.float32).reshape(n, d)
    y = label_t(w.seed, (S_LABEL << 16) | worker, torch.arange(n, dtype=torch.int64, device=device))
    return x.contiguous(), y


def init_layers_int_np(w: TrainWorkload, wmax: int = 4, shift: int = 7):
    """Weights k * 2**-shift with integer k in [-wmax, wmax]; zero biases."""
    out = []
    for l, (i, o) in enumerate(zip(w.dims[:-1], w.dims[1:])):
        b = bits_np(w.seed + SEED_INIT, (S_INT_W << 16) | l, np.arange(o * i, dtype=np.uint64))
        k = (b % np.uint64(2 * wmax + 1)).astype(np.int64) - wmax
        out.append(((k.astype(np.float32) * np.float32(2.0 ** -shift)).reshape(o, i), np.zeros(o, np.float32)))
    return out


# ---- merge microbench inputs ----
def merge_taus(m: MergeWorkload) -> np.ndarray:
    """Random per-worker local-step counts in [1, tau_max] (int32)."""
    rng = np.random.default_rng(m.seed + SEED_SPEED)
    return rng.integers(1, m.tau_max + 1, m.num_workers).astype(np.int32)


def merge_xg_np(m: MergeWorkload, idx: np.ndarray) -> np.ndarray:
    """Initial global model at parameter indices ``idx``: U(-0.05, 0.05)."""
    u = uniform_np(m.seed + SEED_INIT, S_MERGE_XG << 16, np.asarray(idx, dtype=np.uint64))
    return ((u * np.float32(2.0) - np.float32(1.0)) * np.float32(0.05)).astype(np.float32)


def merge_delta_np(m: MergeWorkload, k: int, idx: np.ndarray) -> np.ndarray:
    """Worker k's pushed delta at parameter indices ``idx``."""
    return gauss_np(m.seed, (S_MERGE_DELTA << 16) | k, np.asarray(idx, dtype=np.uint64), m.delta_sd)


def merge_xg_t(m: MergeWorkload, start: int, count: int, device):
    import torch
    idx = torch.arange(start, start + count, dtype=torch.int64, device=device)
    u = uniform_t(m.seed + SEED_INIT, S_MERGE_XG << 16, idx)
    return (u * 2.0 - 1.0) * torch.tensor(np.float32(0.05).item(), dtype=torch.float32, device=device)


def merge_delta_t(m: MergeWorkload, k: int, start: int, count: int, device):
    import torch
    idx = torch.arange(start, start + count, dtype=torch.int64, device=device)
    return gauss_t(m.seed, (S_MERGE_DELTA << 16) | k, idx, m.delta_sd)
