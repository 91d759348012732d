"""The seeded input generators: numpy and torch agree bit for bit, and the
draws have the intended ranges and moments."""
import numpy as np
import torch

import synth


def test_numpy_torch_identical():
    idx = np.arange(0, 200_000, 7, dtype=np.uint64)
    for stream in (1, (synth.S_NOISE << 16) | 5):
        a = synth.gauss_np(3, stream, idx, 1e-3)
        b = synth.gauss_t(3, stream, torch.from_numpy(idx.astype(np.int64)), 1e-3).numpy()
        np.testing.assert_array_equal(a, b)
        a = synth.uniform_np(3, stream, idx)
        b = synth.uniform_t(3, stream, torch.from_numpy(idx.astype(np.int64))).numpy()
        np.testing.assert_array_equal(a, b)
        a = synth.label_np(3, stream, idx)
        b = synth.label_t(3, stream, torch.from_numpy(idx.astype(np.int64))).numpy()
        np.testing.assert_array_equal(a, b)


def test_shards_numpy_torch_identical():
    w = synth.CFG3
    Xn, yn = synth.shard_np(w, 2, n=64)
    Xt, yt = synth.shard_t(w, 2, "cpu", n=64)
    np.testing.assert_array_equal(Xn, Xt.numpy())
    np.testing.assert_array_equal(yn, yt.numpy())
    assert Xn.min() >= -3 and Xn.max() <= 3
    En, _ = synth.eval_np(w, n=16)
    Et, _ = synth.eval_t(w, "cpu", n=16)
    np.testing.assert_array_equal(En, Et.numpy())


def test_merge_inputs_numpy_torch_identical():
    m = synth.CFG4
    idx = np.arange(1000, 3000, dtype=np.uint64)
    np.testing.assert_array_equal(synth.merge_xg_np(m, idx), synth.merge_xg_t(m, 1000, 2000, "cpu").numpy())
    np.testing.assert_array_equal(synth.merge_delta_np(m, 9, idx), synth.merge_delta_t(m, 9, 1000, 2000, "cpu").numpy())


def test_moments():
    g = synth.gauss_np(0, 77, np.arange(400_000, dtype=np.uint64), 2.0)
    assert abs(g.mean()) < 0.02 and abs(g.std() - 2.0) < 0.02
    u = synth.uniform_np(0, 78, np.arange(100_000, dtype=np.uint64))
    assert u.min() >= 0 and u.max() < 1 and abs(u.mean() - 0.5) < 0.01
    y = synth.label_np(0, 79, np.arange(100_000, dtype=np.uint64))
    assert set(np.unique(y).tolist()) == set(range(10))


def test_workload_sizes():
    assert synth.CFG1.num_params == 7850
    assert synth.CFG2.num_params == 407_050
    assert synth.CFG3.num_params == 4_206_602
    layers = synth.init_layers_np(synth.CFG2)
    assert [W.shape for W, _ in layers] == [(512, 784), (10, 512)]
    assert np.abs(layers[0][0]).max() <= 1 / np.sqrt(784)
    s = synth.speeds(synth.CFG2)
    assert s.shape == (16,) and np.all(s > 0)


def test_drifting_speeds():
    import synth
    w = synth.CFG2
    s = synth.drifting_speeds(w, 6, sigma=0.3)
    assert s.shape == (6, w.num_workers)
    np.testing.assert_array_equal(s[0], synth.speeds(w))
    assert np.all(s > 0)
    np.testing.assert_array_equal(s, synth.drifting_speeds(w, 6, sigma=0.3))   # seeded
    r = np.log(s[1:] / s[:-1])
    assert 0.15 < r.std() < 0.45
