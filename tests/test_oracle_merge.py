"""Pins for the oracle merge (Eq. 4, first branch): hand sums, the W=1 and
identical-delta special cases, and equality of the delta form with the
printed average (1/N) sum_k x^k."""
import numpy as np

from oracle import merge


def test_hand_sums():
    x_g = np.array([1.0, 2.0, 3.0, -4.0], np.float32)
    d = [np.array([1.0, 0.0, 0.0, 2.0], np.float32), np.array([0.0, 2.0, -4.0, 2.0], np.float32)]
    out = merge.merge_deltas(x_g, d, [0.5, 0.25])
    # 1 + 0.5*1 ; 2 + 0.25*2 ; 3 + 0.25*(-4) ; -4 + 0.5*2 + 0.25*2
    assert out.tolist() == [1.5, 2.5, 2.0, -2.5]
    out = merge.merge_deltas(x_g, d, [0.5, 0.25], server_lr=2.0)
    assert out.tolist() == [2.0, 3.0, 1.0, -1.0]


def test_single_worker_weight_one_is_the_worker_model():
    rng = np.random.default_rng(0)
    x_g = rng.standard_normal(1000).astype(np.float32)
    x1 = rng.standard_normal(1000).astype(np.float32)
    np.testing.assert_array_equal(merge.merge_models(x_g, [x1], [1.0]), x1)


def test_identical_deltas():
    rng = np.random.default_rng(1)
    x_g = rng.standard_normal(500).astype(np.float32)
    d = (rng.standard_normal(500) * 1e-3).astype(np.float32)
    w = np.array([0.125, 0.375, 0.5], np.float32)
    out = merge.merge_deltas(x_g, [d, d, d], w)
    np.testing.assert_array_equal(out, (x_g.astype(np.float64) + d.astype(np.float64)).astype(np.float32))


def test_delta_form_equals_eq4_average():
    rng = np.random.default_rng(2)
    for W in (1, 2, 3, 7, 16):
        x_g = rng.standard_normal(4096).astype(np.float32)
        models = [(x_g + rng.standard_normal(4096).astype(np.float32) * 0.01).astype(np.float32) for _ in range(W)]
        a = merge.merge_models(x_g, models, np.full(W, np.float32(1.0 / W)))
        b = merge.average(models)
        ulp = np.spacing(np.abs(b).astype(np.float32))
        # w = fp32(1/W) differs from 1/W by < 2^-24 relative, an error on the
        # delta sum that is relative to |x_g| + |b| (cancellation can make b tiny)
        bound = 2 * ulp + 1.2e-7 * (np.abs(x_g) + np.abs(b))
        assert np.all(np.abs(a.astype(np.float64) - b) <= bound)


def test_order_of_workers_is_summation_order():
    x_g = np.zeros(1, np.float32)
    d = [np.array([1e8], np.float32), np.array([1.0], np.float32), np.array([-1e8], np.float32)]
    out = merge.merge_deltas(x_g, d, [1.0, 1.0, 1.0])
    assert out.tolist() == [1.0]           # fp64 accumulation keeps the small term
