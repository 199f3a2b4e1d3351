"""Pins of the seeded input generator (agn_inputs)."""

import math

import numpy as np
import pytest

import agn_inputs as I
from agn_inputs import workloads as WL


def test_splitmix64_published_outputs():
    # First outputs of splitmix64 seeded with 0 (the generator's reference
    # implementation, splitmix64.c by S. Vigna, public domain).
    d = I.draw(0, np.arange(3))
    assert [int(v) for v in d] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_stream_keys_differ_and_draws_are_counter_based():
    keys = {I.stream_key(I.DEFAULT_SEED, s) for s in range(1, 8)}
    assert len(keys) == 7
    k = I.stream_key(123, 1)
    a = I.draw(k, np.arange(1000))
    b = I.draw(k, np.arange(500, 1000))
    assert np.array_equal(a[500:], b)


def test_series_log_and_cos_match_libm():
    x = np.concatenate([np.linspace(0, 1, 20001)[1:], np.logspace(-300, 0, 4001)])
    ln = I.ln_series(x)
    ref = np.log(x)
    assert np.max(np.abs(ln - ref) / np.maximum(1.0, np.abs(ref))) < 1e-15
    t = np.linspace(0, 1, 20001)[:-1]
    assert np.max(np.abs(I.cos2pi_series(t) - np.cos(2 * np.pi * t))) < 2e-15
    assert I.ln_series(np.array([1.0]))[0] == 0.0


def test_uniform_and_normal_variates():
    k = I.stream_key(7, 1)
    u = I.uniform_f32(k, np.arange(200000))
    assert u.dtype == np.float32 and u.min() >= 0 and u.max() < 1
    # exactly representable multiples of 2^-24
    assert np.all((u.astype(np.float64) * 2 ** 24) % 1 == 0)
    assert abs(u.mean() - 0.5) < 0.005
    z = I.normal_f64(k, np.arange(400000))
    assert abs(z.mean()) < 0.01 and abs(z.var() - 1) < 0.01
    # tail mass beyond 3 sigma ~ 0.27 %
    assert 0.0018 < np.mean(np.abs(z) > 3) < 0.0036
    scipy_stats = pytest.importorskip("scipy.stats")
    assert scipy_stats.kstest(z, "norm").pvalue > 1e-4


def test_init_params_glorot_bounds_and_zero_biases():
    dims = (784, 128, 10)
    th = I.init_params(I.DEFAULT_SEED, dims)
    assert th.dtype == np.float32 and th.size == I.num_params(dims) == 101770
    for l, (ow, ob) in enumerate(I.layer_offsets(dims), start=1):
        r = math.sqrt(6.0 / (dims[l - 1] + dims[l]))
        W = th[ow:ob]
        assert np.max(np.abs(W)) <= r and np.max(np.abs(W)) > 0.99 * r
        assert abs(np.var(W.astype(np.float64)) - r * r / 3) < 0.05 * r * r
        assert np.all(th[ob:ob + dims[l]] == 0)


@pytest.mark.parametrize("w", [WL.SMALL, WL.MNIST_SHAPED, WL.WIDE_BF16, WL.LARGE_BF16],
                         ids=lambda w: w.name)
def test_teacher_labels_are_balanced(w):
    ds = I.workload_dataset(w)
    rows = np.arange(0, w.n_samples, max(1, w.n_samples // 3000))
    X = I.make_inputs_x(I.DEFAULT_SEED, w.dims[0], rows, w.dist)
    y = I.teacher_labels(X, ds.teacher, w.dist)
    frac = np.bincount(y, minlength=10) / len(y)
    assert frac.min() >= 0.01, frac


def test_dataset_rows_match_direct_generation():
    w = WL.SMALL
    ds = I.workload_dataset(w)
    rows = np.array([5, 700, 511, 512, 2047])
    X, y = ds(rows[:3])
    assert np.array_equal(X, I.make_inputs_x(I.DEFAULT_SEED, 784, rows[:3], w.dist))
    Xw, yw = ds(rows)          # rows spanning shards
    assert np.array_equal(Xw[:3], X) and np.array_equal(yw[:3], y)


def test_round_robin_schedule_properties():
    n, C = 8, 200
    w, tau = I.make_schedule(n, C, n - 1, n - 1, 5)
    assert np.array_equal(w, np.arange(C) % n)
    # Fig. 1: a homogeneous cluster gives staleness n-1 once every worker has committed
    assert np.all(tau[n - 1:] == n - 1)
    assert np.array_equal(tau[: n - 1], np.arange(n - 1))
    w, tau = I.make_schedule(16, 2000, 0, 15, I.DEFAULT_SEED)
    assert tau.min() == 0 and tau.max() == 15
    prev = np.full(16, -1)
    for c in range(2000):
        assert prev[w[c]] < c - tau[c] <= c
        prev[w[c]] = c


def test_commit_bench_order_and_pulls():
    order, pulls = I.commit_bench_order(I.DEFAULT_SEED, 64, 4)
    assert sorted(order.tolist()) == list(range(64))
    assert pulls.shape == (64, 4)
    for row in pulls:
        assert len(set(row.tolist())) == 4 and row.min() >= 0 and row.max() < 64
    a = I.commit_bench_acc(I.DEFAULT_SEED, 1 << 16, 3)
    assert abs(a.std() - 0.1) < 0.003
    t = I.commit_bench_theta(I.DEFAULT_SEED, 1 << 16, idx=np.array([0, 5, 65535]))
    assert np.array_equal(t, I.commit_bench_theta(I.DEFAULT_SEED, 1 << 16)[[0, 5, 65535]])
