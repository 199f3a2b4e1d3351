"""Pins of the CPU oracle against facts fixed outside it.

Each test ties one part of the oracle to the paper or to mathematics:
finite differences (the minibatch gradient of Eq. 1), the reduction to plain
SGD / DOWNPOUR (Section 2 footnote, Section 3), the commit identity
(Algorithm 1 + Eq. 1: the normalised accumulator is the mean of the local
updates), the closed form of the local iteration on linear least squares
(Section 3's lambda thought experiment, Eq. 3), hand-worked golden examples,
exact-rational float32 rounding of the commit (Eq. 1-2) and the FIFO
staleness semantics (Fig. 1).
"""

import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------
# helpers local to the tests (plain loops, independent of the oracle's loop)
# ----------------------------------------------------------------------------

def _tiny_problem(seed=0, dims=(5, 4, 3), m=3, margin=1e-3):
    """A tiny MLP problem whose pre-activations stay clear of the ReLU kink."""
    rng = np.random.default_rng(seed)
    mlp = O.MLP(dims)
    while True:
        theta = rng.normal(0, 0.7, mlp.num_params)
        X = rng.normal(0, 1, (m, dims[0]))
        y = rng.integers(0, dims[-1], m)
        h = X
        ok = True
        for l, (W, b) in enumerate(mlp.unpack(theta)):
            z = h @ W.T + b
            if l + 1 < len(dims) - 1:
                if np.min(np.abs(z)) < margin:
                    ok = False
                h = np.maximum(z, 0)
            else:
                h = z
        if ok:
            return mlp, theta, X, y


def _loss_only(mlp, theta, X, y):
    h = X
    params = mlp.unpack(theta)
    for l, (W, b) in enumerate(params):
        h = h @ W.T + b
        if l + 1 < len(params):
            h = np.maximum(h, 0)
    # brute-force log-sum-exp without max subtraction (values are small here)
    return float(np.mean([math.log(sum(math.exp(v) for v in row)) - row[t]
                          for row, t in zip(h, y)]))


class _ListData:
    """rows -> (X, y) from in-memory arrays."""

    def __init__(self, X, y):
        self.X, self.y = X, y

    def __call__(self, rows):
        return self.X[rows], self.y[rows]


# ----------------------------------------------------------------------------
# Minibatch gradient (Eq. 1 inner term)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("seed", [0, 1, 2])
def test_gradient_matches_central_differences(seed):
    mlp, theta, X, y = _tiny_problem(seed)
    loss, grad = mlp.loss_grad(theta, X, y)
    assert abs(loss - _loss_only(mlp, theta, X, y)) < 1e-12
    h = 1e-6
    fd = np.zeros_like(theta)
    for i in range(theta.size):
        e = np.zeros_like(theta)
        e[i] = h
        fd[i] = (_loss_only(mlp, theta + e, X, y) - _loss_only(mlp, theta - e, X, y)) / (2 * h)
    err = np.max(np.abs(fd - grad)) / max(1e-12, np.max(np.abs(grad)))
    assert err < 1e-6, err


def test_gradient_three_layers_central_differences():
    mlp, theta, X, y = _tiny_problem(7, dims=(6, 5, 4, 3), m=4)
    _, grad = mlp.loss_grad(theta, X, y)
    h = 1e-6
    fd = np.array([(_loss_only(mlp, theta + h * np.eye(theta.size)[i], X, y)
                    - _loss_only(mlp, theta - h * np.eye(theta.size)[i], X, y)) / (2 * h)
                   for i in range(theta.size)])
    assert np.max(np.abs(fd - grad)) / np.max(np.abs(grad)) < 1e-6


def test_softmax_xent_special_cases():
    # uniform logits: loss = ln C, gradient (1/C - onehot)/m
    C, m = 10, 4
    z = np.full((m, C), 3.25)
    y = np.array([0, 3, 9, 3])
    loss, dz = O.softmax_xent(z, y)
    assert abs(loss - math.log(C)) < 1e-15
    expect = np.full((m, C), 1.0 / C)
    expect[np.arange(m), y] -= 1.0
    assert np.allclose(dz, expect / m, atol=1e-17)
    # every row of the gradient sums to zero; huge logits stay finite
    z = np.array([[1000.0, 0.0, -1000.0], [0.0, 1e4, 5.0]])
    loss, dz = O.softmax_xent(z, np.array([0, 2]))
    assert np.isfinite(loss) and abs(loss - (0.0 + (1e4 - 5.0)) / 2) < 1e-9
    assert np.allclose(dz.sum(axis=1), 0.0, atol=1e-15)


def test_least_squares_gradient_central_differences():
    rng = np.random.default_rng(3)
    lsq = O.LeastSquares(4, 2)
    theta = rng.normal(size=lsq.num_params)
    X, Y = rng.normal(size=(5, 4)), rng.normal(size=(5, 2))
    _, g = lsq.loss_grad(theta, X, Y)
    h = 1e-6
    fd = np.array([(lsq.loss_grad(theta + h * e, X, Y)[0] - lsq.loss_grad(theta - h * e, X, Y)[0]) / (2 * h)
                   for e in np.eye(theta.size)])
    assert np.max(np.abs(fd - g)) < 1e-8


# ----------------------------------------------------------------------------
# Whole iterations
# ----------------------------------------------------------------------------

def _golden_rows():
    rows = []
    with open(os.path.join(GOLDEN, "agn_scalar_examples.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                lam, norm, nc, val = line.split()
                rows.append((int(lam), int(norm), int(nc), Fraction(val)))
    return rows


@pytest.mark.parametrize("lam,normalize,n_commits,expect", _golden_rows())
def test_hand_worked_scalar_examples(lam, normalize, n_commits, expect):
    lsq = O.LeastSquares(1, 1)
    data = _ListData(np.array([[1.0]]), np.array([[0.0]]))
    # the examples have no bias: a model over w alone, built from the
    # least-squares gradient with b pinned at 0
    class WOnly:
        num_params = 1

        def loss_grad(self, theta, X, Y):
            full = np.array([theta[0], 0.0])
            loss, g = lsq.loss_grad(full, X, Y)
            return loss, g[:1]
    r = O.agn_run(WOnly(), np.array([1.0]), 1, lam, 0.5, [0] * n_commits, [0] * n_commits,
                  data, 1, 1, normalize=bool(normalize))
    # exact when the rational is a dyadic number; otherwise within the two
    # roundings of the last division and addition
    assert abs(Fraction(float(r.theta[0])) - expect) <= Fraction(1, 2 ** 52)
    if expect.denominator & (expect.denominator - 1) == 0:
        assert Fraction(float(r.theta[0])) == expect


def test_n1_lambda1_is_plain_minibatch_sgd():
    """n = 1, lambda = 1 (DOWNPOUR without staleness) is textbook SGD."""
    rng = np.random.default_rng(11)
    dims, m, S = (7, 6, 4), 5, 20
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(S, dims[0])), rng.integers(0, dims[-1], S)
    theta0 = rng.normal(0, 0.3, mlp.num_params)
    eta, C = 0.1, 9
    r = O.agn_run(mlp, theta0, 1, 1, eta, [0] * C, [0] * C, _ListData(X, y), m, S)
    theta = theta0.copy()
    for t in range(C):
        rows = (t * m + np.arange(m)) % S
        _, g = mlp.loss_grad(theta, X[rows], y[rows])
        theta = theta - eta * g
    assert np.array_equal(theta, r.theta)


@pytest.mark.parametrize("lam", [2, 5, 8])
def test_commit_is_mean_of_local_updates(lam):
    """Algorithm 1: a/lambda = (theta_lambda - theta_0)/lambda, the mean local update."""
    rng = np.random.default_rng(lam)
    dims, m, S = (6, 5, 3), 4, 12
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(S, dims[0])), rng.integers(0, dims[-1], S)
    theta0 = rng.normal(0, 0.4, mlp.num_params)
    r = O.agn_run(mlp, theta0, 1, lam, 0.2, [0], [0], _ListData(X, y), m, S, keep_locals=[0])
    it = r.locals_[0]
    mean_update = np.mean([it[i + 1] - it[i] for i in range(lam)], axis=0)
    d = r.theta - theta0
    assert np.linalg.norm(d - mean_update) <= 1e-12 * np.linalg.norm(d)
    # the local iterates themselves follow theta_{i+1} = theta_i - eta grad(theta_i)
    for i in range(lam):
        rows = (i * m + np.arange(m)) % S
        _, g = mlp.loss_grad(it[i], X[rows], y[rows])
        assert np.allclose(it[i + 1], it[i] - 0.2 * g, rtol=0, atol=1e-15)


def _lsq_setup(seed=5, d_in=3, d_out=2, S=16):
    rng = np.random.default_rng(seed)
    X = rng.normal(size=(S, d_in))
    Y = rng.normal(size=(S, d_out))
    lsq = O.LeastSquares(d_in, d_out)
    theta0 = rng.normal(size=lsq.num_params)
    Xt = np.hstack([X, np.ones((S, 1))])
    A = Xt.T @ Xt / S
    B = Y.T @ Xt / S
    Theta0 = np.hstack([theta0[: d_out * d_in].reshape(d_out, d_in), theta0[d_out * d_in:, None]])
    Theta_star = np.linalg.solve(A.T, B.T).T
    return lsq, X, Y, theta0, A, Theta0, Theta_star


def _theta_to_flat(Th, d_in):
    return np.concatenate([Th[:, :d_in].ravel(), Th[:, d_in]])


@pytest.mark.parametrize("lam", [1, 3, 17, 60])
def test_least_squares_commit_closed_form(lam):
    """Full-shard batches: Delta = (Theta0 - Theta*)((I - eta A)^lambda - I)/lambda."""
    lsq, X, Y, theta0, A, Theta0, Theta_star = _lsq_setup()
    eta = 0.3
    S = X.shape[0]
    r = O.agn_run(lsq, theta0, 1, lam, eta, [0], [0], _ListData(X, Y), S, S)
    ev, Q = np.linalg.eigh(A)
    Mlam = Q @ np.diag((1 - eta * ev) ** lam) @ Q.T
    Delta = (Theta0 - Theta_star) @ (Mlam - np.eye(A.shape[0])) / lam
    expect = _theta_to_flat(Theta0 + Delta, X.shape[1])
    assert np.max(np.abs(r.theta - expect)) <= 1e-10 * max(1.0, np.max(np.abs(expect)))


def test_least_squares_large_lambda_points_at_minimum():
    """Eq. 3: as lambda grows the normalised delta shrinks like 1/lambda while
    lambda * Delta tends to Theta* - Theta0, a straight line to the minimum."""
    lsq, X, Y, theta0, A, Theta0, Theta_star = _lsq_setup()
    S = X.shape[0]
    target = _theta_to_flat(Theta_star - Theta0, X.shape[1])
    errs = []
    for lam in (50, 400):
        r = O.agn_run(lsq, theta0, 1, lam, 0.3, [0], [0], _ListData(X, Y), S, S)
        d = r.theta - theta0
        errs.append(np.linalg.norm(lam * d - target) / np.linalg.norm(target))
        assert np.linalg.norm(d) < 2 * np.linalg.norm(target) / lam
    assert errs[1] < 1e-8 and errs[1] <= errs[0]


def test_unnormalised_ablation_is_lambda_times_agn():
    rng = np.random.default_rng(2)
    dims, m, S, lam = (5, 4, 3), 3, 9, 6
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(S, dims[0])), rng.integers(0, dims[-1], S)
    theta0 = rng.normal(0, 0.4, mlp.num_params)
    d = _ListData(X, y)
    r1 = O.agn_run(mlp, theta0, 1, lam, 0.1, [0], [0], d, m, S, normalize=True)
    r0 = O.agn_run(mlp, theta0, 1, lam, 0.1, [0], [0], d, m, S, normalize=False)
    assert np.allclose(r0.theta - theta0, lam * (r1.theta - theta0), rtol=0, atol=1e-15)


# ----------------------------------------------------------------------------
# Staleness and data order (Fig. 1, Algorithm 1)
# ----------------------------------------------------------------------------

def _local_delta(mlp, theta_start, X, y, k, t0, lam, eta, m, S):
    theta = theta_start.copy()
    a = np.zeros_like(theta)
    for i in range(lam):
        rows = k * S + ((t0 + i) * m + np.arange(m)) % S
        _, g = mlp.loss_grad(theta, X[rows], y[rows])
        a -= eta * g
        theta -= eta * g
    return a / lam


def test_staleness_reads_the_scheduled_version():
    """Two workers; commit c reads theta~ after c - tau_c commits; each worker's
    data cursor continues across its commits."""
    rng = np.random.default_rng(4)
    dims, m, S, lam, eta, n = (4, 3, 3), 2, 5, 3, 0.25, 2
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(n * S, dims[0])), rng.integers(0, dims[-1], n * S)
    th0 = rng.normal(0, 0.5, mlp.num_params)
    worker = [0, 1, 0, 1, 1]
    tau = [0, 1, 1, 1, 0]
    r = O.agn_run(mlp, th0, n, lam, eta, worker, tau, _ListData(X, y), m, S,
                  snapshot_at=range(5))
    V = [th0]
    steps = [0, 0]
    for c, (w, t) in enumerate(zip(worker, tau)):
        d = _local_delta(mlp, V[c - t], X, y, w, steps[w], lam, eta, m, S)
        steps[w] += lam
        V.append(V[-1] + d)
        assert np.allclose(r.snapshots[c], V[-1], rtol=0, atol=1e-15)


# ----------------------------------------------------------------------------
# DynSGD-style staleness-scaled commit (Section 4's comparison)
# ----------------------------------------------------------------------------

def _local_sum(mlp, theta_start, X, y, k, t0, lam, eta, m, S):
    theta = theta_start.copy()
    a = np.zeros_like(theta)
    for i in range(lam):
        rows = k * S + ((t0 + i) * m + np.arange(m)) % S
        _, g = mlp.loss_grad(theta, X[rows], y[rows])
        a -= eta * g
        theta -= eta * g
    return a


def test_dynsgd_scales_each_commit_by_its_staleness():
    """Commit c adds the worker's accumulated update divided by tau_c + 1,
    tau_c = c - v_c (an independent step-by-step loop)."""
    rng = np.random.default_rng(7)
    dims, m, S, lam, eta, n = (4, 3, 3), 2, 5, 3, 0.25, 3
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(n * S, dims[0])), rng.integers(0, dims[-1], n * S)
    th0 = rng.normal(0, 0.5, mlp.num_params)
    worker = [0, 1, 2, 0, 1, 2, 1]
    tau = [0, 1, 2, 2, 1, 2, 0]
    r = O.agn_run(mlp, th0, n, lam, eta, worker, tau, _ListData(X, y), m, S,
                  snapshot_at=range(len(worker)), staleness_scaled=True)
    V = [th0]
    steps = [0] * n
    for c, (w, t) in enumerate(zip(worker, tau)):
        d = _local_sum(mlp, V[c - t], X, y, w, steps[w], lam, eta, m, S) / (t + 1)
        steps[w] += lam
        V.append(V[-1] + d)
        assert np.allclose(r.snapshots[c], V[-1], rtol=0, atol=1e-15)


def test_dynsgd_without_staleness_is_the_unnormalised_ablation():
    rng = np.random.default_rng(8)
    dims, m, S, lam = (5, 4, 3), 3, 9, 4
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(S, dims[0])), rng.integers(0, dims[-1], S)
    th0 = rng.normal(0, 0.4, mlp.num_params)
    d = _ListData(X, y)
    w, tau = [0, 0, 0], [0, 0, 0]
    r_dyn = O.agn_run(mlp, th0, 1, lam, 0.1, w, tau, d, m, S, staleness_scaled=True)
    r_un = O.agn_run(mlp, th0, 1, lam, 0.1, w, tau, d, m, S, normalize=False)
    assert np.array_equal(r_dyn.theta, r_un.theta)


def test_dynsgd_commits_from_one_version_scale_as_one_over_tau_plus_one():
    """The first n commits all read version 0 (tau_c = c), so every rule
    computes the same accumulated updates a_c; DynSGD adds a_c / (c + 1) where
    the un-normalised ablation adds a_c."""
    rng = np.random.default_rng(9)
    n = 4
    dims, m, S, lam = (4, 3, 3), 2, 6, 3
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(n * S, dims[0])), rng.integers(0, dims[-1], n * S)
    th0 = rng.normal(0, 0.4, mlp.num_params)
    d = _ListData(X, y)
    w, tau = list(range(n)), list(range(n))
    r_dyn = O.agn_run(mlp, th0, n, lam, 0.2, w, tau, d, m, S, staleness_scaled=True,
                      snapshot_at=range(n))
    r_un = O.agn_run(mlp, th0, n, lam, 0.2, w, tau, d, m, S, normalize=False,
                     snapshot_at=range(n))
    prev_un, expect = th0, th0.copy()
    for c in range(n):
        a_c = r_un.snapshots[c] - prev_un
        prev_un = r_un.snapshots[c]
        expect = expect + a_c / (c + 1)
        assert np.allclose(r_dyn.snapshots[c], expect, rtol=0, atol=1e-15)
        assert math.isclose(r_dyn.delta_norm[c] * (c + 1), r_un.delta_norm[c], rel_tol=1e-12)


# ----------------------------------------------------------------------------
# Accumulator elision: commit from the pulled parameters
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("rule", ["agn", "unnormalised", "dynsgd"])
def test_elided_commit_equals_accumulated_commit(rule):
    """(theta_lambda - theta_pull) = sum of the local updates (they telescope),
    so committing from the pull snapshot equals committing the accumulator,
    up to float64 rounding, under every commit rule."""
    rng = np.random.default_rng(12)
    dims, m, S, lam, eta, n = (5, 4, 3), 3, 7, 4, 0.2, 3
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(n * S, dims[0])), rng.integers(0, dims[-1], n * S)
    th0 = rng.normal(0, 0.5, mlp.num_params)
    worker = [0, 1, 2, 0, 1, 2, 0, 1]
    tau = [0, 1, 2, 2, 1, 2, 0, 2]
    kw = dict(normalize=rule != "unnormalised", staleness_scaled=rule == "dynsgd",
              snapshot_at=range(len(worker)))
    r_acc = O.agn_run(mlp, th0, n, lam, eta, worker, tau, _ListData(X, y), m, S, **kw)
    r_eli = O.agn_run(mlp, th0, n, lam, eta, worker, tau, _ListData(X, y), m, S,
                      elide_accumulator=True, **kw)
    for c in range(len(worker)):
        d_acc = r_acc.snapshots[c] - (r_acc.snapshots[c - 1] if c else th0)
        assert np.max(np.abs(r_eli.snapshots[c] - r_acc.snapshots[c])) <= 1e-12 * np.max(np.abs(d_acc))
    assert not np.array_equal(r_eli.theta, th0)


def test_elided_least_squares_commit_closed_form():
    """The elided commit against the closed form of the local iteration."""
    lsq, X, Y, theta0, A, Theta0, Theta_star = _lsq_setup()
    eta, lam = 0.3, 17
    S = X.shape[0]
    r = O.agn_run(lsq, theta0, 1, lam, eta, [0], [0], _ListData(X, Y), S, S,
                  elide_accumulator=True)
    ev, Q = np.linalg.eigh(A)
    Mlam = Q @ np.diag((1 - eta * ev) ** lam) @ Q.T
    Delta = (Theta0 - Theta_star) @ (Mlam - np.eye(A.shape[0])) / lam
    expect = _theta_to_flat(Theta0 + Delta, X.shape[1])
    assert np.max(np.abs(r.theta - expect)) <= 1e-10 * max(1.0, np.max(np.abs(expect)))


def test_schedule_feasibility():
    v = O.schedule_versions(3, [0, 1, 2, 0, 1, 2], [0, 1, 2, 2, 2, 2])
    assert list(v) == [0, 0, 0, 1, 2, 3]
    with pytest.raises(O.ScheduleError):      # pulls before its own commit 0
        O.schedule_versions(2, [0, 0], [0, 1])
    with pytest.raises(O.ScheduleError):      # negative staleness
        O.schedule_versions(2, [0, 1], [0, -1])
    with pytest.raises(O.ScheduleError):      # worker out of range
        O.schedule_versions(2, [0, 2], [0, 0])
    with pytest.raises(O.ScheduleError):
        O.schedule_versions(2, [0, 1, 0], [1, 0, 0])   # commit 0 would read version -1


# ----------------------------------------------------------------------------
# Float32 commit sequence (Eq. 1-2 in float32, no fused multiply-add)
# ----------------------------------------------------------------------------

def _round_f32(q: Fraction) -> Fraction:
    """Round an exact rational to the nearest float32 (ties to even)."""
    if q == 0:
        return Fraction(0)
    sign = -1 if q < 0 else 1
    q = abs(q)
    e = q.numerator.bit_length() - q.denominator.bit_length()
    if Fraction(2) ** e > q:
        e -= 1
    e = max(e, -126)                     # subnormals share the minimum exponent
    ulp = Fraction(2) ** (e - 23)
    k = q / ulp
    fl = k.numerator // k.denominator
    rem = k - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    return sign * fl * ulp


def test_commit_fp32_matches_exact_rounding():
    rng = np.random.default_rng(9)
    P, n = 257, 5
    theta = rng.normal(size=P).astype(np.float32)
    accs = {k: (0.1 * rng.normal(size=P)).astype(np.float32) for k in range(n)}
    order = [3, 0, 4, 1, 2]
    pulls = [[1, 2], [0], [4, 3, 2], [], [0, 1]]
    eta, lam = 0.01, 10
    th, ac, rep, norms = O.commit_pull_fp32(theta, accs, order, pulls, eta, lam)
    s = _round_f32(Fraction(-(eta / lam)))       # fp32 of the double -eta/lambda
    assert Fraction(float(O.commit_scale_fp32(eta, lam))) == s
    exact = [Fraction(float(v)) for v in theta]
    reps = {}
    for c, k in enumerate(order):
        for i in range(P):
            d = _round_f32(Fraction(float(accs[k][i])) * s)
            exact[i] = _round_f32(exact[i] + d)
        for p in pulls[c]:
            reps[p] = list(exact)
    assert all(Fraction(float(th[i])) == exact[i] for i in range(P))
    for p, v in reps.items():
        assert all(Fraction(float(rep[p][i])) == v[i] for i in range(P))
    assert all(np.all(ac[k] == 0) for k in range(n))
    assert norms.shape == (n,) and np.all(norms > 0)


def test_commit_fp32_unnormalised_scale():
    assert np.float32(O.commit_scale_fp32(0.01, 10, normalize=False)) == np.float32(-0.01)


# ----------------------------------------------------------------------------
# Evaluation and temporal efficiency (Section 4, Eq. 4)
# ----------------------------------------------------------------------------

def test_evaluate_hand_worked():
    """One linear layer, logits chosen by hand: accuracy exact, loss closed
    form, ties to the lowest index."""
    mlp = O.MLP((2, 3))
    W = np.array([[1.0, 0.0], [0.0, 1.0], [0.0, 0.0]])
    b = np.zeros(3)
    theta = np.concatenate([W.ravel(), b])
    X = np.array([[2.0, 0.0], [0.0, 3.0], [0.0, 0.0], [1.0, 1.0]])
    y = np.array([0, 2, 0, 1])
    loss, acc, pred = O.evaluate(mlp, theta, X, y)
    # logits: [2,0,0] -> 0; [0,3,0] -> 1; [0,0,0] -> tie -> 0; [1,1,0] -> tie -> 0
    assert pred.tolist() == [0, 1, 0, 0]
    assert acc == 0.5
    e = math.e
    expect = np.mean([math.log(e ** 2 + 2) - 2, math.log(e ** 3 + 2) - 0.0,
                      math.log(3.0), math.log(2 * e + 1) - 1])
    assert math.isclose(loss, expect, rel_tol=1e-14)


def test_evaluate_uniform_logits_is_log_classes():
    mlp = O.MLP((4, 5, 7))
    theta = np.zeros(mlp.num_params)
    X = np.random.default_rng(3).normal(size=(9, 4))
    loss, acc, pred = O.evaluate(mlp, theta, X, np.arange(9) % 7)
    assert math.isclose(loss, math.log(7), rel_tol=1e-15)
    assert np.all(pred == 0)


def test_temporal_efficiency_closed_forms():
    t = np.linspace(0.0, 10.0, 11)
    f = 0.3 + 0.05 * t
    assert O.temporal_efficiency(t, f, t, f) == 1.0
    assert math.isclose(O.temporal_efficiency(t, 2 * f, t, f), 2.0, rel_tol=1e-15)
    # f_a(t) = t, f_b = 1 on [0, 4]: E = (16 / 2) / 4
    assert math.isclose(O.temporal_efficiency([0, 4], [0, 4], [0, 4], [1, 1]), 2.0, rel_tol=1e-15)
    # the longer curve is cut at the shorter one's end, inside a segment:
    # f_a = t on [0, 10] (samples at 0 and 10), f_b = 1 on [0, 3]: E = 4.5 / 3
    assert math.isclose(O.temporal_efficiency([0, 10], [0, 10], [0, 3], [1, 1]), 1.5,
                        rel_tol=1e-15)
    # held at its first value before the first sample: f_a = 2 on [0, 1], then 2 -> 4
    # on [1, 2] (integral 2 + 3 = 5), f_b = 1: E = 5 / 2
    assert math.isclose(O.temporal_efficiency([1, 2], [2, 4], [0, 2], [1, 1]), 2.5,
                        rel_tol=1e-15)


def test_temporal_efficiency_is_exact_for_piecewise_linear_curves():
    rng = np.random.default_rng(13)
    tb = np.sort(rng.uniform(0, 5, 7))
    tb[0] = 0.0
    fb = rng.uniform(0.1, 1, 7)
    ta = np.array([0.0, 5.0])
    fa = np.array([1.0, 1.0])
    # integral of the interpolant of (tb, fb) up to tb[-1], by Fractions
    from fractions import Fraction as F
    area = sum((F(fb[i]) + F(fb[i + 1])) / 2 * (F(tb[i + 1]) - F(tb[i])) for i in range(6))
    e = O.temporal_efficiency(ta, fa, tb, fb)
    assert math.isclose(e, float(F(tb[-1]) / area), rel_tol=1e-14)


# ----------------------------------------------------------------------------
# Adam as the local optimizer (Algorithm 1's gradient line)
# ----------------------------------------------------------------------------

def test_adam_first_step_is_eta_times_the_gradient_sign():
    """At t = 1 the bias corrections give m^ = gr and v^ = gr^2, so the step
    is -eta gr / (|gr| + eps)."""
    mlp, theta, X, y = _tiny_problem(seed=4)
    eta, eps = 0.01, 1e-8
    _, gr = mlp.loss_grad(theta, X, y)
    d = _ListData(X, y)
    r = O.agn_run(mlp, theta, 1, 1, eta, [0], [0], d, len(y), len(y), optimizer="adam",
                  adam=(0.9, 0.999, eps))
    assert np.allclose(r.theta - theta, -eta * gr / (np.abs(gr) + eps), rtol=0, atol=1e-15)


def _adam_golden_rows():
    rows = []
    with open(os.path.join(GOLDEN, "adam_scalar_examples.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                lam, nc, val = line.split()
                rows.append((int(lam), int(nc), Fraction(val)))
    return rows


@pytest.mark.parametrize("lam,n_commits,expect", _adam_golden_rows())
def test_adam_hand_worked_two_steps(lam, n_commits, expect):
    """Two Adam steps worked by hand in exact rationals (the bias corrections
    at t = 1 and t = 2, moments kept across a commit): the oracle within a few
    roundings of the exact value."""
    lsq = O.LeastSquares(1, 1)
    data = _ListData(np.array([[1.0]]), np.array([[0.0]]))

    class WOnly:
        num_params = 1

        def loss_grad(self, theta, X, Y):
            loss, g = lsq.loss_grad(np.array([theta[0], 0.0]), X, Y)
            return loss, g[:1]
    r = O.agn_run(WOnly(), np.array([1.0]), 1, lam, 0.5, [0] * n_commits, [0] * n_commits,
                  data, 1, 1, optimizer="adam", adam=(0.5, 11 / 64, 0.0))
    assert abs(Fraction(float(r.theta[0])) - expect) <= Fraction(1, 2 ** 48)


def test_adam_moments_persist_across_commits():
    """An independent loop: moments per worker, bias corrections at the
    worker's step count, staleness as scheduled."""
    rng = np.random.default_rng(14)
    dims, m, S, lam, eta, n = (4, 3, 3), 2, 5, 3, 0.05, 2
    b1, b2, eps = 0.8, 0.99, 1e-6
    mlp = O.MLP(dims)
    X, y = rng.uniform(size=(n * S, dims[0])), rng.integers(0, dims[-1], n * S)
    th0 = rng.normal(0, 0.5, mlp.num_params)
    worker = [0, 1, 0, 1, 1, 0]
    tau = [0, 1, 1, 1, 0, 2]
    r = O.agn_run(mlp, th0, n, lam, eta, worker, tau, _ListData(X, y), m, S,
                  snapshot_at=range(len(worker)), optimizer="adam", adam=(b1, b2, eps))
    V = [th0]
    steps = [0] * n
    mom = [(np.zeros_like(th0), np.zeros_like(th0)) for _ in range(n)]
    for c, (w, t) in enumerate(zip(worker, tau)):
        theta = V[c - t].copy()
        a = np.zeros_like(theta)
        m1, m2 = mom[w]
        for i in range(lam):
            rows = w * S + ((steps[w] + i) * m + np.arange(m)) % S
            _, gr = mlp.loss_grad(theta, X[rows], y[rows])
            m1 = b1 * m1 + (1 - b1) * gr
            m2 = b2 * m2 + (1 - b2) * gr ** 2
            k = steps[w] + i + 1
            g = -eta * (m1 / (1 - b1 ** k)) / (np.sqrt(m2 / (1 - b2 ** k)) + eps)
            a += g
            theta += g
        mom[w] = (m1, m2)
        steps[w] += lam
        V.append(V[-1] + a / lam)
        assert np.allclose(r.snapshots[c], V[-1], rtol=0, atol=1e-14)
