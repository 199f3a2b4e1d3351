"""CPU oracle of the AGN hot path (Accumulated Gradient Normalization,
Hermans, Spanakis & Moeckel, ACML 2017).

TEST INFRASTRUCTURE ONLY.  Plain, slow, obviously correct NumPy.  Only the
tests, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` may
import or run anything in this package; the library's product path never
does, and this file imports nothing from the CUDA library.  Its inputs come
from `agn_inputs` (the seeded generator, which holds none of the method's
arithmetic).

What it computes, in the paper's order and notation:

* Worker procedure, Algorithm 1: theta_k <- Pull(); a <- 0; lambda times:
  fetch the next minibatch, g <- -eta grad L(theta_k; x, y), a <- a + g,
  theta_k <- theta_k + g; then a <- a / lambda (the normalisation step),
  Commit(a), Pull.
* Worker delta, Eq. 1: Delta theta^k = -(1/lambda) sum_i eta (1/m) sum_j
  grad L(theta_i; x_ij, y_ij).  The sum runs over the lambda local steps of
  Algorithm 1 (i = 0 .. lambda-1); see `agn_run`.
* Parameter-server update, Eq. 2: theta~_{t+1} = theta~_t + Delta theta^k,
  commits applied one at a time in FIFO order (Fig. 1).
* Minibatch gradient (Section 3): the mean over m samples of the per-sample
  gradient; the loss is softmax cross-entropy (classification, Section 4).

Readings where the paper is silent or inconsistent (each is also listed in
the design notes):
  - Eq. 1 and Eq. 3 sum i = 0..lambda but divide by lambda; Algorithm 1 runs
    i < lambda.  The oracle takes lambda terms (Algorithm 1).
  - Section 3 speaks of "m - 1 samples" while its sum has m terms; the
    oracle averages over m samples.
  - Minibatches: Algorithm 1's FetchNextMiniBatch over the worker's shard,
    read cyclically: rows (t m + j) mod S of shard k, t the worker's step
    counter, which is never reset (Algorithm 1 keeps t across commits).
  - Staleness: an explicit schedule (w_c, tau_c); commit c was computed from
    theta~ after v_c = c - tau_c commits (Fig. 1's FIFO queue).  A worker pulls
    only after its own previous commit (Algorithm 1), so prev(w_c) < v_c <= c.
  - Un-normalised ablation (Fig. 3, "accumulated gradient DOWNPOUR"):
    the same loop without the division by lambda.
  - Learning rate eta constant (Section 4: no decay).
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "ScheduleError", "MLP", "LeastSquares", "softmax_xent", "batch_rows",
    "schedule_versions", "agn_run", "AGNResult", "commit_pull_fp32",
    "commit_scale_fp32", "evaluate", "temporal_efficiency",
]


class ScheduleError(ValueError):
    """An infeasible (worker, staleness) pair."""


# ----------------------------------------------------------------------------
# Models and the minibatch gradient (Eq. 1 inner term)
# ----------------------------------------------------------------------------

def softmax_xent(z: np.ndarray, y: np.ndarray):
    """Mean softmax cross-entropy over the rows of z and its gradient.

    loss = (1/m) sum_j [logsumexp(z_j) - z_j[y_j]] (log-sum-exp with the row
    maximum subtracted); dL/dz = (softmax(z) - onehot(y)) / m.
    """
    m = z.shape[0]
    zmax = z.max(axis=1, keepdims=True)
    e = np.exp(z - zmax)
    s = e.sum(axis=1, keepdims=True)
    lse = np.log(s) + zmax
    rows = np.arange(m)
    loss = float(np.mean(lse[:, 0] - z[rows, y]))
    dz = e / s
    dz[rows, y] -= 1.0
    dz /= m
    return loss, dz


class MLP:
    """ReLU MLP with a softmax cross-entropy head.

    Parameters live in one flat vector: for l = 1..L, W_l row-major
    [d_l][d_{l-1}], then b_l [d_l].  Hidden layers h_l = relu(h_{l-1} W_l^T + b_l),
    output z = h_{L-1} W_L^T + b_L.
    """

    def __init__(self, dims, dtype=np.float64):
        self.dims = tuple(int(d) for d in dims)
        self.dtype = dtype
        self.offsets = []
        off = 0
        for l in range(1, len(self.dims)):
            fi, fo = self.dims[l - 1], self.dims[l]
            self.offsets.append((off, off + fo * fi, off + fo * fi + fo))
            off += fo * fi + fo
        self.num_params = off

    def unpack(self, theta):
        out = []
        for l, (ow, ob, oe) in enumerate(self.offsets, start=1):
            fi, fo = self.dims[l - 1], self.dims[l]
            out.append((theta[ow:ob].reshape(fo, fi), theta[ob:oe]))
        return out

    def loss_grad(self, theta, X, y):
        """Minibatch loss and gradient (1/m) sum_j grad L(theta; x_j, y_j)."""
        params = self.unpack(theta)
        L = len(params)
        h = [X.astype(self.dtype, copy=False)]
        for l, (W, b) in enumerate(params):
            z = h[-1] @ W.T + b
            if l + 1 < L:
                z = np.maximum(z, 0.0)
            h.append(z)
        loss, dz = softmax_xent(h[-1], y)
        grad = np.zeros(self.num_params, dtype=self.dtype)
        for l in range(L - 1, -1, -1):
            W, _ = params[l]
            ow, ob, oe = self.offsets[l]
            grad[ow:ob] = (dz.T @ h[l]).ravel()
            grad[ob:oe] = dz.sum(axis=0)
            if l > 0:
                dz = (dz @ W) * (h[l] > 0)
        return loss, grad


class LeastSquares:
    """Linear model f(x) = W x + b with loss (1/m) sum_j 1/2 ||f(x_j) - y_j||^2.

    An oracle-only model whose local SGD iteration has a closed form, used to
    pin the AGN loop (Section 3's thought experiment on lambda).
    Flat order: W row-major [d_out][d_in], then b.
    """

    def __init__(self, d_in, d_out, dtype=np.float64):
        self.d_in, self.d_out = int(d_in), int(d_out)
        self.dtype = dtype
        self.num_params = self.d_out * self.d_in + self.d_out

    def loss_grad(self, theta, X, Y):
        W = theta[: self.d_out * self.d_in].reshape(self.d_out, self.d_in)
        b = theta[self.d_out * self.d_in:]
        m = X.shape[0]
        r = X @ W.T + b - Y
        loss = float(0.5 * np.sum(r * r) / m)
        gW = (r.T @ X) / m
        gb = r.sum(axis=0) / m
        return loss, np.concatenate([gW.ravel(), gb])


# ----------------------------------------------------------------------------
# Data access and schedule
# ----------------------------------------------------------------------------

def batch_rows(k: int, t: int, m: int, shard: int) -> np.ndarray:
    """Dataset rows of worker k's minibatch at its local step t.

    Shard k holds rows [k S, (k+1) S); the minibatch is rows
    k S + (t m + j) mod S, j = 0..m-1 (FetchNextMiniBatch, Algorithm 1).
    """
    return k * shard + (t * m + np.arange(m, dtype=np.int64)) % shard


def schedule_versions(n: int, worker, tau, prev=None):
    """Versions v_c = c - tau_c read by each commit, after checking feasibility.

    `prev[w]` is the index of worker w's last commit before this schedule
    starts (-1 for none); indices continue from `start = ` the number of
    commits already applied, given by `prev` (see `agn_run`).
    """
    worker = np.asarray(worker, dtype=np.int64)
    tau = np.asarray(tau, dtype=np.int64)
    if worker.shape != tau.shape:
        raise ScheduleError("worker and staleness arrays differ in length")
    prev = np.full(n, -1, dtype=np.int64) if prev is None else np.array(prev, dtype=np.int64)
    v = np.empty_like(tau)
    for c in range(len(worker)):
        w = int(worker[c])
        if not 0 <= w < n:
            raise ScheduleError(f"commit {c}: worker {w} out of range")
        vc = c - int(tau[c])
        if tau[c] < 0 or vc <= prev[w]:
            raise ScheduleError(
                f"commit {c}: worker {w} cannot read version {vc} "
                f"(its previous commit is {prev[w]})")
        v[c] = vc
        prev[w] = c
    return v


# ----------------------------------------------------------------------------
# The AGN event loop
# ----------------------------------------------------------------------------

@dataclass
class AGNResult:
    theta: np.ndarray                       # final central variable
    loss: np.ndarray                        # per commit: mean of the lambda minibatch losses
    delta_norm: np.ndarray                  # per commit: ||Delta||_2
    theta_norm: np.ndarray                  # per commit: ||theta~||_2 after it
    snapshots: dict = field(default_factory=dict)   # commit index -> theta~ after it
    locals_: dict = field(default_factory=dict)     # commit index -> list of local iterates


def agn_run(model, theta0, n, lam, eta, worker, tau, data, batch, shard,
            normalize=True, snapshot_at=(), keep_locals=(), dtype=np.float64,
            staleness_scaled=False, elide_accumulator=False, optimizer="sgd",
            adam=(0.9, 0.999, 1e-8)):
    """Run the commits of one schedule through the FIFO parameter server.

    model      : object with loss_grad(theta, X, y) -> (loss, grad)
    theta0     : initial central variable (flat)
    data       : callable rows -> (X, y) (dataset rows, float array, labels)
    batch      : m; shard: S (rows per worker)
    worker,tau : the schedule (commit c by worker[c] from version c - tau[c])

    Commit c (in FIFO order, Eq. 2): the worker's replica is theta~ after
    v_c commits (its Pull); it takes lambda local steps (Algorithm 1):
        g = -eta * grad;  a = a + g;  theta = theta + g
    then a = a / lambda (skipped when normalize is False) and theta~ += a.

    staleness_scaled: the DynSGD-style commit the paper compares against
    (Section 4): the accumulated update divided by tau_c + 1, where
    tau_c = c - v_c is the number of commits between the worker's pull and
    its commit, instead of by lambda (`normalize` is then ignored).

    elide_accumulator: no accumulator; the commit is formed from the local
    iterate and the pulled parameters, (theta_lambda - theta_pull) scaled the
    same way.  Equal to the accumulated form in exact arithmetic (the
    accumulated updates telescope).

    optimizer="adam": the local step g of Algorithm 1 comes from Adam (named
    there as an example): with the minibatch gradient gr at the worker's
    step count t = 1, 2, ... (never reset), m = b1 m + (1 - b1) gr,
    v = b2 v + (1 - b2) gr^2, g = -eta (m / (1 - b1^t)) / (sqrt(v / (1 - b2^t))
    + eps); the moments belong to the worker and persist across its commits.
    """
    worker = np.asarray(worker, dtype=np.int64)
    v = schedule_versions(n, worker, tau)
    C = len(worker)
    theta_c = np.array(theta0, dtype=dtype, copy=True)
    eta = dtype(eta)
    # Versions still to be read, and the snapshot of theta~ at each of them.
    readers = {}
    for c in range(C):
        readers.setdefault(int(v[c]), []).append(c)
    snaps = {}
    if 0 in readers:
        snaps[0] = theta_c.copy()
    step = np.zeros(n, dtype=np.int64)
    if optimizer not in ("sgd", "adam"):
        raise ValueError("optimizer must be 'sgd' or 'adam'")
    b1, b2, eps_a = (dtype(x) for x in adam)
    mom = {}                                            # worker -> (m, v)
    loss = np.zeros(C)
    dnorm = np.zeros(C)
    tnorm = np.zeros(C)
    out_snap = {}
    out_locals = {}
    snapshot_at = set(int(s) for s in snapshot_at)
    keep_locals = set(int(s) for s in keep_locals)
    for c in range(C):
        k = int(worker[c])
        vc = int(v[c])
        theta = snaps[vc].copy()                       # Pull
        snaps_pull = theta.copy() if elide_accumulator else None
        readers[vc].remove(c)
        if not readers[vc]:
            del snaps[vc]
        a = np.zeros_like(theta)
        losses = []
        iterates = [theta.copy()] if c in keep_locals else None
        for _ in range(lam):
            X, y = data(batch_rows(k, int(step[k]), batch, shard))
            li, grad = model.loss_grad(theta, X.astype(dtype, copy=False), y)
            if optimizer == "adam":
                m1, m2 = mom.get(k, (np.zeros_like(theta), np.zeros_like(theta)))
                m1 = b1 * m1 + (1 - b1) * grad
                m2 = b2 * m2 + (1 - b2) * grad * grad
                mom[k] = (m1, m2)
                t = int(step[k]) + 1
                g = -eta * (m1 / (1 - b1 ** t)) / (np.sqrt(m2 / (1 - b2 ** t)) + eps_a)
            else:
                g = -eta * grad
            a = a + g
            theta = theta + g
            step[k] += 1
            losses.append(li)
            if iterates is not None:
                iterates.append(theta.copy())
        if elide_accumulator:
            a = theta - snaps_pull                      # sum of the local updates
        if staleness_scaled:
            a = a / dtype(c - vc + 1)                   # DynSGD: 1 / (tau_c + 1)
        elif normalize:
            a = a / dtype(lam)                          # normalisation step
        theta_c = theta_c + a                           # Eq. 2
        loss[c] = float(np.mean(losses))
        dnorm[c] = float(np.sqrt(np.sum(a.astype(np.float64) ** 2)))
        tnorm[c] = float(np.sqrt(np.sum(theta_c.astype(np.float64) ** 2)))
        if (c + 1) in readers:
            snaps[c + 1] = theta_c.copy()
        if c in snapshot_at:
            out_snap[c] = theta_c.copy()
        if iterates is not None:
            out_locals[c] = iterates
    return AGNResult(theta_c, loss, dnorm, tnorm, out_snap, out_locals)


# ----------------------------------------------------------------------------
# Commit + pull in float32, in a fixed order (the standalone workload)
# ----------------------------------------------------------------------------

def commit_scale_fp32(eta: float, lam: int, normalize: bool = True) -> np.float32:
    """Commit scale of Eq. 1 applied to a raw gradient sum a: Delta = s a.

    s = fp32(-eta / lambda) computed in double (fp32(-eta) without the
    normalisation).  Algorithm 1 folds -eta into g; the sum of raw gradients
    times s is the same quantity.
    """
    return np.float32(-(float(eta) / float(lam)) if normalize else -float(eta))


def commit_pull_fp32(theta_c, accs, order, pulls, eta, lam, normalize=True,
                     replicas=None):
    """Apply the commits of `order` to theta~ in float32, then the pulls.

    For commit c of accumulator k = order[c]: Delta = fp32(a_k * s) and
    theta~ = fp32(theta~ + Delta), element by element, with no fused
    multiply-add (Eq. 1-2); a_k <- 0 (Algorithm 1 restarts the accumulator);
    every worker in pulls[c] then copies theta~ (Pull).  Works on any subset
    of parameter indices, since each element is independent.
    Returns (theta~, accs, replicas, per-commit ||Delta||_2 in float64).
    """
    s = commit_scale_fp32(eta, lam, normalize)
    theta_c = np.array(theta_c, dtype=np.float32, copy=True)
    accs = {k: np.array(v, dtype=np.float32, copy=True) for k, v in accs.items()}
    replicas = {} if replicas is None else {k: np.array(v, dtype=np.float32) for k, v in replicas.items()}
    norms = np.zeros(len(order))
    for c, k in enumerate(order):
        k = int(k)
        delta = np.multiply(accs[k], s, dtype=np.float32)
        theta_c = np.add(theta_c, delta, dtype=np.float32)
        accs[k][:] = 0.0
        norms[c] = math.sqrt(float(np.sum(delta.astype(np.float64) ** 2)))
        for p in pulls[c]:
            replicas[int(p)] = theta_c.copy()
    return theta_c, accs, replicas, norms


# ----------------------------------------------------------------------------
# Evaluation and temporal efficiency (Section 4, Eq. 4)
# ----------------------------------------------------------------------------

def evaluate(model, theta, X, y, dtype=np.float64):
    """(mean softmax cross-entropy, accuracy, predictions) of parameters theta
    on the rows of X: the forward pass of the model, log-sum-exp with the row
    maximum subtracted, prediction = argmax with the lowest index on ties."""
    h = np.asarray(X, dtype=dtype)
    params = model.unpack(np.asarray(theta, dtype=dtype))
    for l, (W, b) in enumerate(params):
        h = h @ W.T + b
        if l + 1 < len(params):
            h = np.maximum(h, 0)
    y = np.asarray(y, dtype=np.int64)
    zmax = h.max(axis=1, keepdims=True)
    lse = np.log(np.exp(h - zmax).sum(axis=1)) + zmax[:, 0]
    loss = float(np.mean(lse - h[np.arange(len(y)), y]))
    pred = np.argmax(h, axis=1)          # first maximum: the lowest index on ties
    return loss, float(np.mean(pred == y)), pred


def _curve_integral(t, f, m):
    """Integral over [0, m] of the piecewise-linear interpolation of (t, f),
    held at f[0] on [0, t[0]]."""
    t = np.asarray(t, dtype=np.float64)
    f = np.asarray(f, dtype=np.float64)
    total = f[0] * min(t[0], m)
    for i in range(len(t) - 1):
        t0, t1 = t[i], t[i + 1]
        if t0 >= m:
            break
        if t1 <= t0:
            continue
        if t1 > m:                       # the segment is cut at m
            f_m = f[i] + (f[i + 1] - f[i]) * (m - t0) / (t1 - t0)
            total += 0.5 * (f[i] + f_m) * (m - t0)
            break
        total += 0.5 * (f[i] + f[i + 1]) * (t1 - t0)
    return total


def temporal_efficiency(ta, fa, tb, fb):
    """Eq. 4: E(a, b) = int_0^m f_a dt / int_0^m f_b dt, m the minimal shared
    training time (the shorter curve's end).  Each curve is the piecewise-
    linear interpolation of its samples (the paper leaves the quadrature open)."""
    m = min(float(ta[-1]), float(tb[-1]))
    if not m > 0:
        raise ValueError("no shared training time")
    return _curve_integral(ta, fa, m) / _curve_integral(tb, fb, m)
