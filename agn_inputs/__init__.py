"""Seeded synthetic inputs for the AGN hot path.

This package generates every input both implementations consume: the
dataset X, the teacher labels y, the initial central variable, the
(worker, staleness) commit schedule, and the inputs of the standalone
commit+pull workload.  It holds none of AGN's arithmetic (no gradient, no
local step, no commit); it is shared by the CPU oracle, the tests and the
benchmark, and the CUDA library carries its own implementation of the same
generator in C++ (checked bit for bit against this one by the tests).

Generator (counter-based splitmix64, Steele, Lea & Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014; output function as in Vigna's
public-domain splitmix64.c):

    G  = 0x9E3779B97F4A7C15,  mix(z) = z ^= z>>30, z *= 0xBF58476D1CE4E5B9,
                                       z ^= z>>27, z *= 0x94D049BB133111EB,
                                       z ^ z>>31            (all mod 2^64)
    key(seed, stream) = mix(seed ^ (stream * G))
    draw(key, i)      = mix(key + (i + 1) * G)   (the i-th splitmix64 output
                                                  of a generator seeded with key)

Derived variates, written with correctly rounded IEEE-754 double operations
only (+, -, *, /, sqrt, frexp), so any language reproduces them exactly
(C/C++ must compile them without FMA contraction):

    U[0,1) float32 : (d >> 40) * 2^-24          (exact in float32)
    U[0,1) float64 : (d >> 11) * 2^-53
    N(0,1)         : Box-Muller, cos branch, from draws 2i and 2i+1:
                     r = sqrt(-2 ln(1 - u1)), z = r cos(2 pi u2), with ln and
                     cos evaluated by the fixed series in `ln_series` / `cos2pi_series`
                     (atanh series after frexp; Taylor series on [-pi, pi)).

The paper's experiments use MNIST (Section 4), which is not available here;
these seeded sets take its shape (784 features, 10 classes) and stand in for
it, with labels from a random ReLU teacher network.
"""

from __future__ import annotations

import numpy as np

__all__ = [
    "G", "STREAM_DATA", "STREAM_TEACHER", "STREAM_INIT", "STREAM_SCHEDULE",
    "STREAM_COMMIT_ACC", "STREAM_COMMIT_THETA", "STREAM_COMMIT_ORDER",
    "mix64", "stream_key", "draw", "uniform_f32", "uniform_f64", "normal_f64",
    "ln_series", "cos2pi_series", "make_inputs_x", "teacher_params",
    "teacher_labels", "init_params", "layer_offsets", "num_params",
    "make_schedule", "commit_bench_order", "commit_bench_acc",
    "commit_bench_theta", "normal_f32", "DEFAULT_SEED",
    "SyntheticDataset", "workload_dataset", "workload_schedule",
]

_M64 = (1 << 64) - 1
G = 0x9E3779B97F4A7C15
_C1 = 0xBF58476D1CE4E5B9
_C2 = 0x94D049BB133111EB

STREAM_DATA = 1
STREAM_TEACHER = 2
STREAM_INIT = 3
STREAM_SCHEDULE = 4
STREAM_COMMIT_ACC = 5
STREAM_COMMIT_THETA = 6
STREAM_COMMIT_ORDER = 7

DEFAULT_SEED = 1710023680

_U64 = np.uint64


def mix64(z):
    """splitmix64 output function on a uint64 array (wrapping arithmetic)."""
    z = np.asarray(z, dtype=_U64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> _U64(30))) * _U64(_C1)
        z = (z ^ (z >> _U64(27))) * _U64(_C2)
    return z ^ (z >> _U64(31))


def _mix_int(z: int) -> int:
    z &= _M64
    z = ((z ^ (z >> 30)) * _C1) & _M64
    z = ((z ^ (z >> 27)) * _C2) & _M64
    return z ^ (z >> 31)


def stream_key(seed: int, stream: int) -> int:
    """Key of one named stream: mix(seed ^ stream*G)."""
    return _mix_int((seed & _M64) ^ ((stream * G) & _M64))


def draw(key: int, idx) -> np.ndarray:
    """draw(key, i) = mix(key + (i+1)*G) for every i in `idx` (uint64 array)."""
    idx = np.asarray(idx, dtype=_U64)
    with np.errstate(over="ignore"):
        z = _U64(key) + (idx + _U64(1)) * _U64(G)
    return mix64(z)


def uniform_f32(key: int, idx) -> np.ndarray:
    """U[0,1) in float32: top 24 bits of the draw times 2^-24 (exact)."""
    d = draw(key, idx)
    return ((d >> _U64(40)).astype(np.float64) * (2.0 ** -24)).astype(np.float32)


def uniform_f64(key: int, idx) -> np.ndarray:
    """U[0,1) in float64: top 53 bits of the draw times 2^-53 (exact)."""
    d = draw(key, idx)
    return (d >> _U64(11)).astype(np.float64) * (2.0 ** -53)


# Constants shared digit for digit with the C++ generator.
_LN2 = 0.6931471805599453094
_SQRT_HALF = 0.70710678118654752440
_PI = 3.14159265358979323846
_TWO_PI = 6.28318530717958647692
_LN_TERMS = 12      # atanh series terms: |s| <= 0.1716, s^25/25 < 1e-20
_COS_TERMS = 17     # Taylor terms on [-pi, pi): pi^32/32! < 1e-19


def _ln_coeffs():
    return [1.0 / float(2 * k + 1) for k in range(_LN_TERMS)]


def _cos_coeffs():
    c = [1.0]
    for k in range(1, _COS_TERMS):
        c.append(-c[-1] / float((2 * k - 1) * (2 * k)))
    return c


def ln_series(x: np.ndarray) -> np.ndarray:
    """Natural log of x in (0, 1] from frexp + the atanh series.

    x = f 2^e with f in [sqrt(1/2), sqrt(2)); ln f = 2 atanh(s), s=(f-1)/(f+1),
    atanh(s) = s (1 + s^2/3 + s^4/5 + ...), evaluated by Horner from the top.
    """
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)                      # f in [0.5, 1)
    small = f < _SQRT_HALF
    f = np.where(small, f * 2.0, f)
    e = np.where(small, e - 1, e).astype(np.float64)
    s = (f - 1.0) / (f + 1.0)
    s2 = s * s
    co = _ln_coeffs()
    p = np.full_like(s, co[-1])
    for k in range(_LN_TERMS - 2, -1, -1):
        p = p * s2 + co[k]
    lnf = (2.0 * s) * p
    return e * _LN2 + lnf


def cos2pi_series(t: np.ndarray) -> np.ndarray:
    """cos(2 pi t) for t in [0, 1): -cos(th) with th = 2 pi t - pi in [-pi, pi)."""
    t = np.asarray(t, dtype=np.float64)
    th = t * _TWO_PI - _PI
    th2 = th * th
    co = _cos_coeffs()
    p = np.full_like(th, co[-1])
    for k in range(_COS_TERMS - 2, -1, -1):
        p = p * th2 + co[k]
    return -p


def normal_f64(key: int, idx) -> np.ndarray:
    """N(0,1) variate number i, from draws 2i (radius) and 2i+1 (angle)."""
    idx = np.asarray(idx, dtype=_U64)
    u1 = uniform_f64(key, idx * _U64(2))
    u2 = uniform_f64(key, idx * _U64(2) + _U64(1))
    r = np.sqrt(-2.0 * ln_series(1.0 - u1))
    return r * cos2pi_series(u2)


# ----------------------------------------------------------------------------
# Dataset, teacher labels, initial parameters
# ----------------------------------------------------------------------------

DIST_UNIFORM = 0   # x ~ U[0,1)^d0, centred by 0.5 for the teacher
DIST_NORMAL = 1    # x ~ N(0,1)^d0, centred by 0


def make_inputs_x(seed: int, d0: int, rows, dist: int) -> np.ndarray:
    """Rows `rows` of the float32 dataset X[N, d0] (row-major, element r*d0+c)."""
    rows = np.asarray(rows, dtype=np.int64)
    key = stream_key(seed, STREAM_DATA)
    idx = (rows[:, None].astype(_U64) * _U64(d0) + np.arange(d0, dtype=_U64)[None, :])
    if dist == DIST_UNIFORM:
        return uniform_f32(key, idx)
    if dist == DIST_NORMAL:
        return normal_f64(key, idx).astype(np.float32)
    raise ValueError(f"unknown input distribution {dist}")


def teacher_params(seed: int, teacher_dims) -> list:
    """Teacher ReLU MLP weights in float64 (biases are zero).

    W_l ~ N(0, 2/fan_in), element (o, i) of layer l at draw index
    offset_l + o*fan_in + i.  Every layer after the first takes ReLU outputs,
    whose mean is positive; its rows are centred (row sum taken sequentially
    over i) so that no class dominates the argmax labels.
    """
    key = stream_key(seed, STREAM_TEACHER)
    Ws = []
    off = 0
    for l in range(1, len(teacher_dims)):
        fi, fo = int(teacher_dims[l - 1]), int(teacher_dims[l])
        idx = np.arange(off, off + fo * fi, dtype=_U64)
        std = np.sqrt(2.0 / float(fi))
        W = (normal_f64(key, idx) * std).reshape(fo, fi)
        if l > 1:
            s = np.zeros(fo, dtype=np.float64)
            for i in range(fi):
                s = s + W[:, i]
            W = W - (s / float(fi))[:, None]
        Ws.append(W)
        off += fo * fi
    return Ws


def teacher_labels(X: np.ndarray, Ws: list, dist: int) -> np.ndarray:
    """argmax of the teacher (float64, lowest index on ties) on centred X."""
    h = X.astype(np.float64) - (0.5 if dist == DIST_UNIFORM else 0.0)
    for l, W in enumerate(Ws):
        h = h @ W.T
        if l + 1 < len(Ws):
            h = np.maximum(h, 0.0)
    return np.argmax(h, axis=1).astype(np.int32)


def layer_offsets(dims) -> list:
    """(offset of W_l, offset of b_l) in the flat parameter vector.

    Flat order: for l = 1..L, W_l row-major [d_l][d_{l-1}], then b_l [d_l].
    """
    out = []
    off = 0
    for l in range(1, len(dims)):
        fi, fo = int(dims[l - 1]), int(dims[l])
        out.append((off, off + fo * fi))
        off += fo * fi + fo
    return out


def num_params(dims) -> int:
    return sum(int(dims[l]) * int(dims[l - 1]) + int(dims[l]) for l in range(1, len(dims)))


def init_params(seed: int, dims) -> np.ndarray:
    """Initial central variable, float32, flat order.

    Glorot-uniform weights (Keras' default initialiser; the paper's
    experiments use Keras, Section 4): W ~ U[-r, r], r = sqrt(6/(fan_in+fan_out)),
    element at flat index j from draw j: fp32((2u - 1) r).  Biases are 0.
    """
    key = stream_key(seed, STREAM_INIT)
    theta = np.zeros(num_params(dims), dtype=np.float32)
    for l, (ow, ob) in enumerate(layer_offsets(dims), start=1):
        fi, fo = int(dims[l - 1]), int(dims[l])
        r = np.sqrt(6.0 / float(fi + fo))
        u = uniform_f64(key, np.arange(ow, ob, dtype=_U64))
        theta[ow:ob] = ((2.0 * u - 1.0) * r).astype(np.float32)
    return theta


# ----------------------------------------------------------------------------
# Commit schedule
# ----------------------------------------------------------------------------

SCHED_ROUND_ROBIN = 0


def make_schedule(n: int, n_commits: int, tau_lo: int, tau_hi: int, seed: int,
                  kind: int = SCHED_ROUND_ROBIN):
    """Seeded (worker, staleness) schedule.

    Round robin: commit c belongs to worker c mod n; its staleness
    tau_c = lo + ((d_c >> 40) * (hi - lo + 1)) >> 24 is clamped to
    c - prev(w_c) - 1 so that the worker's pull follows its own previous
    commit (prev = -1 before the first).  Returns int32 arrays (worker, tau).
    """
    if kind != SCHED_ROUND_ROBIN:
        raise ValueError("unknown schedule kind")
    if not (0 <= tau_lo <= tau_hi):
        raise ValueError("need 0 <= tau_lo <= tau_hi")
    key = stream_key(seed, STREAM_SCHEDULE)
    d = draw(key, np.arange(n_commits, dtype=_U64))
    span = _U64(tau_hi - tau_lo + 1)
    tau = (tau_lo + (((d >> _U64(40)) * span) >> _U64(24))).astype(np.int64)
    worker = np.arange(n_commits, dtype=np.int64) % n
    prev = np.full(n, -1, dtype=np.int64)
    for c in range(n_commits):
        w = worker[c]
        tau[c] = min(tau[c], c - prev[w] - 1)
        prev[w] = c
    return worker.astype(np.int32), tau.astype(np.int32)


# ----------------------------------------------------------------------------
# Standalone commit+pull workload
# ----------------------------------------------------------------------------

def _bounded(key: int, ctr: int, bound: int) -> int:
    """Integer in [0, bound) from draw ctr: ((d >> 40) * bound) >> 24."""
    d = int(draw(key, np.array([ctr], dtype=_U64))[0])
    return ((d >> 40) * bound) >> 24


def commit_bench_order(seed: int, n: int, pulls_per_commit: int):
    """Commit order (a permutation of the n accumulators) and pulls.

    Permutation: Fisher-Yates, for i = n-1 .. 1 swap p[i] with p[j],
    j = bounded(draw ctr n-1-i, i+1).  Pulls after commit c: a partial
    Fisher-Yates on the identity, r = 0..R-1, j = r + bounded(ctr n + c*R + r,
    n - r), swap, pull q[r].  Returns (order int32 [n], pulls int32 [n, R]).
    """
    if not (1 <= pulls_per_commit <= n):
        raise ValueError("need 1 <= pulls_per_commit <= n")
    key = stream_key(seed, STREAM_COMMIT_ORDER)
    p = list(range(n))
    ctr = 0
    for i in range(n - 1, 0, -1):
        j = _bounded(key, ctr, i + 1)
        ctr += 1
        p[i], p[j] = p[j], p[i]
    R = pulls_per_commit
    pulls = np.zeros((n, R), dtype=np.int32)
    for c in range(n):
        q = list(range(n))
        for r in range(R):
            j = r + _bounded(key, n + c * R + r, n - r)
            q[r], q[j] = q[j], q[r]
            pulls[c, r] = q[r]
    return np.array(p, dtype=np.int32), pulls


# float32 variant of the normal variate, used by the standalone commit
# workload (hundreds of millions of draws per accumulator, generated on the
# GPU): the same Box-Muller with float32 series, every operation a correctly
# rounded float32 +, -, *, / or sqrt.
_LN_TERMS_F32 = 6      # s^11/11 < 3e-10
_COS_TERMS_F32 = 12    # pi^24/24! < 5e-13
_F32 = np.float32


def normal_f32(key: int, idx) -> np.ndarray:
    """N(0,1) variate number i in float32 arithmetic (draws 2i and 2i+1)."""
    idx = np.asarray(idx, dtype=_U64)
    d1 = draw(key, idx * _U64(2))
    d2 = draw(key, idx * _U64(2) + _U64(1))
    u1 = ((d1 >> _U64(40)).astype(np.float64) * (2.0 ** -24)).astype(_F32)
    u2 = ((d2 >> _U64(40)).astype(np.float64) * (2.0 ** -24)).astype(_F32)
    x = _F32(1.0) - u1                                   # exact, in (0, 1]
    f, e = np.frexp(x)
    small = f < _F32(_SQRT_HALF)
    f = np.where(small, f * _F32(2.0), f).astype(_F32)
    e = np.where(small, e - 1, e).astype(_F32)
    s = (f - _F32(1.0)) / (f + _F32(1.0))
    s2 = s * s
    p = np.full_like(s, _F32(1.0) / _F32(2 * (_LN_TERMS_F32 - 1) + 1))
    for k in range(_LN_TERMS_F32 - 2, -1, -1):
        p = p * s2 + _F32(1.0) / _F32(2 * k + 1)
    ln = e * _F32(_LN2) + (_F32(2.0) * s) * p
    r = np.sqrt(_F32(-2.0) * ln)
    c = [_F32(1.0)]
    for k in range(1, _COS_TERMS_F32):
        c.append(_F32(-c[-1] / _F32((2 * k - 1) * (2 * k))))
    th = u2 * _F32(_TWO_PI) - _F32(_PI)
    th2 = th * th
    q = np.full_like(th, c[-1])
    for k in range(_COS_TERMS_F32 - 2, -1, -1):
        q = q * th2 + c[k]
    return (r * (-q)).astype(_F32)


def commit_bench_acc(seed: int, P: int, k: int, idx=None) -> np.ndarray:
    """Accumulator k, a_k ~ N(0, 1e-2): fp32(0.1) * z, z = float32 normal number k*P + i."""
    key = stream_key(seed, STREAM_COMMIT_ACC)
    i = np.arange(P, dtype=_U64) if idx is None else np.asarray(idx, dtype=_U64)
    return normal_f32(key, _U64(k) * _U64(P) + i) * _F32(0.1)


def commit_bench_theta(seed: int, P: int, idx=None) -> np.ndarray:
    """Initial central variable of the commit workload: float32 normal number i."""
    key = stream_key(seed, STREAM_COMMIT_THETA)
    i = np.arange(P, dtype=_U64) if idx is None else np.asarray(idx, dtype=_U64)
    return normal_f32(key, i)


class SyntheticDataset:
    """The seeded dataset of one workload: X rows and teacher labels on demand.

    Rows are generated shard by shard (rows [k S, (k+1) S)) and cached.
    """

    def __init__(self, seed: int, d0: int, n_samples: int, dist: int,
                 teacher_dims, shard: int):
        self.seed, self.d0, self.n_samples, self.dist = seed, int(d0), int(n_samples), dist
        self.shard = int(shard)
        self.teacher = teacher_params(seed, teacher_dims)
        self._cache = {}

    def _shard(self, k: int):
        if k not in self._cache:
            rows = np.arange(k * self.shard, (k + 1) * self.shard, dtype=np.int64)
            X = make_inputs_x(self.seed, self.d0, rows, self.dist)
            self._cache[k] = (X, teacher_labels(X, self.teacher, self.dist))
        return self._cache[k]

    def __call__(self, rows):
        rows = np.asarray(rows, dtype=np.int64)
        k = int(rows[0]) // self.shard
        if np.any(rows // self.shard != k):
            X = make_inputs_x(self.seed, self.d0, rows, self.dist)
            return X, teacher_labels(X, self.teacher, self.dist)
        X, y = self._shard(k)
        local = rows - k * self.shard
        return X[local], y[local]

    def all_rows(self):
        rows = np.arange(self.n_samples, dtype=np.int64)
        X = make_inputs_x(self.seed, self.d0, rows, self.dist)
        return X, teacher_labels(X, self.teacher, self.dist)


def workload_dataset(w, seed: int = DEFAULT_SEED) -> SyntheticDataset:
    return SyntheticDataset(seed, w.dims[0], w.n_samples, w.dist, w.teacher_dims, w.shard)


def workload_schedule(w, seed: int = DEFAULT_SEED, n_commits=None):
    return make_schedule(w.n, w.commits if n_commits is None else n_commits,
                         w.tau_lo, w.tau_hi, seed)
