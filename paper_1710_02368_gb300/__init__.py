"""GB300 implementation of the hot path of Accumulated Gradient Normalization
(Hermans, Spanakis & Moeckel, ACML 2017).

A thin Python binding of the C ABI in include/agn.h: the functions below carry
the C names and only marshal arguments (numpy host arrays, device pointers
given as ints or tensors with `data_ptr()`).  Every step of the path runs in
the library's CUDA kernels; without the built library the calls raise.
"""

from __future__ import annotations

import ctypes as C

import numpy as np

from . import _lib
from ._lib import (AGN_COMMIT_AGN, AGN_COMMIT_DYNSGD, AGN_OPT_ADAM, AGN_OPT_SGD,  # noqa: F401
                   AGN_DIST_NORMAL, AGN_DIST_UNIFORM, AGN_GEMM_AUTO, AGN_GEMM_SIMT,  # noqa: F401
                   AGN_GEMM_TCGEN05, AGN_PREC_BF16, AGN_PREC_FP32, AGN_OK, AGN_E_INVALID,
                   AGN_E_SCHEDULE, AGN_E_OOM, AGN_E_CUDA, AGN_E_TIMEOUT, AGN_E_NONFINITE,
                   AGN_E_UNSUPPORTED, AGN_E_BOUNDS, agn_options)

__all__ = [
    "AGNError", "AGN", "agn_default_options", "agn_create", "agn_run", "agn_central",
    "agn_replica", "agn_loss", "agn_delta_norm", "agn_num_params", "agn_num_commits",
    "agn_last_run_stats", "agn_profile", "agn_kernel_stats", "agn_generate_inputs", "agn_export_inputs", "agn_last_error",
    "agn_destroy", "agn_make_schedule", "agn_plan_waves", "agn_commit_pull",
    "agn_commit_pull_noalloc",
    "agn_fill_commit_inputs", "agn_debug_waits",
    "library_path",
]


class AGNError(RuntimeError):
    def __init__(self, code: int, msg: str):
        self.code = code
        self.name = _lib.ERROR_NAMES.get(code, str(code))
        super().__init__(f"{self.name}: {msg}")


def library_path() -> str:
    return _lib.library_file()


def _L():
    return _lib.load()


def _check(rc: int, handle=None):
    if rc != AGN_OK:
        msg = _L().agn_last_error(handle)
        raise AGNError(rc, msg.decode() if msg else "")


def _i32(a):
    a = np.ascontiguousarray(a, dtype=np.int32)
    return a, a.ctypes.data_as(_lib._I32P)


def _ptr(x):
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return C.c_void_p(x.data_ptr())
    return C.c_void_p(int(x))


def agn_default_options() -> agn_options:
    o = agn_options()
    _L().agn_default_options(C.byref(o))
    return o


def agn_create(dims, n_workers, lam, eta, seed, options: agn_options | None = None,
               keep=None):
    """Returns an opaque handle (c_void_p).  `keep` collects arrays that the
    options point to, so that they outlive the call."""
    d, dp = _i32(dims)
    h = C.c_void_p()
    rc = _L().agn_create(dp, len(d), int(n_workers), int(lam), float(eta), int(seed),
                         C.byref(options) if options is not None else None, C.byref(h))
    _check(rc, None)
    return h


def agn_run(h, n_commits, worker=None, staleness=None):
    if worker is None and staleness is None:
        _check(_L().agn_run(h, int(n_commits), None, None, 0), h)
        return
    w, wp = _i32(worker)
    t, tp = _i32(staleness)
    if len(w) != len(t):
        raise ValueError("worker and staleness differ in length")
    _check(_L().agn_run(h, int(n_commits), wp, tp, len(w)), h)


def _read_params(fn, h, *extra):
    P = _L().agn_num_params(h)
    out = np.empty(P, dtype=np.float32)
    _check(fn(h, *extra, out.ctypes.data_as(_lib._F32P), P), h)
    return out


def agn_central(h) -> np.ndarray:
    return _read_params(_L().agn_central, h)


def agn_replica(h, k) -> np.ndarray:
    return _read_params(_L().agn_replica, h, int(k))


def _read_commits(fn, h):
    C_ = _L().agn_num_commits(h)
    out = np.empty(max(C_, 0), dtype=np.float32)
    _check(fn(h, out.ctypes.data_as(_lib._F32P), len(out)), h)
    return out


def agn_loss(h) -> np.ndarray:
    return _read_commits(_L().agn_loss, h)


def agn_delta_norm(h) -> np.ndarray:
    return _read_commits(_L().agn_delta_norm, h)


def agn_evaluate(h, pred=None):
    """(loss, accuracy) of theta~ on the handle's held-out set; `pred`, an int32
    array of n_eval entries, also receives the predictions."""
    loss, acc = C.c_float(), C.c_float()
    pp, cap = None, 0
    if pred is not None:
        if pred.dtype != np.int32 or not pred.flags.c_contiguous:
            raise ValueError("pred must be a contiguous int32 array")
        pp, cap = pred.ctypes.data_as(_lib._I32P), len(pred)
    _check(_L().agn_evaluate(h, C.byref(loss), C.byref(acc), pp, cap), h)
    return loss.value, acc.value


def agn_temporal_efficiency(ta, fa, tb, fb) -> float:
    """Eq. 4 on two sampled curves (times non-decreasing, >= 0)."""
    arrs = [np.ascontiguousarray(x, dtype=np.float64) for x in (ta, fa, tb, fb)]
    if arrs[0].shape != arrs[1].shape or arrs[2].shape != arrs[3].shape:
        raise ValueError("each curve needs as many values as times")
    out = C.c_double()
    p = [a.ctypes.data_as(_lib._F64P) for a in arrs]
    _check(_L().agn_temporal_efficiency(p[0], p[1], len(arrs[0]), p[2], p[3], len(arrs[2]),
                                        C.byref(out)))
    return out.value


def agn_num_params(h) -> int:
    return int(_L().agn_num_params(h))


def agn_num_commits(h) -> int:
    return int(_L().agn_num_commits(h))


def agn_last_run_stats(h) -> dict:
    out = (C.c_double * 5)()
    _check(_L().agn_last_run_stats(h, out, 5), h)
    return {"waves": out[0], "launches": out[1], "gpu_ms": out[2], "worker_steps": out[3],
            "host_ms": out[4]}


def agn_profile(h, mode):
    _check(_L().agn_profile(h, int(mode)), h)


def agn_kernel_stats(h) -> dict:
    n = len(_lib.KERNEL_CLASSES)
    out = (C.c_double * (4 * n))()
    _check(_L().agn_kernel_stats(h, out, 4 * n), h)
    return {name: {"launches": out[4 * i], "ms": out[4 * i + 1], "flops": out[4 * i + 2],
                   "bytes": out[4 * i + 3]} for i, name in enumerate(_lib.KERNEL_CLASSES)}


def agn_generate_inputs(dims, input_dist, seed, row0, n_rows, teacher_dims=None,
                        want_x=True, want_y=True, want_theta=True):
    d, dp = _i32(dims)
    td, tdp = (None, None) if teacher_dims is None else _i32(teacher_dims)
    x = np.empty((n_rows, d[0]), dtype=np.float32) if want_x else None
    y = np.empty(n_rows, dtype=np.int32) if want_y else None
    P = sum(int(d[l]) * int(d[l - 1]) + int(d[l]) for l in range(1, len(d)))
    th = np.empty(P, dtype=np.float32) if want_theta else None
    rc = _L().agn_generate_inputs(
        dp, len(d), int(input_dist), tdp, 0 if td is None else len(td), int(seed), int(row0),
        int(n_rows), None if x is None else x.ctypes.data_as(_lib._F32P),
        None if y is None else y.ctypes.data_as(_lib._I32P),
        None if th is None else th.ctypes.data_as(_lib._F32P))
    _check(rc, None)
    return x, y, th


def agn_export_inputs(h, n_samples, d0):
    x = np.empty((n_samples, d0), dtype=np.float32)
    y = np.empty(n_samples, dtype=np.int32)
    th = np.empty(agn_num_params(h), dtype=np.float32)
    _check(_L().agn_export_inputs(h, x.ctypes.data_as(_lib._F32P), y.ctypes.data_as(_lib._I32P),
                                  th.ctypes.data_as(_lib._F32P)), h)
    return x, y, th


def agn_last_error(h=None) -> str:
    m = _L().agn_last_error(h)
    return m.decode() if m else ""


def agn_destroy(h):
    if h:
        _L().agn_destroy(h)


def agn_make_schedule(n, n_commits, tau_lo, tau_hi, seed):
    w = np.empty(n_commits, dtype=np.int32)
    t = np.empty(n_commits, dtype=np.int32)
    _check(_L().agn_make_schedule(int(n), int(n_commits), int(tau_lo), int(tau_hi), int(seed),
                                  w.ctypes.data_as(_lib._I32P), t.ctypes.data_as(_lib._I32P)))
    return w, t


def agn_plan_waves(n, lam, n_commits, worker, staleness):
    """The wave plan agn_run follows on a fresh handle (host only): returns
    (wave_slots, wave_end, slot_commit, slot_t0, pulls) with pulls an [n_pulls, 2]
    array of (version, worker) in order."""
    w, wp = _i32(worker)
    t, tp = _i32(staleness)
    k = int(n_commits)
    cap = max(1, k)
    ws = np.empty(cap, dtype=np.int32)
    we = np.empty(cap, dtype=np.int32)
    sc = np.empty(cap, dtype=np.int32)
    st = np.empty(cap, dtype=np.int64)
    pcap = len(w) + int(n) + 1
    pv = np.empty(pcap, dtype=np.int32)
    pw = np.empty(pcap, dtype=np.int32)
    nw = C.c_int32(0)
    npl = C.c_int64(0)
    _check(_L().agn_plan_waves(int(n), int(lam), k, wp, tp, len(w), C.byref(nw),
                               ws.ctypes.data_as(_lib._I32P), we.ctypes.data_as(_lib._I32P),
                               sc.ctypes.data_as(_lib._I32P), st.ctypes.data_as(_lib._I64P),
                               pcap, pv.ctypes.data_as(_lib._I32P),
                               pw.ctypes.data_as(_lib._I32P), C.byref(npl)))
    nwv, npv = nw.value, npl.value
    return (ws[:nwv].copy(), we[:nwv].copy(), sc[:k].copy(), st[:k].copy(),
            np.stack([pv[:npv], pw[:npv]], axis=1))


def agn_commit_pull(theta_c, acc, replicas, replicas_bf16, P, ld, n, commit_worker,
                    pull_offsets, pull_workers, eta, lam, normalize=1, delta_norm=None,
                    stream=None):
    cw, cwp = _i32(commit_worker)
    po, pop = _i32(pull_offsets)
    pw, pwp = _i32(pull_workers if len(pull_workers) else [0])
    _check(_L().agn_commit_pull(_ptr(theta_c), _ptr(acc), _ptr(replicas), _ptr(replicas_bf16),
                                int(P), int(ld), int(n), len(cw), cwp, pop, pwp, float(eta),
                                int(lam), int(normalize), _ptr(delta_norm), _ptr(stream)))


def agn_commit_pull_noalloc(theta_c, acc, replicas, replicas_bf16, P, ld, n, commit_worker,
                            pull_offsets, pull_workers, eta, lam, normalize=1, delta_norm=None,
                            stream=None):
    """agn_commit_pull without any device allocation (scratch in a fixed
    device array); for callers that may not allocate on this path."""
    cw, cwp = _i32(commit_worker)
    po, pop = _i32(pull_offsets)
    pw, pwp = _i32(pull_workers if len(pull_workers) else [0])
    _check(_L().agn_commit_pull_noalloc(
        _ptr(theta_c), _ptr(acc), _ptr(replicas), _ptr(replicas_bf16), int(P), int(ld), int(n),
        len(cw), cwp, pop, pwp, float(eta), int(lam), int(normalize), _ptr(delta_norm),
        _ptr(stream)))


def agn_debug_waits(h, wait_ns, withhold_rank=-1):
    """Test hook: bound the device waits of later runs by wait_ns (0 = 2 s) and
    make one split-K rank withhold its arrival (-1 = none)."""
    _check(_L().agn_debug_waits(h, int(wait_ns), int(withhold_rank)), h)


def agn_fill_commit_inputs(theta_c, acc, replicas, P, ld, n, seed, stream=None):
    _check(_L().agn_fill_commit_inputs(_ptr(theta_c), _ptr(acc), _ptr(replicas), int(P), int(ld),
                                       int(n), int(seed), _ptr(stream)))


class AGN:
    """Owning wrapper of one handle (the C calls above, bound to it)."""

    def __init__(self, dims, n_workers, lam, eta, seed, *, precision=AGN_PREC_FP32, batch=32,
                 n_samples=2048, input_dist=AGN_DIST_UNIFORM, teacher_dims=None, normalize=1,
                 gemm=AGN_GEMM_AUTO, tau_lo=0, tau_hi=0, stream=None, x=None, y=None,
                 theta0=None, tc_mask=0, commit_rule=AGN_COMMIT_AGN, elide_accumulator=0,
                 n_eval=0, local_optimizer=AGN_OPT_SGD, adam=(0.0, 0.0, 0.0)):
        o = agn_default_options()
        o.precision, o.batch, o.n_samples = int(precision), int(batch), int(n_samples)
        o.input_dist, o.normalize, o.gemm = int(input_dist), int(normalize), int(gemm)
        o.tau_lo, o.tau_hi = int(tau_lo), int(tau_hi)
        o.tc_mask = int(tc_mask)
        o.commit_rule = int(commit_rule)
        o.elide_accumulator = int(elide_accumulator)
        o.n_eval = int(n_eval)
        o.local_optimizer = int(local_optimizer)
        o.adam_beta1, o.adam_beta2, o.adam_eps = (float(x) for x in adam)
        self.n_eval = int(n_eval)
        keep = []
        if teacher_dims is not None:
            td, tdp = _i32(teacher_dims)
            keep.append(td)
            o.teacher_dims, o.n_teacher_dims = tdp, len(td)
        if stream is not None:
            o.stream = _ptr(stream)
        for name, arr, dt, pt in (("x_init", x, np.float32, _lib._F32P),
                                  ("y_init", y, np.int32, _lib._I32P),
                                  ("theta_init", theta0, np.float32, _lib._F32P)):
            if arr is not None:
                a = np.ascontiguousarray(arr, dtype=dt)
                keep.append(a)
                setattr(o, name, a.ctypes.data_as(pt))
        self.dims = tuple(int(v) for v in dims)
        self.n_samples = int(n_samples)
        self.h = agn_create(dims, n_workers, lam, eta, seed, o)

    def evaluate(self, with_pred=False):
        """(loss, accuracy[, predictions]) of theta~ on the held-out set."""
        if not with_pred:
            return agn_evaluate(self.h)
        pred = np.empty(self.n_eval, dtype=np.int32)
        loss, acc = agn_evaluate(self.h, pred)
        return loss, acc, pred

    def run(self, n_commits, worker=None, staleness=None):
        agn_run(self.h, n_commits, worker, staleness)

    def central(self):
        return agn_central(self.h)

    def replica(self, k):
        return agn_replica(self.h, k)

    def loss(self):
        return agn_loss(self.h)

    def delta_norm(self):
        return agn_delta_norm(self.h)

    @property
    def num_params(self):
        return agn_num_params(self.h)

    @property
    def num_commits(self):
        return agn_num_commits(self.h)

    def last_run_stats(self):
        return agn_last_run_stats(self.h)

    def profile(self, mode):
        agn_profile(self.h, mode)

    def kernel_stats(self):
        return agn_kernel_stats(self.h)

    def export_inputs(self):
        return agn_export_inputs(self.h, self.n_samples, self.dims[0])

    def close(self):
        if getattr(self, "h", None):
            agn_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()
