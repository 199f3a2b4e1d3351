"""Parity of the CUDA path with the CPU oracle, through the C ABI.

fp32 mode: ||theta~_gpu - theta~_oracle||_2 / ||theta~_oracle||_2 <= 1e-5 after
each checked commit and <= 1e-4 after the whole run (the oracle runs in fp64).
bf16 mode: every per-commit loss within 2e-2 of the fp32 oracle's.
"""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu

REL_STEP = 1e-5
REL_FINAL = 1e-4
LOSS_BF16 = 2e-2


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _rel(a, b):
    return float(np.linalg.norm(a.astype(np.float64) - b) / np.linalg.norm(b))


def _dataset(dims, N, n, seed, dist=I.DIST_UNIFORM, tdims=None):
    tdims = tdims or (dims[0], 64, dims[-1])
    return I.SyntheticDataset(seed, dims[0], N, dist, tdims, N // n)


def _oracle_snapshots(dims, n, lam, eta, m, N, seed, w, tau, upto, snap, normalize=True,
                      dist=I.DIST_UNIFORM, tdims=None, dtype=np.float64):
    ds = _dataset(dims, N, n, seed, dist, tdims)
    th0 = I.init_params(seed, dims)
    return O.agn_run(O.MLP(dims, dtype), th0, n, lam, eta, w[:upto], tau[:upto], ds, m, N // n,
                     normalize=normalize, snapshot_at=snap, dtype=dtype)


def _run_in_steps(h, w, tau, bounds):
    """Run commits [b_i, b_{i+1}) per call, giving the rest of the schedule as look-ahead."""
    out = {}
    for a, b in zip(bounds[:-1], bounds[1:]):
        h.run(b - a, w[a:], tau[a:])
        out[b - 1] = h.central()
    return out


def test_small_workload_every_commit(agn):
    """n=4, lambda=5, 784-128-10 fp32, m=32, 2048 samples, tau in {0,1,2}, 50 commits."""
    wl = WL.SMALL
    seed = I.DEFAULT_SEED
    w, tau = I.make_schedule(wl.n, wl.commits + wl.n, wl.tau_lo, wl.tau_hi, seed)
    ref = _oracle_snapshots(wl.dims, wl.n, wl.lam, wl.eta, wl.batch, wl.n_samples, seed, w, tau,
                            wl.commits, range(wl.commits))
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        got = _run_in_steps(h, w, tau, list(range(wl.commits + 1)))
        loss = h.loss()
        dn = h.delta_norm()
    errs = [_rel(got[c], ref.snapshots[c]) for c in range(wl.commits)]
    assert max(errs) <= REL_STEP, max(errs)
    assert errs[-1] <= REL_FINAL
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)
    assert np.allclose(dn, ref.delta_norm, rtol=1e-4)


def test_wave_grouping_does_not_change_results(agn):
    """One call over all commits (large waves) equals one call per commit (waves of one)."""
    wl = WL.SMALL
    seed = 11
    w, tau = I.make_schedule(wl.n, 30 + wl.n, 0, 3, seed)
    res = []
    for bounds in ([0, 30], list(range(31)), [0, 7, 8, 19, 30]):
        with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                     gemm=agn.AGN_GEMM_SIMT) as h:
            _run_in_steps(h, w, tau, bounds)
            res.append((h.central(), h.loss(), h.delta_norm()))
    for r in res[1:]:
        assert np.array_equal(r[0], res[0][0])
        assert np.array_equal(r[1], res[0][1])
        assert np.array_equal(r[2], res[0][2])


@pytest.mark.parametrize("case", ["downpour", "unnormalised", "round_robin", "ragged"])
def test_schedule_variants(agn, case):
    seed = 3
    dims, n, lam, eta, m, N, C, lo, hi, norm = (40, 72, 10), 5, 4, 0.05, 12, 400, 24, 0, 4, 1
    if case == "downpour":          # lambda = 1: AGN reduces to DOWNPOUR (Section 2)
        lam = 1
    elif case == "unnormalised":    # accumulated-gradient DOWNPOUR ablation (Fig. 3)
        norm = 0
    elif case == "round_robin":     # homogeneous cluster, tau = n - 1 (Fig. 1)
        lo = hi = n - 1
    elif case == "ragged":          # sizes that leave partial tiles everywhere; N mod n != 0
        dims, m, N = (37, 65, 13, 7), 9, 403
    w, tau = I.make_schedule(n, C + n, lo, hi, seed)
    ref = _oracle_snapshots(dims, n, lam, eta, m, N, seed, w, tau, C, range(C), normalize=bool(norm))
    with agn.AGN(dims, n, lam, eta, seed, batch=m, n_samples=N, normalize=norm,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        got = _run_in_steps(h, w, tau, [0, 5, 6, 13, C])
        loss = h.loss()
    for c, th in got.items():
        assert _rel(th, ref.snapshots[c]) <= REL_STEP
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)


def test_builtin_schedule_matches_explicit(agn):
    seed, dims, n = 21, (16, 12, 4), 3
    with agn.AGN(dims, n, 2, 0.1, seed, batch=4, n_samples=60, tau_lo=0, tau_hi=2,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        h.run(7)
        h.run(5)
        a = h.central()
    w, tau = I.make_schedule(n, 12 + n, 0, 2, seed)
    with agn.AGN(dims, n, 2, 0.1, seed, batch=4, n_samples=60, gemm=agn.AGN_GEMM_SIMT) as h:
        h.run(12, w, tau)
        b = h.central()
    assert np.array_equal(a, b)


def test_infeasible_schedule_is_rejected(agn):
    with agn.AGN((16, 8, 4), 2, 2, 0.1, 1, batch=4, n_samples=40,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        before = h.central()
        with pytest.raises(agn.AGNError) as e:
            h.run(2, [0, 0], [0, 1])          # worker 0 would read version 0 twice
        assert e.value.code == agn.AGN_E_SCHEDULE
        with pytest.raises(agn.AGNError) as e:
            h.run(1, [5], [0])
        assert e.value.code == agn.AGN_E_SCHEDULE
        assert h.num_commits == 0 and np.array_equal(h.central(), before)
        # a version that passed without a pull cannot be read later
        h.run(2, [0, 1], [0, 0])              # no look-ahead: worker 0's next pull unknown
        with pytest.raises(agn.AGNError) as e:
            h.run(1, [0], [1])                # would read version 1, already passed
        assert e.value.code == agn.AGN_E_SCHEDULE
        h.run(1, [0], [0])                    # version 2 is current: pulled at the start
        assert h.num_commits == 3


def test_divergence_is_reported_as_nonfinite(agn):
    """A huge learning rate makes the loss overflow; the run completes and says so."""
    with agn.AGN((16, 32, 4), 2, 3, 1e30, 1, batch=8, n_samples=64, normalize=0,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        with pytest.raises(agn.AGNError) as e:
            h.run(6, [0, 1] * 4, [0] * 8)
        assert e.value.code == agn.AGN_E_NONFINITE
        assert h.num_commits == 6
        assert not np.all(np.isfinite(h.loss()))


def test_inputs_match_generator(agn):
    wl = WL.SMALL
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, I.DEFAULT_SEED, batch=wl.batch,
                 n_samples=wl.n_samples) as h:
        x, y, th = h.export_inputs()
    ds = I.workload_dataset(wl)
    X, Y = ds.all_rows()
    assert np.array_equal(x, X) and np.array_equal(y, Y)
    assert np.array_equal(th, I.init_params(I.DEFAULT_SEED, wl.dims))


def test_mnist_shaped_workload_full_size_prefix(agn):
    """n=16, lambda=15, 784-1000-1000-10 fp32, m=128, 60k samples, staleness up to 15:
    every one of the first 32 commits at full size within 1e-5.  (Float32
    arithmetic itself leaves 1e-5 of the float64 trajectory near commit 40:
    the oracle run in float32 is 1.02e-5 away at commit 40.)"""
    wl = WL.MNIST_SHAPED
    seed = I.DEFAULT_SEED
    C = 32
    w, tau = I.make_schedule(wl.n, wl.commits, wl.tau_lo, wl.tau_hi, seed)
    ref = _oracle_snapshots(wl.dims, wl.n, wl.lam, wl.eta, wl.batch, wl.n_samples, seed, w, tau,
                            C, range(C))
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        got = _run_in_steps(h, w, tau, list(range(0, C + 1, 4)))
        loss = h.loss()
    for c, th in got.items():
        assert _rel(th, ref.snapshots[c]) <= REL_STEP, c
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)


@pytest.mark.parametrize("gemm", ["simt"])
def test_bf16_loss_within_tolerance(agn, gemm):
    """bf16 operands / fp32 master on a mid-size net: per-commit loss within 2e-2."""
    seed = 5
    dims, n, lam, eta, m, N, C = (256, 512, 256, 10), 8, 5, 0.05, 64, 4096, 40
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)
    ref = _oracle_snapshots(dims, n, lam, eta, m, N, seed, w, tau, C, (), dtype=np.float32)
    with agn.AGN(dims, n, lam, eta, seed, batch=m, n_samples=N, precision=agn.AGN_PREC_BF16,
                 gemm=agn.AGN_GEMM_SIMT) as h:
        h.run(C, w, tau)
        loss = h.loss()
    assert np.max(np.abs(loss - ref.loss)) <= LOSS_BF16


# ----------------------------------------------------------------------------
# tcgen05 (bf16) GEMMs against the CUDA-core bf16 kernels on the same inputs
# ----------------------------------------------------------------------------

def _bf16_run(agn, dims, m, gemm, tc_mask=0, n=4, lam=2, C=4, N=None, seed=9):
    N = N or n * 3 * m
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)
    with agn.AGN(dims, n, lam, 0.05, seed, batch=m, n_samples=N, precision=agn.AGN_PREC_BF16,
                 gemm=gemm, tc_mask=tc_mask) as h:
        th0 = h.central()
        h.run(C, w, tau)
        return th0, h.central(), h.loss(), h.last_run_stats()


@pytest.mark.parametrize("dims,m", [((256, 512, 384, 10), 64),
                                    ((784, 200, 10), 128),
                                    ((192, 256, 256, 10), 256)])
@pytest.mark.parametrize("mask", [1, 2, 4, 7])
def test_tcgen05_gemms_match_cuda_core_bf16(agn, dims, m, mask):
    """Each GEMM kind alone (mask bit) and all together, on shapes with ragged
    tiles: the update theta~ - theta~0 agrees with the CUDA-core bf16 kernels
    up to bf16 rounding-order differences."""
    if mask == 2 and len(dims) < 4:
        pytest.skip("dX of a hidden layer needs two hidden layers")
    th0, a, la, _ = _bf16_run(agn, dims, m, agn.AGN_GEMM_SIMT)
    th0b, b, lb, _ = _bf16_run(agn, dims, m, agn.AGN_GEMM_TCGEN05, tc_mask=mask)
    assert np.array_equal(th0, th0b)
    da, db = a - th0, b - th0
    err = np.linalg.norm(db - da) / np.linalg.norm(da)
    assert err < 2e-2, err
    assert np.max(np.abs(la - lb)) < 5e-3
