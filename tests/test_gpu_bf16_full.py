"""bf16 mode (tcgen05 bf16 GEMMs, fp32 master replicas and accumulators)
against the float32 oracle: every per-commit loss within 2e-2.

At full size, the first commits of the 32-worker 3072-2048x3-10 workload and
of the 64-worker 784-4096-4096-10 workload, past the first wave so that
later commits read versions that earlier commits created.  The lambda sweep
{1, 5, 10, 20, 40} and the un-normalised ablation run on a narrower net of
the same shape family.
"""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu

LOSS_BF16 = 2e-2


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _oracle_loss(dims, n, lam, eta, m, N, dist, tdims, seed, w, tau, C, normalize=True):
    ds = I.SyntheticDataset(seed, dims[0], N, dist, tdims, N // n)
    r = O.agn_run(O.MLP(dims, np.float32), I.init_params(seed, dims), n, lam, eta, w[:C], tau[:C],
                  ds, m, N // n, normalize=normalize, dtype=np.float32)
    return r.loss


def _gpu_loss(agn, dims, n, lam, eta, m, N, dist, tdims, seed, w, tau, C, normalize=1):
    with agn.AGN(dims, n, lam, eta, seed, precision=agn.AGN_PREC_BF16, batch=m, n_samples=N,
                 input_dist=dist, teacher_dims=tdims, normalize=normalize,
                 gemm=agn.AGN_GEMM_TCGEN05) as h:
        h.run(C, w, tau)
        return h.loss()


@pytest.mark.parametrize("wl,C", [(WL.WIDE_BF16, 40), (WL.LARGE_BF16, 70)],
                         ids=["wide_3072x2048x3", "large_784x4096x2"])
def test_bf16_full_size_prefix(agn, wl, C):
    seed = I.DEFAULT_SEED
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    ref = _oracle_loss(wl.dims, wl.n, wl.lam, wl.eta, wl.batch, wl.n_samples, wl.dist,
                       wl.teacher_dims, seed, w, tau, C)
    got = _gpu_loss(agn, wl.dims, wl.n, wl.lam, wl.eta, wl.batch, wl.n_samples, wl.dist,
                    wl.teacher_dims, seed, w, tau, C)
    err = np.abs(got - ref)
    assert np.max(err) <= LOSS_BF16, (int(np.argmax(err)), float(np.max(err)))


@pytest.mark.parametrize("lam", [1, 5, 10, 20, 40])
@pytest.mark.parametrize("normalize", [1, 0])
def test_bf16_lambda_sweep_and_ablation(agn, lam, normalize):
    """The large workload's lambda sweep and un-normalised ablation (Fig. 3) on
    784-1024-1024-10, n = 4, m = 64, tau = n - 1, 12 commits."""
    if normalize == 0 and lam == 1:
        pytest.skip("lambda = 1: normalised and un-normalised commits coincide")
    dims, n, m, seed, C = (784, 1024, 1024, 10), 4, 64, 5, 12
    N = n * 6 * m
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)
    tdims = (784, 64, 10)
    ref = _oracle_loss(dims, n, lam, 0.01, m, N, I.DIST_UNIFORM, tdims, seed, w, tau, C,
                       normalize=bool(normalize))
    got = _gpu_loss(agn, dims, n, lam, 0.01, m, N, I.DIST_UNIFORM, tdims, seed, w, tau, C,
                    normalize=normalize)
    finite = np.isfinite(ref)
    assert np.max(np.abs(got[finite] - ref[finite])) <= LOSS_BF16
