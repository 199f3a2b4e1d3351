"""The DynSGD-style commit rule (Section 4's comparison): commit c adds the
worker's accumulated update divided by tau_c + 1 instead of by lambda.

Same bars as the AGN rule: fp32 theta~ within 1e-5 (relative L2) of the
float64 oracle after every commit; bf16 per-commit loss within 2e-2 of the
float32 oracle.
"""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu

REL_STEP = 1e-5
LOSS_BF16 = 2e-2


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _rel(a, b):
    return float(np.linalg.norm(a.astype(np.float64) - b) / np.linalg.norm(b))


def _oracle(dims, n, lam, eta, m, N, seed, w, tau, C, dtype=np.float64):
    ds = I.SyntheticDataset(seed, dims[0], N, I.DIST_UNIFORM, (dims[0], 64, dims[-1]), N // n)
    return O.agn_run(O.MLP(dims, dtype), I.init_params(seed, dims), n, lam, eta, w[:C], tau[:C],
                     ds, m, N // n, snapshot_at=range(C), dtype=dtype, staleness_scaled=True)


@pytest.mark.parametrize("gemm", ["tcgen05", "simt"])
@pytest.mark.parametrize("lam", [5, 1])
def test_dynsgd_every_commit_fp32(agn, gemm, lam):
    """784-128-10, n = 4, m = 32, tau drawn from {0, 1, 2}; lambda = 1 is the
    staleness-scaled first-order (DOWNPOUR-style) rule."""
    wl = WL.SMALL
    seed, C = I.DEFAULT_SEED, 30
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    assert len(set(tau[:C])) > 1          # the scale really varies per commit
    ref = _oracle(wl.dims, wl.n, lam, wl.eta, wl.batch, wl.n_samples, seed, w, tau, C)
    g = agn.AGN_GEMM_TCGEN05 if gemm == "tcgen05" else agn.AGN_GEMM_SIMT
    got = {}
    with agn.AGN(wl.dims, wl.n, lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 gemm=g, commit_rule=agn.AGN_COMMIT_DYNSGD) as h:
        for c in range(C):
            h.run(1, w[c:], tau[c:])
            got[c] = h.central()
        loss, dn = h.loss(), h.delta_norm()
    errs = [_rel(got[c], ref.snapshots[c]) for c in range(C)]
    assert max(errs) <= REL_STEP, (int(np.argmax(errs)), max(errs))
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)
    assert np.allclose(dn, ref.delta_norm, rtol=1e-4)


def test_dynsgd_differs_from_agn(agn):
    """The rule is wired through: with tau + 1 != lambda the runs differ."""
    wl = WL.SMALL
    seed, C = I.DEFAULT_SEED, 8
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    out = []
    for rule in (agn.AGN_COMMIT_AGN, agn.AGN_COMMIT_DYNSGD):
        with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch,
                     n_samples=wl.n_samples, commit_rule=rule) as h:
            h.run(C, w, tau)
            out.append(h.central())
    assert _rel(out[0], out[1].astype(np.float64)) > 1e-3


def test_dynsgd_bf16_loss(agn):
    dims, n, lam, m, seed, C = (784, 256, 256, 10), 4, 5, 64, 11, 24
    N = n * 4 * m
    w, tau = I.make_schedule(n, C + n, 0, n - 1, seed)
    ref = _oracle(dims, n, lam, 0.05, m, N, seed, w, tau, C, dtype=np.float32)
    with agn.AGN(dims, n, lam, 0.05, seed, precision=agn.AGN_PREC_BF16, batch=m, n_samples=N,
                 gemm=agn.AGN_GEMM_TCGEN05, commit_rule=agn.AGN_COMMIT_DYNSGD) as h:
        h.run(C, w, tau)
        loss = h.loss()
    assert np.max(np.abs(loss - ref.loss)) <= LOSS_BF16
