"""Adam as the local optimizer: the dW kernels store the raw gradients and a
streaming kernel takes Adam's step (moments per worker, persisting across
commits).  Against the oracle run the same way: fp32 theta~ within 1e-5
(relative L2) after every commit, bf16 loss within 2e-2.
"""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu

REL_STEP = 1e-5
LOSS_BF16 = 2e-2
ETA = 1e-3


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _rel(a, b):
    return float(np.linalg.norm(a.astype(np.float64) - b) / np.linalg.norm(b))


def _oracle(dims, n, lam, eta, m, N, seed, w, tau, C, dtype=np.float64, **kw):
    ds = I.SyntheticDataset(seed, dims[0], N, I.DIST_UNIFORM, (dims[0], 64, dims[-1]), N // n)
    return O.agn_run(O.MLP(dims, dtype), I.init_params(seed, dims), n, lam, eta, w[:C], tau[:C],
                     ds, m, N // n, snapshot_at=range(C), dtype=dtype, optimizer="adam", **kw)


@pytest.mark.parametrize("gemm", ["tcgen05", "simt"])
@pytest.mark.parametrize("elide", [0, 1])
def test_adam_every_commit_fp32(agn, gemm, elide):
    wl = WL.SMALL
    seed, C = I.DEFAULT_SEED, 30
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    ref = _oracle(wl.dims, wl.n, wl.lam, ETA, wl.batch, wl.n_samples, seed, w, tau, C,
                  elide_accumulator=bool(elide))
    got = {}
    with agn.AGN(wl.dims, wl.n, wl.lam, ETA, seed, batch=wl.batch, n_samples=wl.n_samples,
                 gemm=agn.AGN_GEMM_TCGEN05 if gemm == "tcgen05" else agn.AGN_GEMM_SIMT,
                 local_optimizer=agn.AGN_OPT_ADAM, elide_accumulator=elide) as h:
        for c in range(C):
            h.run(1, w[c:], tau[c:])
            got[c] = h.central()
        loss = h.loss()
    errs = [_rel(got[c], ref.snapshots[c]) for c in range(C)]
    assert max(errs) <= REL_STEP, (int(np.argmax(errs)), max(errs))
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)


def test_adam_dynsgd_fp32(agn):
    wl = WL.SMALL
    seed, C = I.DEFAULT_SEED, 16
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    ref = _oracle(wl.dims, wl.n, wl.lam, ETA, wl.batch, wl.n_samples, seed, w, tau, C,
                  staleness_scaled=True)
    with agn.AGN(wl.dims, wl.n, wl.lam, ETA, seed, batch=wl.batch, n_samples=wl.n_samples,
                 local_optimizer=agn.AGN_OPT_ADAM, commit_rule=agn.AGN_COMMIT_DYNSGD) as h:
        h.run(C, w, tau)
        got = h.central()
    assert _rel(got, ref.snapshots[C - 1]) <= REL_STEP


def test_adam_bf16_loss(agn):
    dims, n, lam, m, seed, C = (784, 1024, 1024, 10), 4, 10, 64, 5, 12
    N = n * 6 * m
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)
    ref = _oracle(dims, n, lam, ETA, m, N, seed, w, tau, C, dtype=np.float32)
    with agn.AGN(dims, n, lam, ETA, seed, precision=agn.AGN_PREC_BF16, batch=m, n_samples=N,
                 gemm=agn.AGN_GEMM_TCGEN05, local_optimizer=agn.AGN_OPT_ADAM) as h:
        h.run(C, w, tau)
        loss = h.loss()
    assert np.max(np.abs(loss - ref.loss)) <= LOSS_BF16
