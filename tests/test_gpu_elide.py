"""Accumulator elision: the workers keep no gradient accumulator and a commit
adds (theta_k - theta_pull) scaled by 1/lambda (1/(tau+1), 1), the pulled
parameters kept as a snapshot.  Against the oracle run the same way: fp32
theta~ within 1e-5 (relative L2) after every commit, bf16 loss within 2e-2.
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


def _oracle(dims, n, lam, eta, m, N, seed, w, tau, C, dtype=np.float64, **kw):
    ds = I.SyntheticDataset(seed, dims[0], N, I.DIST_UNIFORM, (dims[0], 64, dims[-1]), N // n)
    return O.agn_run(O.MLP(dims, dtype), I.init_params(seed, dims), n, lam, eta, w[:C], tau[:C],
                     ds, m, N // n, snapshot_at=range(C), dtype=dtype, elide_accumulator=True,
                     **kw)


@pytest.mark.parametrize("gemm", ["tcgen05", "simt"])
@pytest.mark.parametrize("rule", ["agn", "unnormalised", "dynsgd"])
def test_elided_every_commit_fp32(agn, gemm, rule):
    wl = WL.SMALL
    seed, C = I.DEFAULT_SEED, 30
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    kw = dict(normalize=rule != "unnormalised", staleness_scaled=rule == "dynsgd")
    ref = _oracle(wl.dims, wl.n, wl.lam, wl.eta, wl.batch, wl.n_samples, seed, w, tau, C, **kw)
    got = {}
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 gemm=agn.AGN_GEMM_TCGEN05 if gemm == "tcgen05" else agn.AGN_GEMM_SIMT,
                 normalize=int(rule != "unnormalised"),
                 commit_rule=agn.AGN_COMMIT_DYNSGD if rule == "dynsgd" else agn.AGN_COMMIT_AGN,
                 elide_accumulator=1) as h:
        for c in range(C):
            h.run(1, w[c:], tau[c:])
            got[c] = h.central()
        loss, dn = h.loss(), h.delta_norm()
    errs = [_rel(got[c], ref.snapshots[c]) for c in range(C)]
    assert max(errs) <= REL_STEP, (int(np.argmax(errs)), max(errs))
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)
    assert np.allclose(dn, ref.delta_norm, rtol=1e-3)


def test_elided_mnist_shaped_prefix_fp32(agn):
    """The 16-worker 784-1000-1000-10 workload at full size, first 32 commits."""
    wl = WL.MNIST_SHAPED
    seed, C = I.DEFAULT_SEED, 32
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    ds = I.workload_dataset(wl, seed)
    ref = O.agn_run(O.MLP(wl.dims), I.init_params(seed, wl.dims), wl.n, wl.lam, wl.eta, w[:C],
                    tau[:C], ds, wl.batch, wl.shard, snapshot_at=(C - 1,),
                    elide_accumulator=True)
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 input_dist=wl.dist, teacher_dims=wl.teacher_dims, elide_accumulator=1) as h:
        h.run(C, w, tau)
        got = h.central()
    assert _rel(got, ref.snapshots[C - 1]) <= REL_STEP


def test_elided_bf16_loss(agn):
    dims, n, lam, m, seed, C = (784, 1024, 1024, 10), 4, 10, 64, 5, 12
    N = n * 6 * m
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)
    ref = _oracle(dims, n, lam, 0.01, m, N, seed, w, tau, C, dtype=np.float32)
    with agn.AGN(dims, n, lam, 0.01, seed, precision=agn.AGN_PREC_BF16, batch=m, n_samples=N,
                 gemm=agn.AGN_GEMM_TCGEN05, elide_accumulator=1) as h:
        h.run(C, w, tau)
        loss = h.loss()
    assert np.max(np.abs(loss - ref.loss)) <= LOSS_BF16
