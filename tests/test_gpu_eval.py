"""Held-out evaluation of theta~ (agn_evaluate) and temporal efficiency (Eq. 4)
on curves measured through the C ABI.

The evaluation set is rows [N, N + n_eval) of the seeded generator with the
teacher's labels.  The library's loss and predictions are compared with the
oracle's evaluation of the same theta~ (read back through agn_central) in
float32: loss within 1e-5, predictions equal wherever the top two logits are
not within 1e-4 of each other (the argmax is then decided the same way in
either summation order), and the accuracy equal to the predictions' mean.
"""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _eval_rows(wl, seed, n_eval):
    rows = np.arange(wl.n_samples, wl.n_samples + n_eval, dtype=np.int64)
    X = I.make_inputs_x(seed, wl.dims[0], rows, wl.dist)
    return X, I.teacher_labels(X, I.teacher_params(seed, wl.teacher_dims), wl.dist)


def _check_against_oracle(dims, theta, X, y, loss, acc, pred):
    ol, oa, op = O.evaluate(O.MLP(dims, np.float32), theta, X, y, dtype=np.float32)
    # margins from float64 logits
    h = X.astype(np.float64)
    params = O.MLP(dims).unpack(theta.astype(np.float64))
    for l, (W, b) in enumerate(params):
        h = h @ W.T + b
        if l + 1 < len(params):
            h = np.maximum(h, 0)
    top2 = np.sort(h, axis=1)[:, -2:]
    clear = (top2[:, 1] - top2[:, 0]) > 1e-4
    assert clear.mean() > 0.95
    assert np.array_equal(pred[clear], op[clear])
    assert acc == pytest.approx(float(np.mean(pred == y)), abs=1e-6)
    assert loss == pytest.approx(ol, rel=1e-5)


@pytest.mark.parametrize("wl,C,gemm", [(WL.SMALL, 20, "tcgen05"), (WL.SMALL, 20, "simt"),
                                       (WL.MNIST_SHAPED, 10, "tcgen05")],
                         ids=["small-tc", "small-simt", "mnist-shaped"])
def test_evaluate_matches_oracle(agn, wl, C, gemm):
    seed, n_eval = I.DEFAULT_SEED, 5000
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    X, y = _eval_rows(wl, seed, n_eval)
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 input_dist=wl.dist, teacher_dims=wl.teacher_dims, n_eval=n_eval,
                 gemm=agn.AGN_GEMM_TCGEN05 if gemm == "tcgen05" else agn.AGN_GEMM_SIMT) as h:
        l0, a0, p0 = h.evaluate(with_pred=True)
        _check_against_oracle(wl.dims, h.central(), X, y, l0, a0, p0)
        h.run(C, w, tau)
        l1, a1, p1 = h.evaluate(with_pred=True)
        _check_against_oracle(wl.dims, h.central(), X, y, l1, a1, p1)
    assert l1 < l0          # training lowered the held-out loss


def test_evaluate_without_set_is_rejected(agn):
    wl = WL.SMALL
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, 1, batch=wl.batch, n_samples=wl.n_samples) as h:
        with pytest.raises(agn.AGNError) as e:
            h.evaluate()
        assert e.value.code == agn.AGN_E_INVALID


def test_temporal_efficiency_of_agn_against_the_ablation(agn):
    """Accuracy-versus-time curves of AGN and of the un-normalised ablation on
    the small workload (time = cumulative device time of agn_run), and Eq. 4
    on them through the library, against the oracle's Eq. 4 on the same
    samples."""
    wl = WL.SMALL
    seed, C, n_eval = I.DEFAULT_SEED, 24, 2000
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    curves = []
    for normalize in (1, 0):
        with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch,
                     n_samples=wl.n_samples, normalize=normalize, n_eval=n_eval) as h:
            t, f = [0.0], [h.evaluate()[1]]
            for c in range(0, C, 4):
                h.run(4, w[c:], tau[c:])
                t.append(t[-1] + h.last_run_stats()["gpu_ms"])
                f.append(h.evaluate()[1])
            curves.append((np.array(t), np.array(f)))
    (ta, fa), (tb, fb) = curves
    e = agn.agn_temporal_efficiency(ta, fa, tb, fb)
    assert e == pytest.approx(O.temporal_efficiency(ta, fa, tb, fb), rel=1e-12)
    assert agn.agn_temporal_efficiency(ta, fa, ta, fa) == 1.0
    assert np.isfinite(e) and e > 0
