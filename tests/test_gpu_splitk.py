"""Split K in the forward and dX GEMMs (small waves): the ks CTAs of an output
tile each sum a range of k steps; rank j % ks finishes column chunk j of the
tile from the other ranks' partial sums, added in rank order.

Against the same runs with one CTA per output tile (tc_mask bit 4): the two
differ only in the fp32 summation order of the partial sums, so with every
ReLU unit kept away from its kink, theta~ and the losses agree to 3e-5
(fp32 mode) or to bf16 rounding of the stored activations (bf16 mode).  Few
workers make small waves, so the launches split K widely: up to 13 ranks on
784-wide inputs, more ranks than column chunks (ranks that only hand over
partial sums), uneven chunk ownership (3 ranks on 192- and 160-wide inputs),
column tiles of 64, 128 and 256 samples and ragged M and K.
"""

import numpy as np
import pytest

import agn_inputs as I

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _active_theta0(dims, seed, N):
    """The seeded initial parameters with every hidden bias raised so that each
    unit's pre-activation is at least 1 on all N training rows.  With a small
    step (pre-activations move by a few 1e-2 per local step) no ReLU comes
    near its kink during the run, so rounding differences of the GEMMs cannot
    switch a unit (which changes a sample's gradient discretely and would
    swamp the comparison)."""
    th = I.init_params(seed, dims).astype(np.float64)
    h = I.make_inputs_x(seed, dims[0], np.arange(N, dtype=np.int64), I.DIST_UNIFORM).astype(np.float64)
    offs = I.layer_offsets(dims)
    for l, (wo, bo) in enumerate(offs[:-1]):
        fi, fo = dims[l], dims[l + 1]
        z = h @ th[wo:bo].reshape(fo, fi).T
        th[bo:bo + fo] = 1.0 - z.min(axis=0)
        h = np.maximum(z + th[bo:bo + fo], 0.0)
    return th.astype(np.float32)


def _run(agn, dims, m, n, prec, mask, lam=2, seed=31):
    N, C = n * 4 * m, n + 2
    w, tau = I.make_schedule(n, C + n, 0, n - 1, seed)
    with agn.AGN(dims, n, lam, 1e-3, seed, batch=m, n_samples=N, precision=prec,
                 gemm=agn.AGN_GEMM_TCGEN05, tc_mask=mask,
                 theta0=_active_theta0(dims, seed, N)) as h:
        th0 = h.central()
        h.run(C, w, tau)
        return th0, h.central(), h.loss()


CASES = [((784, 1000, 1000, 10), 128, 1), ((784, 1000, 1000, 10), 128, 2),
         ((784, 1000, 1000, 10), 64, 3), ((200, 392, 264, 10), 128, 2),
         ((1024, 512, 512, 10), 256, 1), ((96, 168, 136, 10), 48, 2),
         ((192, 256, 160, 10), 128, 2)]


@pytest.mark.parametrize("dims,m,n", CASES)
@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_split_k_matches_one_cta_per_tile(agn, dims, m, n, prec):
    p = agn.AGN_PREC_FP32 if prec == "fp32" else agn.AGN_PREC_BF16
    th0, a, la = _run(agn, dims, m, n, p, 7)          # split K where waves are small
    th0b, b, lb = _run(agn, dims, m, n, p, 7 | 16)    # one CTA per output tile
    assert np.array_equal(th0, th0b)
    da, db = (a - th0).astype(np.float64), (b - th0).astype(np.float64)
    err = np.linalg.norm(da - db) / np.linalg.norm(db)
    tol = 3e-5 if prec == "fp32" else 1e-2
    assert err < tol, err
    assert np.max(np.abs(la - lb)) <= tol * max(1.0, float(np.max(np.abs(lb))))
