"""The persistent dW kernel against the earlier one-tile-per-CTA dW kernel.

Both issue the same tcgen05.mma sequence per tile (same k order, same piece
pairs) and the same epilogue arithmetic, so theta~, the losses and every
replica agree bit for bit.  Shapes cover ragged input tiles (d_{l-1} not a
multiple of 128), ragged feature tiles and chunks (d_l not a multiple of the
column tile or of 32), m not a multiple of 64, and waves with more tiles than
SMs (several tiles per persistent CTA).
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


def _run(agn, dims, m, n, precision, mask, lam=2, C=6, seed=21):
    N = n * 3 * m
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)
    with agn.AGN(dims, n, lam, 0.05, seed, batch=m, n_samples=N, precision=precision,
                 gemm=agn.AGN_GEMM_TCGEN05, tc_mask=mask) as h:
        h.run(C, w, tau)
        reps = np.stack([h.replica(k) for k in range(n)])
        return h.central(), h.loss(), reps


CASES = [((256, 512, 384, 10), 64, 4), ((784, 200, 10), 128, 4), ((192, 256, 256, 10), 256, 4),
         ((96, 64, 64, 10), 48, 4), ((1024, 2048, 10), 64, 8), ((1024, 1000, 10), 128, 8)]


@pytest.mark.parametrize("dims,m,n", CASES)
@pytest.mark.parametrize("prec", ["bf16", "fp32"])
def test_persistent_dw_matches_tiled_dw(agn, dims, m, n, prec):
    precision = agn.AGN_PREC_BF16 if prec == "bf16" else agn.AGN_PREC_FP32
    c1, l1, r1 = _run(agn, dims, m, n, precision, 7)     # persistent dW (default)
    c2, l2, r2 = _run(agn, dims, m, n, precision, 15)    # one tile per CTA
    assert np.array_equal(c1, c2)
    assert np.array_equal(l1, l2)
    assert np.array_equal(r1, r2)
