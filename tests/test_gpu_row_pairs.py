"""Two 128-row tiles per CTA in the bf16 forward and dX GEMMs of full waves
(the tiles of a launch outnumber the SMs): the two tiles share each B stage
and keep one TMEM accumulator each.  Against the same runs with one tile per
CTA (tc_mask bit 7) the MMAs of every output element run over the same k
steps in the same order, so both agree bit for bit.  Cases: column tiles of
256 and 128 samples, a row count that leaves the last CTA's second tile
partly (and one that leaves it wholly) past the layer's rows, forward of
layer 1 from the padded shards, and the dX of every hidden layer above it.
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


def _run(agn, dims, m, n, mask, lam=2, seed=43):
    N, C = n * 2 * m, n + 3
    w, tau = I.make_schedule(n, C + n, n - 1, n - 1, seed)   # round robin: full waves
    with agn.AGN(dims, n, lam, 0.01, seed, batch=m, n_samples=N,
                 precision=agn.AGN_PREC_BF16, gemm=agn.AGN_GEMM_TCGEN05, tc_mask=mask) as h:
        h.run(C, w, tau)
        return h.central(), h.loss()


# (dims, m, n): 16 x 10, 16 x 10, 15 x 11 and 13 x 12 row tiles per layer and wave
CASES = [((3072, 2048, 2048, 10), 256, 10), ((1024, 2048, 2048, 10), 128, 10),
         ((512, 1920, 1920, 10), 256, 11), ((768, 1664, 1600, 10), 128, 12)]


@pytest.mark.parametrize("dims,m,n", CASES)
def test_row_pairs_match_one_tile_per_cta(agn, dims, m, n):
    a, la = _run(agn, dims, m, n, 7)          # two row tiles per CTA where the wave is full
    b, lb = _run(agn, dims, m, n, 7 | 128)    # one row tile per CTA
    assert np.isfinite(a).all() and np.isfinite(la).all()
    assert np.array_equal(a, b), float(np.max(np.abs(a - b)))
    assert np.array_equal(la, lb), float(np.max(np.abs(la - lb)))
