"""The persistent multi-layer dW kernel against the earlier one-tile-per-CTA
dW kernel (layer by layer, biases from a separate reduction kernel, the
output layer on CUDA cores).

Both issue the same tcgen05.mma sequence for the weight tiles (same k order,
same piece pairs) and the same epilogue arithmetic, so after one local step
the weight updates agree bit for bit.  The bias gradients differ only in
summation order (the persistent kernel sums dZ_l through a row of ones in the
GEMM), so they agree to fp32 rounding, and so do whole runs.  Shapes cover
ragged input tiles (d_{l-1} not a multiple of 128, where the bias row sits in
the last tile), inputs that are a multiple of 128 (the bias row gets a tile of
its own), ragged feature tiles and chunks (d_l not a multiple of the column
tile or of 32), m not a multiple of 64, and waves with more tiles than SMs.
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
        th0 = h.central()
        h.run(C, w, tau)
        return th0, h.central(), h.loss()


CASES = [((256, 512, 384, 10), 64, 4), ((784, 200, 10), 128, 4), ((192, 256, 256, 10), 256, 4),
         ((96, 64, 64, 10), 48, 4), ((1024, 2048, 10), 64, 8), ((1024, 1000, 10), 128, 8)]
PRECS = ["bf16", "fp32"]


def _prec(agn, p):
    return agn.AGN_PREC_BF16 if p == "bf16" else agn.AGN_PREC_FP32


@pytest.mark.parametrize("dims,m,n", CASES)
@pytest.mark.parametrize("prec", PRECS)
def test_first_step_weights_bit_identical(agn, dims, m, n, prec):
    """One commit of one local step: the weight part of theta~ is equal bit
    for bit; the bias part to fp32 rounding of the gradient sum."""
    th0, c1, _ = _run(agn, dims, m, n, _prec(agn, prec), 7, lam=1, C=1)
    _, c2, _ = _run(agn, dims, m, n, _prec(agn, prec), 15, lam=1, C=1)
    offs = I.layer_offsets(dims)
    for l, (wo, bo) in enumerate(offs):
        fo = dims[l + 1]
        if l + 1 < len(offs):   # hidden layers: the same MMA sequence and epilogue
            assert np.array_equal(c1[wo:bo], c2[wo:bo]), l
        else:   # the output layer: tensor-core tiles vs the CUDA-core kernel
            d1 = (c1[wo:bo] - th0[wo:bo]).astype(np.float64)
            d2 = (c2[wo:bo] - th0[wo:bo]).astype(np.float64)
            assert np.max(np.abs(d1 - d2)) <= 1e-5 * np.max(np.abs(d2)) + 1e-12, l
        d1 = (c1[bo:bo + fo] - th0[bo:bo + fo]).astype(np.float64)
        d2 = (c2[bo:bo + fo] - th0[bo:bo + fo]).astype(np.float64)
        assert np.max(np.abs(d1 - d2)) <= 1e-5 * np.max(np.abs(d2)) + 1e-12, l


@pytest.mark.parametrize("dims,m,n", CASES)
@pytest.mark.parametrize("prec", PRECS)
def test_persistent_dw_matches_tiled_dw(agn, dims, m, n, prec):
    th0, c1, l1 = _run(agn, dims, m, n, _prec(agn, prec), 7)     # persistent dW (default)
    _, c2, l2 = _run(agn, dims, m, n, _prec(agn, prec), 15)      # one tile per CTA
    d1, d2 = (c1 - th0).astype(np.float64), (c2 - th0).astype(np.float64)
    tol = 1e-2 if prec == "bf16" else 1e-4
    assert np.linalg.norm(d1 - d2) <= tol * np.linalg.norm(d2)
    assert np.max(np.abs(l1 - l2)) <= tol * np.max(np.abs(l2))


@pytest.mark.parametrize("dims,m,n", CASES)
@pytest.mark.parametrize("prec", PRECS)
def test_accumulator_l2_adds_match_ring(agn, dims, m, n, prec):
    """a_k += g as L2 adds (red.add, the default for waves whose accumulators
    fit well within the L2: all cases but the 8-worker 1024-2048-10 one,
    whose 65 MB take the ring either way) against a_k's chunks read
    through the parameter ring and stored back (tc_mask bit 8): one add of
    the same two floats per element and local step either way, so after
    several commits of three local steps theta~ and the losses agree bit for
    bit."""
    _, c1, l1 = _run(agn, dims, m, n, _prec(agn, prec), 7, lam=3, C=2 * n)
    _, c2, l2 = _run(agn, dims, m, n, _prec(agn, prec), 7 | 256, lam=3, C=2 * n)
    assert np.isfinite(c1).all()
    assert np.array_equal(c1, c2), float(np.max(np.abs(c1 - c2)))
    assert np.array_equal(l1, l2)
