"""Minibatches read in place from the padded shards (the tensor-core path's
default) against the same runs that gather each local step's minibatch into
a buffer of its own (tc_mask bit 6).

Worker w's shard is stored as S + m rows, row r holding dataset row
w S + (r mod S), so the minibatch of rows (t m + j) mod S (Algorithm 1's
FetchNextMiniBatch) is the m consecutive rows from (t m) mod S.  The forward
of layer 1 and the dW of layer 1 read their operand there and the output
layer reads its labels there.  A tile that reaches past the minibatch reads
the next rows of the shard instead of zero fill: those rows only meet
accumulator columns that are never stored (forward) or dZ rows that are zero
fill (dW), so both runs must agree bit for bit.  Cases: minibatches that wrap
around the end of the shard, a shard smaller than the minibatch (rows repeat
within one minibatch), one hidden layer (the output layer fused into layer
1's forward), the output layer as a kernel of its own, split K and column
tiles of 64, 128 and 256 samples, fp32 and bf16.
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


def _run(agn, dims, m, n, S, prec, mask, lam=3, seed=41):
    N, C = n * S, 3 * n + 1
    w, tau = I.make_schedule(n, C + n, 0, n - 1, seed)
    with agn.AGN(dims, n, lam, 0.02, seed, batch=m, n_samples=N, precision=prec,
                 gemm=agn.AGN_GEMM_TCGEN05, tc_mask=mask) as h:
        h.run(C, w, tau)
        return h.central(), h.loss()


# (dims, m, n, S): S not a multiple of m (minibatches wrap around the shard
# end), S < m, one hidden layer, wide inputs
CASES = [((784, 1000, 1000, 10), 128, 4, 300), ((256, 200, 136, 10), 48, 3, 100),
         ((96, 168, 136, 10), 48, 2, 40), ((256, 200, 10), 64, 3, 150),
         ((1024, 512, 512, 10), 256, 2, 600), ((192, 256, 160, 10), 32, 5, 70)]


@pytest.mark.parametrize("dims,m,n,S", CASES)
@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("head", ["fused", "kernel"])
def test_padded_shards_match_gather(agn, dims, m, n, S, prec, head):
    p = agn.AGN_PREC_FP32 if prec == "fp32" else agn.AGN_PREC_BF16
    base = 7 | (32 if head == "kernel" else 0)
    a, la = _run(agn, dims, m, n, S, p, base)          # padded shards, no gather
    b, lb = _run(agn, dims, m, n, S, p, base | 64)     # one gather launch per local step
    assert np.isfinite(a).all() and np.isfinite(la).all()
    assert np.array_equal(a, b), float(np.max(np.abs(a - b)))
    assert np.array_equal(la, lb), float(np.max(np.abs(la - lb)))
