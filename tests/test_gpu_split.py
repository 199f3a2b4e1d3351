"""fp32 mode on the tensor cores: every fp32 operand enters tcgen05.mma as
three exact bf16 pieces (x = x0 + x1 + x2) and the six piece products with
i + j <= 2 are accumulated in fp32, which keeps fp32-level accuracy.

Checked against the fp32 CUDA-core kernels (each GEMM kind alone and all
together, on shapes with partial tiles) and against the float64 oracle with
the fp32 tolerance (1e-5 relative L2 on theta~ after every checked commit).
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


def _run(agn, dims, m, gemm, mask=0, n=4, lam=2, C=5, seed=13, tau=(1, 2)):
    N = n * 3 * m
    w, t = I.make_schedule(n, C + n, tau[0], tau[1], seed)
    with agn.AGN(dims, n, lam, 0.05, seed, batch=m, n_samples=N, gemm=gemm, tc_mask=mask) as h:
        th0 = h.central()
        h.run(C, w, t)
        return th0, h.central(), h.loss()


@pytest.mark.parametrize("dims,m", [((256, 200, 136, 10), 48), ((784, 128, 10), 32),
                                    ((96, 64, 64, 10), 256)])
@pytest.mark.parametrize("mask", [1, 2, 4, 7])
def test_split_gemms_match_cuda_core_fp32(agn, dims, m, mask):
    if mask == 2 and len(dims) < 4:
        pytest.skip("dX of a hidden layer needs two hidden layers")
    th0, a, la = _run(agn, dims, m, agn.AGN_GEMM_SIMT)
    th0b, b, lb = _run(agn, dims, m, agn.AGN_GEMM_TCGEN05, mask)
    assert np.array_equal(th0, th0b)
    da, db = (a - th0).astype(np.float64), (b - th0).astype(np.float64)
    err = np.linalg.norm(db - da) / np.linalg.norm(da)
    assert err < 1e-3, err
    assert np.allclose(la, lb, rtol=1e-5, atol=1e-6)


def _rel(a, b):
    return float(np.linalg.norm(a.astype(np.float64) - b) / np.linalg.norm(b))


@pytest.mark.parametrize("wl,C", [(WL.SMALL, 50), (WL.MNIST_SHAPED, 32)],
                         ids=["small", "mnist_shaped_prefix"])
def test_split_mode_matches_oracle_every_commit(agn, wl, C):
    seed = I.DEFAULT_SEED
    w, tau = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    ds = I.workload_dataset(wl, seed)
    ref = O.agn_run(O.MLP(wl.dims), I.init_params(seed, wl.dims), wl.n, wl.lam, wl.eta, w[:C],
                    tau[:C], ds, wl.batch, wl.shard, snapshot_at=range(C))
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 gemm=agn.AGN_GEMM_TCGEN05) as h:
        errs = []
        for c in range(C):
            h.run(1, w[c:], tau[c:])
            errs.append(_rel(h.central(), ref.snapshots[c]))
        loss = h.loss()
    assert max(errs) <= 1e-5, (int(np.argmax(errs)), max(errs))
    assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6)


def test_split_mode_is_the_default_for_fp32(agn):
    """AUTO picks the tensor cores for an eligible fp32 net and the CUDA cores
    for one whose widths are not multiples of 8; both give the same result up
    to fp32 rounding."""
    dims, m = (40, 72, 10), 16
    th0, auto, _ = _run(agn, dims, m, agn.AGN_GEMM_AUTO)
    _, tc, _ = _run(agn, dims, m, agn.AGN_GEMM_TCGEN05)
    assert np.array_equal(auto, tc)
    with pytest.raises(agn.AGNError) as e:
        _run(agn, (37, 65, 10), 8, agn.AGN_GEMM_TCGEN05)
    assert e.value.code == agn.AGN_E_UNSUPPORTED


@pytest.mark.parametrize("dims,m,n", [((256, 200, 136, 10), 48, 4), ((96, 64, 64, 10), 256, 3),
                                      ((784, 128, 10), 32, 4), ((64, 40, 3), 16, 5),
                                      ((128, 1000, 16), 128, 2)])
def test_output_layer_in_forward_epilogue(agn, dims, m, n):
    """The output layer (forward, softmax-CE, dZ_L, dX) folded into the last
    hidden layer's forward GEMM against the oracle (float64) and against the
    output layer as a kernel of its own (tc_mask bit 5), on shapes with
    partial feature tiles, partial 32-sample chunks, few classes and 16
    classes: theta~ and every loss within the fp32 tolerance."""
    seed, lam, C = 17, 3, 9
    N = n * 3 * m
    w, tau = I.make_schedule(n, C + n, 0, 2, seed)
    ds = I.SyntheticDataset(seed, dims[0], N, I.DIST_UNIFORM, (dims[0], 64, dims[-1]), N // n)
    ref = O.agn_run(O.MLP(dims), I.init_params(seed, dims), n, lam, 0.05, w[:C], tau[:C], ds, m,
                    N // n, snapshot_at=[C - 1])
    out = {}
    for mask in (0, 32):
        with agn.AGN(dims, n, lam, 0.05, seed, batch=m, n_samples=N, gemm=agn.AGN_GEMM_TCGEN05,
                     tc_mask=mask) as h:
            h.run(C, w, tau)
            out[mask] = (h.central(), h.loss())
    for mask, (th, loss) in out.items():
        assert _rel(th, ref.snapshots[C - 1]) <= 1e-5, mask
        assert np.allclose(loss, ref.loss, rtol=1e-5, atol=1e-6), mask
    assert _rel(out[0][0], out[32][0].astype(np.float64)) <= 1e-5
