"""The failure path of the bounded device waits, made to run out on purpose
without faulting or hanging the GPU.

The split-K ranks of a tensor-core forward or dX GEMM wait on the device for
each other's partial sums, and the fused output layer's feature tiles for
each other's partial logits.  Every such wait gives up after a time limit;
the kernel then skips its results, flags the run, and agn_run returns
AGN_E_TIMEOUT.  Here one split-K rank withholds its arrival (agn_debug_waits)
with a 2 ms limit: the run must end with AGN_E_TIMEOUT, the process's CUDA
context must stay usable, and a fresh handle must then match the oracle.
"""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


# small waves of a net whose forward and dX GEMMs split K (4 ranks and more)
DIMS, N_WORKERS, LAM, ETA, M, SEED, C = (256, 512, 256, 10), 2, 2, 0.05, 64, 31, 4


def _handle(agn):
    return agn.AGN(DIMS, N_WORKERS, LAM, ETA, SEED, batch=M, n_samples=N_WORKERS * 4 * M,
                   gemm=agn.AGN_GEMM_TCGEN05)


@pytest.mark.parametrize("rank", [0, 1])
def test_withheld_arrival_times_out_and_the_next_handle_is_correct(agn, rank):
    w, tau = I.make_schedule(N_WORKERS, C + N_WORKERS, 0, 1, SEED)
    with _handle(agn) as h:
        agn.agn_debug_waits(h.h, 2_000_000, rank)
        with pytest.raises(agn.AGNError) as e:
            h.run(C, w, tau)
        assert e.value.code == agn.AGN_E_TIMEOUT
    N = N_WORKERS * 4 * M
    ds = I.SyntheticDataset(SEED, DIMS[0], N, I.DIST_UNIFORM, (DIMS[0], 64, DIMS[-1]), N // N_WORKERS)
    ref = O.agn_run(O.MLP(DIMS), I.init_params(SEED, DIMS), N_WORKERS, LAM, ETA, w[:C], tau[:C],
                    ds, M, N // N_WORKERS)
    with _handle(agn) as h:
        h.run(C, w, tau)
        got = h.central().astype(np.float64)
    assert np.linalg.norm(got - ref.theta) / np.linalg.norm(ref.theta) <= 1e-5


def test_debug_waits_off_again_gives_a_normal_run(agn):
    """Setting the hook and clearing it before a run leaves the run untouched."""
    w, tau = I.make_schedule(N_WORKERS, C + N_WORKERS, 0, 1, SEED)
    with _handle(agn) as h:
        agn.agn_debug_waits(h.h, 2_000_000, 0)
        agn.agn_debug_waits(h.h, 0, -1)
        h.run(C, w, tau)
        assert np.all(np.isfinite(h.loss()))
