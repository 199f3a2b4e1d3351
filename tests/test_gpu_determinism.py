"""Run-to-run determinism at the benchmark's shapes.

Given the schedule, AGN's result is a function of its inputs (Algorithm 1
with a fixed FIFO order of commits).  The GPU path keeps it so: split-K
partial sums are added in rank order, the output layer's partial logits in
feature-tile order, norms and losses by fixed trees, and every accumulator
element gets exactly one add per local step (also where that add is done by
the L2).  Two runs of the same handle arguments therefore agree bit for bit:
theta~, the per-commit losses and the per-commit update norms, on the
16-worker 784-1000-1000-10 fp32 workload (random staleness, waves of 1 to 16
workers) and on a full-wave bf16 workload.
"""

import numpy as np
import pytest

import agn_inputs as I
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def _run(agn, wl, C, n=None):
    n = n or wl.n
    seed = I.DEFAULT_SEED
    w, tau = I.make_schedule(n, C + n, min(wl.tau_lo, n - 1), min(wl.tau_hi, n - 1), seed)
    with agn.AGN(wl.dims, n, wl.lam, wl.eta, seed, precision=wl.precision, batch=wl.batch,
                 n_samples=wl.shard * n, input_dist=wl.dist,
                 teacher_dims=wl.teacher_dims) as h:
        h.run(C // 2, w, tau)
        h.run(C - C // 2, w[C // 2:], tau[C // 2:])
        return h.central(), h.loss(), h.delta_norm()


@pytest.mark.parametrize("name,C,n", [("MNIST_SHAPED", 48, None), ("WIDE_BF16", 24, 12)])
def test_two_runs_bit_identical(agn, name, C, n):
    wl = getattr(WL, name)
    a = _run(agn, wl, C, n)
    b = _run(agn, wl, C, n)
    assert np.isfinite(a[0]).all()
    for x, y in zip(a, b):
        assert np.array_equal(x, y), float(np.max(np.abs(x - y)))
