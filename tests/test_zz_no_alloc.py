"""agn_commit_pull_noalloc, the commit+pull entry point for callers that may
not allocate device memory (its scratch is a fixed device array), checked
against agn_commit_pull through the C ABI on two calls in a row.  This file
is collected last so that a run stopping at its first failure has already run
every other test."""

import numpy as np
import pytest

import agn_inputs as I

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import __graft_entry__ as g
    g.build()
    import torch
    import paper_1710_02368_gb300 as agn
    return agn, torch, torch.device("cuda:0")


def _buffers(agn, torch, dev, P, ld, n, seed):
    theta = torch.empty(P, device=dev)
    acc = torch.empty(n, ld, device=dev)
    reps = torch.empty(n, ld, device=dev)
    repb = torch.zeros(n, ld, dtype=torch.bfloat16, device=dev)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, ld, n, seed)
    return theta, acc, reps, repb


def test_noalloc_matches_allocating_entry_point_twice(env):
    agn, torch, dev = env
    P, ld, n, seed = (1 << 20) + 5, (1 << 20) + 8, 24, 41
    a = _buffers(agn, torch, dev, P, ld, n, seed)
    b = _buffers(agn, torch, dev, P, ld, n, seed)
    rng = np.random.default_rng(2)
    for call in range(2):                     # two calls in a row on the same buffers
        order = rng.permutation(n)[:20]
        if call == 1:
            # a worker that commits twice within one launch's 16 commits
            # makes both entry points end the launch early (the second commit
            # reads the accumulator that the first one zeroed)
            order[5] = order[2]
        pulls = [sorted(rng.choice(n, rng.integers(0, 5), replace=False)) for _ in order]
        offs = np.cumsum([0] + [len(p) for p in pulls]).astype(np.int32)
        flat = np.array([p for ps in pulls for p in ps] or [0], dtype=np.int32)
        na = torch.full((len(order),), -1.0, device=dev)
        nb = torch.full((len(order),), -1.0, device=dev)
        agn.agn_commit_pull(a[0], a[1], a[2], a[3], P, ld, n, order, offs, flat, 0.01, 10,
                            delta_norm=na)
        agn.agn_commit_pull_noalloc(b[0], b[1], b[2], b[3], P, ld, n, order, offs, flat, 0.01,
                                    10, delta_norm=nb)
        torch.cuda.synchronize()
        for x, y in zip(a, b):
            assert torch.equal(x, y), call
        # the first call commits fresh accumulators; the second call re-commits
        # some that the first one zeroed, whose norms are then exactly 0
        assert torch.all(nb >= 0) and (call > 0 or torch.all(nb > 0))
        # the same kernels with the same grid: the norms' fixed-order
        # reductions agree bit for bit
        assert torch.equal(na, nb), call
        if call == 1:
            assert float(nb[5]) == 0.0


def test_noalloc_rejects_more_pulls_than_it_carries(env):
    agn, torch, dev = env
    P, n = 64, 300
    theta, acc, reps, _ = _buffers(agn, torch, dev, P, P, n, 1)
    with pytest.raises(agn.AGNError) as e:
        agn.agn_commit_pull_noalloc(theta, acc, reps, None, P, P, n, [0], [0, n],
                                    list(range(n)), 0.01, 10)
    assert e.value.code == agn.AGN_E_INVALID and "at most 256" in str(e.value)
