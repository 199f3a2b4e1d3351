"""The wave plan that agn_run follows (host logic, no GPU): checked against
the schedule semantics of the FIFO server (Figure 1) and Algorithm 1's
Pull / local steps / Commit, not against the planner's own code.

Commit c of worker w_c reads theta~ after v_c = c - tau_c commits.  A plan is
valid when every commit's local steps run exactly once, in a wave that starts
after version v_c exists and before commit c is applied; commits are applied
in index order; each worker's commits run in order with its step counter
advancing by lambda per commit (never reset); each worker pulls exactly the
versions its commits read (version 0 is every replica's initial state); and
waves are maximal (a worker whose next commit's version exists runs in the
wave), which is what makes the plan the fastest one for a schedule.
"""

import numpy as np
import pytest

import agn_inputs as I


@pytest.fixture(scope="module")
def agn():
    import __graft_entry__ as g
    g.build()
    import paper_1710_02368_gb300 as agn
    return agn


def check_plan(agn, n, lam, w, tau, k):
    w, tau = np.asarray(w), np.asarray(tau)
    ws, we, sc, st, pulls = agn.agn_plan_waves(n, lam, k, w, tau)
    v = np.arange(len(w)) - tau
    # every commit's local steps exactly once
    assert sorted(sc.tolist()) == list(range(k))
    assert int(ws.sum()) == k and np.all(ws > 0)
    # commits applied in order, all of them by the end
    assert np.all(np.diff(we) > 0) and int(we[-1]) == k
    starts = np.concatenate([[0], we[:-1]])            # versions applied when each wave starts
    wave_of_slot = np.repeat(np.arange(len(ws)), ws)
    wave_of = np.empty(k, dtype=int)
    wave_of[sc] = wave_of_slot
    for c in range(k):
        wv = wave_of[c]
        assert v[c] <= starts[wv], (c, v[c], starts[wv])   # its version exists
        assert c >= starts[wv]                             # and it is not applied yet
    for wv in range(len(ws)):
        assert np.all(wave_of[starts[wv]:we[wv]] <= wv)    # applied only once computed
        if we[wv] < k:
            assert wave_of[we[wv]] > wv                    # the longest computed run
    # per worker: order, step counters, maximal waves, pulls
    t0 = np.empty(k, dtype=np.int64)
    t0[sc] = st
    for worker in range(n):
        cs = [c for c in range(k) if w[c] == worker]
        assert [wave_of[c] for c in cs] == sorted(wave_of[c] for c in cs)
        assert len(set(wave_of[c] for c in cs)) == len(cs)   # one commit per wave
        assert t0[cs].tolist() == [lam * i for i in range(len(cs))]
        for i, c in enumerate(cs):
            first_possible = 0 if i == 0 else wave_of[cs[i - 1]] + 1
            for wv in range(first_possible, wave_of[c]):
                assert v[c] > starts[wv], (worker, c, wv)    # could not have run earlier
        got = pulls[pulls[:, 1] == worker, 0].tolist()
        assert got == [int(v[c]) for c in cs if v[c] > 0]
    assert np.all(np.diff(pulls[:, 0]) >= 0)                 # pulls in version order
    return ws


@pytest.mark.parametrize("n,C,lo,hi,seed", [(4, 50, 0, 2, 1), (16, 300, 0, 15, 2),
                                            (16, 300, 15, 15, 3), (7, 120, 2, 5, 4),
                                            (1, 20, 0, 0, 5), (64, 400, 63, 63, 6)])
def test_plan_of_seeded_schedules(agn, n, C, lo, hi, seed):
    w, tau = I.make_schedule(n, C, lo, hi, seed)
    ws = check_plan(agn, n, 5, w, tau, C)
    if lo == hi == n - 1:       # round robin, homogeneous: every wave has all n workers
        assert np.all(ws[:-1] == n) and int(ws[-1]) == C - n * (len(ws) - 1)
    if n == 1:
        assert np.all(ws == 1)


@pytest.mark.parametrize("seed", range(6))
def test_plan_of_random_feasible_schedules(agn, seed):
    """Workers in random order (not round robin), versions drawn anywhere in
    the feasible range prev(w) < v_c <= c."""
    rng = np.random.default_rng(seed)
    n, C = int(rng.integers(2, 9)), 80
    prev = [-1] * n
    w, tau = [], []
    for c in range(C):
        k = int(rng.integers(0, n))
        v = int(rng.integers(prev[k] + 1, c + 1))
        w.append(k)
        tau.append(c - v)
        prev[k] = c
    check_plan(agn, n, 3, w, tau, C)


def test_plan_with_look_ahead_pulls(agn):
    """Entries past n_commits only add the pulls this run must make."""
    n, C = 4, 40
    w, tau = I.make_schedule(n, C + n, 0, 3, 11)
    ws, we, sc, st, pulls = agn.agn_plan_waves(n, 2, C, w, tau)
    assert int(we[-1]) == C and sorted(sc.tolist()) == list(range(C))
    v = np.arange(len(w)) - tau
    extra = [(int(v[c]), int(w[c])) for c in range(C, C + n) if 0 < v[c] <= C]
    inside = [(int(v[c]), int(w[c])) for c in range(C) if v[c] > 0]
    assert sorted(map(tuple, pulls.tolist())) == sorted(inside + extra)


def test_plan_rejects_infeasible_schedules(agn):
    with pytest.raises(agn.AGNError) as e:
        agn.agn_plan_waves(2, 1, 3, [0, 0, 1], [0, 1, 0])   # worker 0 reads before its own commit
    assert e.value.code == agn.AGN_E_SCHEDULE
    with pytest.raises(agn.AGNError) as e:
        agn.agn_plan_waves(2, 1, 2, [0, 3], [0, 0])         # no worker 3
    assert e.value.code == agn.AGN_E_SCHEDULE
    with pytest.raises(agn.AGNError) as e:
        agn.agn_plan_waves(2, 1, 3, [0, 1], [0, 0])         # fewer entries than commits
    assert e.value.code == agn.AGN_E_INVALID


def test_plan_rejects_more_workers_than_create_accepts(agn):
    """agn_create takes 1 .. 256 workers; the planner rejects n = 257 alike
    (a version pulled by more workers than one commit launch carries)."""
    n = 257
    w = np.arange(n, dtype=np.int32)
    tau = np.zeros(n, dtype=np.int32)
    tau[1:] = np.arange(n - 1)            # commits 1 .. n-1 all read version 1
    with pytest.raises(agn.AGNError) as e:
        agn.agn_plan_waves(n, 1, n, w, tau)
    assert e.value.code == agn.AGN_E_INVALID
    check_plan(agn, 256, 1, w[:256], tau[:256], 256)
