"""The standalone commit+pull kernel against the float32 oracle: bit-exact."""

import numpy as np
import pytest

import agn_inputs as I
import oracle as O
from agn_inputs import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import __graft_entry__ as g
    g.build()
    import torch
    import paper_1710_02368_gb300 as agn
    return agn, torch, torch.device("cuda:0")


def _csr(pulls):
    offs = np.cumsum([0] + [len(p) for p in pulls]).astype(np.int32)
    flat = np.array([p for ps in pulls for p in ps] or [0], dtype=np.int32)
    return offs, flat


def _alloc(torch, dev, P, ld, n):
    theta = torch.empty(P, device=dev)
    acc = torch.empty(n, ld, device=dev)
    reps = torch.zeros(n, ld, device=dev)
    return theta, acc, reps


def test_device_inputs_match_generator(env):
    agn, torch, dev = env
    P, ld, n, seed = 4099, 4100, 5, 17
    theta, acc, reps = _alloc(torch, dev, P, ld, n)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, ld, n, seed)
    torch.cuda.synchronize()
    assert np.array_equal(theta.cpu().numpy(), I.commit_bench_theta(seed, P))
    for k in range(n):
        assert np.array_equal(acc[k, :P].cpu().numpy(), I.commit_bench_acc(seed, P, k))
        assert np.array_equal(reps[k, :P].cpu().numpy(), I.commit_bench_theta(seed, P))


@pytest.mark.parametrize("P", [1 << 20, (1 << 20) + 3, 37])
def test_commit_pull_bit_exact(env, P):
    """64 accumulators, the seeded order, 4 pulls after every commit (lambda=10, eta=0.01)."""
    agn, torch, dev = env
    wl = WL.COMMIT_PULL
    n, seed = wl.n, I.DEFAULT_SEED
    ld = (P + 3) // 4 * 4
    theta, acc, reps = _alloc(torch, dev, P, ld, n)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, ld, n, seed)
    order, pulls = I.commit_bench_order(seed, n, wl.pulls_per_commit)
    offs, flat = _csr(pulls)
    dn = torch.zeros(n, device=dev)
    th0 = I.commit_bench_theta(seed, P)
    accs = {k: I.commit_bench_acc(seed, P, k) for k in range(n)}
    agn.agn_commit_pull(theta, acc, reps, None, P, ld, n, order, offs, flat, wl.eta, wl.lam,
                        delta_norm=dn)
    torch.cuda.synchronize()
    exp_t, exp_a, exp_r, exp_n = O.commit_pull_fp32(th0, accs, order, pulls, wl.eta, wl.lam,
                                                    replicas={k: th0 for k in range(n)})
    assert np.array_equal(theta.cpu().numpy(), exp_t)
    got_r = reps[:, :P].cpu().numpy()
    got_a = acc[:, :P].cpu().numpy()
    for k in range(n):
        assert np.array_equal(got_r[k], exp_r[k]), k
        assert np.all(got_a[k] == 0)
    assert np.allclose(dn.cpu().numpy(), exp_n, rtol=1e-6)


def test_commit_pull_bf16_copy_and_unnormalised(env):
    agn, torch, dev = env
    P, ld, n, seed = 50001, 50004, 6, 3
    theta, acc, reps = _alloc(torch, dev, P, ld, n)
    repb = torch.zeros(n, ld, dtype=torch.bfloat16, device=dev)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, ld, n, seed)
    order = [5, 1, 4, 4, 0]           # accumulator 4 twice: its second commit adds zeros
    pulls = [[0, 2], [], list(range(n)), [3], [1]]
    offs, flat = _csr(pulls)
    th0 = I.commit_bench_theta(seed, P)
    accs = {k: I.commit_bench_acc(seed, P, k) for k in range(n)}
    agn.agn_commit_pull(theta, acc, reps, repb, P, ld, n, order, offs, flat, 0.01, 10,
                        normalize=0)
    torch.cuda.synchronize()
    exp_t, _, exp_r, _ = O.commit_pull_fp32(th0, accs, order, pulls, 0.01, 10, normalize=False)
    assert np.array_equal(theta.cpu().numpy(), exp_t)
    for k, v in exp_r.items():
        assert np.array_equal(reps[k, :P].cpu().numpy(), v)
        b = torch.from_numpy(v).to(torch.bfloat16).float().numpy()
        assert np.array_equal(repb[k, :P].float().cpu().numpy(), b)


def test_commit_pull_many_pulls_one_commit(env):
    """More pulls after one commit than one launch carries (300 replicas)."""
    agn, torch, dev = env
    P, ld, n, seed = 1000, 1000, 300, 8
    theta, acc, reps = _alloc(torch, dev, P, ld, n)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, ld, n, seed)
    order = [7, 299]
    pulls = [list(range(n)), [0]]
    offs, flat = _csr(pulls)
    th0 = I.commit_bench_theta(seed, P)
    accs = {7: I.commit_bench_acc(seed, P, 7), 299: I.commit_bench_acc(seed, P, 299)}
    agn.agn_commit_pull(theta, acc, reps, None, P, ld, n, order, offs, flat, 0.01, 10)
    torch.cuda.synchronize()
    exp_t, _, exp_r, _ = O.commit_pull_fp32(th0, accs, order, pulls, 0.01, 10)
    assert np.array_equal(theta.cpu().numpy(), exp_t)
    got = reps.cpu().numpy()
    for k in range(n):
        assert np.array_equal(got[k], exp_r[k])


def test_commit_pull_rejects_bad_arguments(env):
    agn, torch, dev = env
    theta, acc, reps = _alloc(torch, dev, 16, 16, 2)
    with pytest.raises(agn.AGNError) as e:        # ld not a multiple of 4
        agn.agn_commit_pull(theta, acc, reps, None, 14, 14, 2, [0], [0, 0], [0], 0.01, 10)
    assert e.value.code == agn.AGN_E_INVALID
    with pytest.raises(agn.AGNError) as e:        # worker out of range
        agn.agn_commit_pull(theta, acc, reps, None, 16, 16, 2, [2], [0, 0], [0], 0.01, 10)
    assert e.value.code == agn.AGN_E_INVALID
    with pytest.raises(agn.AGNError) as e:        # misaligned device pointer
        agn.agn_commit_pull(theta.data_ptr() + 4, acc, reps, None, 8, 16, 2, [0], [0, 0], [0],
                            0.01, 10)
    assert e.value.code == agn.AGN_E_INVALID


@pytest.mark.parametrize("P", [1 << 28])
def test_commit_pull_full_size_sampled(env, P):
    """P = 2^28, the launch configuration the benchmark times; 4096 sampled
    parameters of theta~, of every replica and of every accumulator are
    compared bit for bit with the oracle run on those parameters."""
    agn, torch, dev = env
    wl = WL.COMMIT_PULL
    n, seed = wl.n, I.DEFAULT_SEED
    theta, acc, reps = _alloc(torch, dev, P, P, n)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, P, n, seed)
    order, pulls = I.commit_bench_order(seed, n, wl.pulls_per_commit)
    offs, flat = _csr(pulls)
    agn.agn_commit_pull(theta, acc, reps, None, P, P, n, order, offs, flat, wl.eta, wl.lam)
    rng = np.random.default_rng(0)
    idx = np.unique(np.concatenate([rng.integers(0, P, 4090), [0, 1, 2, P - 3, P - 2, P - 1]]))
    ti = torch.from_numpy(idx).to(dev)
    got_t = theta[ti].cpu().numpy()
    got_r = reps[:, ti].cpu().numpy()
    got_a = acc[:, ti].cpu().numpy()
    th0 = I.commit_bench_theta(seed, P, idx)
    accs = {k: I.commit_bench_acc(seed, P, k, idx) for k in range(n)}
    exp_t, _, exp_r, _ = O.commit_pull_fp32(th0, accs, order, pulls, wl.eta, wl.lam,
                                            replicas={k: th0 for k in range(n)})
    del theta, acc, reps
    torch.cuda.empty_cache()
    assert np.array_equal(got_t, exp_t)
    assert np.all(got_a == 0)
    for k in range(n):
        assert np.array_equal(got_r[k], exp_r[k])
