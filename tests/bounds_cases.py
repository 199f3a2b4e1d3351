"""Cases run against the bounds-checked build of the library (test infrastructure).

`python tests/bounds_cases.py <case>` with AGN_LIB_VARIANT=check in the
environment loads `libagn_gb300_check.so` (every wrapped kernel access checked
against the library's table of device buffers, see csrc/bounds.cuh), runs one
case on cuda:0, compares it with the oracle and prints one JSON line.  The
checked library is loaded once per process, so tests/test_gpu_bounds.py runs
each case in a child process.  Shapes are small and ragged (partial tiles,
partial 32-sample chunks, split K) so that every kernel reaches its edges.
"""

from __future__ import annotations

import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import agn_inputs as I  # noqa: E402
import oracle as O  # noqa: E402


def _rel(a, b):
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(np.asarray(a, dtype=np.float64) - b) / np.linalg.norm(b))


def _mlp(agn, dims, m, n, lam, C, seed, eta=0.05, tau=(0, 2), **kw):
    """Run C commits through the checked library and the float64 oracle."""
    N = n * 3 * m
    w, t = I.make_schedule(n, C + n, tau[0], tau[1], seed)
    ds = I.SyntheticDataset(seed, dims[0], N, I.DIST_UNIFORM, (dims[0], 64, dims[-1]), N // n)
    oracle_kw = {}
    if kw.get("commit_rule") == agn.AGN_COMMIT_DYNSGD:
        oracle_kw["staleness_scaled"] = True
    if kw.get("elide_accumulator"):
        oracle_kw["elide_accumulator"] = True
    if kw.get("local_optimizer") == agn.AGN_OPT_ADAM:
        oracle_kw["optimizer"] = "adam"
    with agn.AGN(dims, n, lam, eta, seed, batch=m, n_samples=N, **kw) as h:
        h.run(C, w, t)
        got, loss = h.central(), h.loss()
    ref = O.agn_run(O.MLP(dims), I.init_params(seed, dims), n, lam, eta, w[:C], t[:C], ds, m,
                    N // n, **oracle_kw)
    return {"rel": _rel(got, ref.theta), "loss_err": float(np.max(np.abs(loss - ref.loss)))}


def case_fp32_tc(agn):
    # tensor-core GEMMs, output layer in the forward epilogue, split K
    return _mlp(agn, (256, 200, 136, 10), 48, 4, 3, 9, 17, gemm=agn.AGN_GEMM_TCGEN05)


def case_fp32_tc_kernels(agn):
    # the output layer as a kernel of its own, the one-tile-per-CTA dW, no split K
    return _mlp(agn, (96, 64, 64, 10), 40, 3, 2, 7, 5, gemm=agn.AGN_GEMM_TCGEN05,
                tc_mask=32 | 8 | 16)


def case_fp32_simt(agn):
    return _mlp(agn, (70, 33, 10), 20, 3, 2, 7, 9, gemm=agn.AGN_GEMM_SIMT)


def case_variants(agn):
    out = {}
    for name, kw in (("dynsgd", {"commit_rule": agn.AGN_COMMIT_DYNSGD}),
                     ("elide", {"elide_accumulator": 1}),
                     ("adam", {"local_optimizer": agn.AGN_OPT_ADAM})):
        eta = 1e-3 if name == "adam" else 0.05
        r = _mlp(agn, (128, 64, 64, 10), 32, 3, 3, 7, 11, eta=eta, **kw)
        out[name + "_rel"] = r["rel"]
    return out


def case_bf16(agn):
    dims, m, n, lam, C, seed = (256, 128, 128, 10), 64, 4, 3, 9, 23
    N = n * 3 * m
    w, t = I.make_schedule(n, C + n, 0, 2, seed)
    ds = I.SyntheticDataset(seed, dims[0], N, I.DIST_UNIFORM, (dims[0], 64, dims[-1]), N // n)
    ref = O.agn_run(O.MLP(dims), I.init_params(seed, dims), n, lam, 0.05, w[:C], t[:C], ds, m,
                    N // n)
    errs = []
    for mask in (0, 32):   # output layer fused, and as a kernel of its own
        with agn.AGN(dims, n, lam, 0.05, seed, precision=agn.AGN_PREC_BF16, batch=m,
                     n_samples=N, gemm=agn.AGN_GEMM_TCGEN05, tc_mask=mask) as h:
            h.run(C, w, t)
            errs.append(float(np.max(np.abs(h.loss() - ref.loss))))
    return {"loss_err": max(errs)}


def case_mnist_shaped(agn):
    # the 16-worker 784-1000-1000-10 workload at full size, one 16-commit call
    from agn_inputs import workloads as WL
    wl = WL.MNIST_SHAPED
    seed, C = I.DEFAULT_SEED, 16
    w, t = I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, seed)
    with agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, batch=wl.batch, n_samples=wl.n_samples,
                 teacher_dims=wl.teacher_dims) as h:
        h.run(C, w, t)
        got = h.central()
    ds = I.SyntheticDataset(seed, wl.dims[0], wl.n_samples, wl.dist, wl.teacher_dims, wl.shard)
    ref = O.agn_run(O.MLP(wl.dims), I.init_params(seed, wl.dims), wl.n, wl.lam, wl.eta, w[:C],
                    t[:C], ds, wl.batch, wl.shard)
    return {"rel": _rel(got, ref.theta)}


def case_eval(agn):
    dims, m, n, lam, C, seed, ne = (64, 48, 10), 16, 3, 2, 5, 31, 300
    N = n * 3 * m
    w, t = I.make_schedule(n, C + n, 0, 2, seed)
    with agn.AGN(dims, n, lam, 0.05, seed, batch=m, n_samples=N, n_eval=ne) as h:
        h.run(C, w, t)
        loss, acc = h.evaluate()
        theta = h.central()
    rows = np.arange(N, N + ne, dtype=np.int64)
    xe = I.make_inputs_x(seed, dims[0], rows, I.DIST_UNIFORM)
    ye = I.teacher_labels(xe, I.teacher_params(seed, (dims[0], 64, dims[-1])), I.DIST_UNIFORM)
    ref_loss, _, _ = O.evaluate(O.MLP(dims, np.float32), theta, xe, ye, dtype=np.float32)
    return {"loss_rel": abs(loss - ref_loss) / abs(ref_loss)}


def _commit_inputs(agn, torch, P, ld, n, seed):
    dev = torch.device("cuda:0")
    theta = torch.empty(P, device=dev)
    acc = torch.empty(n, ld, device=dev)
    reps = torch.zeros(n, ld, device=dev)
    agn.agn_fill_commit_inputs(theta, acc, reps, P, ld, n, seed)
    torch.cuda.synchronize()
    return theta, acc, reps


def case_commit(agn):
    import torch
    out = {}
    for P, ld in ((1003, 1004), ((1 << 16) + 3, (1 << 16) + 4)):
        n, seed = 6, 3
        order = [2, 0, 5, 3, 1, 4, 0]
        pulls = [[1], [2, 3], [], [0, 4, 5], [1], [2], [3]]
        offs = np.cumsum([0] + [len(p) for p in pulls]).astype(np.int32)
        flat = np.array([p for ps in pulls for p in ps], dtype=np.int32)
        for fn in ("agn_commit_pull", "agn_commit_pull_noalloc"):
            theta, acc, reps = _commit_inputs(agn, torch, P, ld, n, seed)
            th0 = theta.cpu().numpy().copy()
            accs = {k: acc[k, :P].cpu().numpy().copy() for k in range(n)}
            dn = torch.zeros(len(order), device=theta.device)
            getattr(agn, fn)(theta, acc, reps, None, P, ld, n, order, offs, flat, 0.01, 10,
                             delta_norm=dn)
            torch.cuda.synchronize()
            exp_t, _, exp_r, _ = O.commit_pull_fp32(th0, accs, order, pulls, 0.01, 10)
            ok = np.array_equal(theta.cpu().numpy(), exp_t) and all(
                np.array_equal(reps[k, :P].cpu().numpy(), exp_r[k]) for k in exp_r)
            out[f"{fn}_{P}"] = bool(ok)
    return out


def case_detect(agn):
    """The checker itself: with AGN_BOUNDS_TEST_SHRINK=64 every buffer the
    library knows is registered 64 bytes short of its end, so the kernel's
    accesses to the last 16 floats of theta~ (inside the real allocation) are
    refused: the call must report AGN_E_BOUNDS and leave those floats as they
    were, while the rest is committed as usual."""
    import torch
    P, ld, n, seed = 1003, 1004, 4, 7
    theta, acc, reps = _commit_inputs(agn, torch, P, ld, n, seed)
    th0 = theta.cpu().numpy().copy()
    accs = {k: acc[k, :P].cpu().numpy().copy() for k in range(n)}
    order, pulls = [1, 3], [[0], [2]]
    offs = np.cumsum([0] + [len(p) for p in pulls]).astype(np.int32)
    flat = np.array([p for ps in pulls for p in ps], dtype=np.int32)
    code = 0
    try:
        agn.agn_commit_pull(theta, acc, reps, None, P, ld, n, order, offs, flat, 0.01, 10)
    except agn.AGNError as e:
        code = e.code
    torch.cuda.synchronize()
    got = theta.cpu().numpy()
    exp_t, _, _, _ = O.commit_pull_fp32(th0, accs, order, pulls, 0.01, 10)
    tail = P - 16
    return {"code": int(code), "tail_untouched": bool(np.array_equal(got[tail:], th0[tail:])),
            "head_committed": bool(np.array_equal(got[:tail - 4], exp_t[:tail - 4]))}


CASES = {k[5:]: v for k, v in globals().items() if k.startswith("case_")}


def main():
    if os.environ.get("AGN_LIB_VARIANT") != "check":
        raise SystemExit("run with AGN_LIB_VARIANT=check")
    import torch
    torch.cuda.set_device(0)
    import paper_1710_02368_gb300 as agn
    assert agn.library_path().endswith("libagn_gb300_check.so")
    result = CASES[sys.argv[1]](agn)
    print(json.dumps(result))


if __name__ == "__main__":
    main()
