"""Write the float32 oracle's per-commit record of the two bf16 MLP workloads
at their full sizes, from the CPU oracle alone.

Each variant runs the oracle (Algorithm 1 workers, Eq. 1 normalised delta,
Eq. 2 FIFO server) in NumPy float32 on the workload's seeded inputs and its
homogeneous round-robin schedule (tau = n - 1, Fig. 1), and stores per commit
the mean of the lambda minibatch losses, ||Delta_c||_2 and ||theta~||_2 after
the commit.  The bf16 GPU mode is judged on the loss (within 2e-2 of these
values for every commit); the norms are kept for the report.

Variants (name: workload, lambda, normalisation, commits):
  wide          3072-2048x3-10, n=32, lambda=10, AGN,            320 commits
  large_lam10   784-4096-4096-10, n=64, lambda=10, AGN,          320 commits
  large_lam1    the same net, lambda=1 (AGN = DOWNPOUR),          320 commits
  large_lam5    lambda=5,  AGN,                                   128 commits
  large_lam20   lambda=20, AGN,                                   128 commits
  large_lam40   lambda=40, AGN,                                    64 commits
  large_lam10_unnorm  lambda=10 without the 1/lambda (Fig. 3),    128 commits
The oracle takes about 0.3 s per worker-step on these nets, so the runs are
bounded: every variant covers at least one full wave of n commits.

Usage: python tests/golden/make_bf16_goldens.py <variant> [<variant> ...]
       (each variant writes tests/golden/bf16_<variant>.txt)
"""

import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import agn_inputs as I  # noqa: E402
import oracle as O  # noqa: E402
from agn_inputs import workloads as WL  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))

# name -> (workload, lambda, normalize, commits)
VARIANTS = {
    "wide": (WL.WIDE_BF16, 10, 1, 320),
    "large_lam10": (WL.LARGE_BF16, 10, 1, 320),
    "large_lam1": (WL.LARGE_BF16, 1, 1, 320),
    "large_lam5": (WL.LARGE_BF16, 5, 1, 128),
    "large_lam20": (WL.LARGE_BF16, 20, 1, 128),
    "large_lam40": (WL.LARGE_BF16, 40, 1, 64),
    "large_lam10_unnorm": (WL.LARGE_BF16, 10, 0, 128),
}


def path(name):
    return os.path.join(HERE, f"bf16_{name}.txt")


def schedule(name):
    """The round-robin schedule of a variant (with n entries of look-ahead)."""
    wl, lam, normalize, C = VARIANTS[name]
    return I.make_schedule(wl.n, C + wl.n, wl.tau_lo, wl.tau_hi, I.DEFAULT_SEED)


def run(name):
    wl, lam, normalize, C = VARIANTS[name]
    seed = I.DEFAULT_SEED
    w, tau = schedule(name)
    ds = I.workload_dataset(wl, seed)
    th0 = I.init_params(seed, wl.dims)
    t0 = time.time()
    r = O.agn_run(O.MLP(wl.dims, np.float32), th0, wl.n, lam, wl.eta, w[:C], tau[:C], ds,
                  wl.batch, wl.shard, normalize=bool(normalize), dtype=np.float32)
    dt = time.time() - t0
    with open(path(name), "w") as f:
        f.write(f"# Float32 oracle record of {wl.name} with lambda={lam}, "
                f"{'AGN (normalised, Eq. 1)' if normalize else 'un-normalised ablation (Fig. 3)'}"
                f",\n# dims {'-'.join(map(str, wl.dims))}, n={wl.n}, eta={wl.eta}, m={wl.batch}, "
                f"N={wl.n_samples}, tau = n-1 round robin, seed {seed}, {C} commits.\n"
                "# Algorithm 1 (workers), Eq. 1 (delta), Eq. 2 (FIFO server).\n"
                "# Written by tests/golden/make_bf16_goldens.py from oracle/ only "
                f"({dt:.0f} s).\n"
                "# columns: commit loss ||Delta_c|| ||theta~||\n")
        for c in range(C):
            f.write(f"{c} {r.loss[c]:.9g} {r.delta_norm[c]:.9g} {r.theta_norm[c]:.9g}\n")
    print("wrote", path(name), f"{dt:.0f} s", flush=True)


def load(name):
    """(loss[C], delta_norm[C], theta_norm[C]) of a variant's stored record."""
    a = np.loadtxt(path(name), comments="#", ndmin=2)
    return a[:, 1], a[:, 2], a[:, 3]


if __name__ == "__main__":
    names = sys.argv[1:] or sorted(VARIANTS)
    for nm in names:
        if nm not in VARIANTS:
            sys.exit(f"unknown variant {nm}; one of {sorted(VARIANTS)}")
    for nm in names:
        run(nm)
