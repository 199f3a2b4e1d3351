"""Write tests/golden/mnist_shaped_2000.txt from the CPU oracle alone.

The 16-worker fp32 workload (784-1000-1000-10, lambda = 15, eta = 0.01,
m = 128, 60k samples, staleness uniform in {0..15}) run for its 2000 commits
by the oracle (Algorithm 1 workers, Eq. 1-2 server) twice: in float64 (the
reference) and in float32 (NumPy single precision throughout).  The float32
run measures how far float32 arithmetic itself drifts from float64 on this
trajectory; the GPU parity test uses that drift as its envelope.

Stored: per commit the float64 loss (mean of the lambda minibatch losses)
and ||Delta_c||; at checkpoints c = 0, 100, .., 1900, 1999 the float64
||theta~||, the float32 run's relative L2 deviation, and theta~ (float64) at
256 seeded parameter indices; and, in mnist_shaped_2000_full.npz, the whole
theta~ after the last commit from both runs (float64 values rounded to
float32, a relative change of at most 2^-24 per element).  Takes about 30
minutes on 8 cores.

Usage: python tests/golden/make_mnist_shaped_golden.py
"""

import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import agn_inputs as I  # noqa: E402
import oracle as O  # noqa: E402
from agn_inputs import workloads as WL  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "mnist_shaped_2000.txt")
FULL_OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "mnist_shaped_2000_full.npz")
N_SAMPLED = 256


def checkpoints(C):
    return sorted(set(list(range(0, C, 100)) + [C - 1]))


def sampled_indices(P):
    return np.sort(np.random.default_rng(1710).choice(P, N_SAMPLED, replace=False))


def main():
    wl = WL.MNIST_SHAPED
    seed = I.DEFAULT_SEED
    C = wl.commits
    w, tau = I.make_schedule(wl.n, C, wl.tau_lo, wl.tau_hi, seed)
    ds = I.workload_dataset(wl, seed)
    th0 = I.init_params(seed, wl.dims)
    cps = checkpoints(C)
    r64 = O.agn_run(O.MLP(wl.dims), th0, wl.n, wl.lam, wl.eta, w, tau, ds, wl.batch, wl.shard,
                    snapshot_at=cps)
    r32 = O.agn_run(O.MLP(wl.dims, np.float32), th0, wl.n, wl.lam, wl.eta, w, tau, ds, wl.batch,
                    wl.shard, snapshot_at=cps, dtype=np.float32)
    idx = sampled_indices(th0.size)
    with open(OUT, "w") as f:
        f.write("# Oracle reference for the 16-worker fp32 workload (784-1000-1000-10,\n"
                "# n=16, lambda=15, eta=0.01, m=128, N=60000, tau ~ U{0..15}, seed "
                f"{seed}), 2000 commits.\n"
                "# Algorithm 1 (workers), Eq. 1 (normalised delta), Eq. 2 (FIFO server).\n"
                "# Written by tests/golden/make_mnist_shaped_golden.py from oracle/ only.\n")
        f.write("indices " + " ".join(str(int(i)) for i in idx) + "\n")
        for c in range(C):
            f.write(f"commit {c} {r64.loss[c]:.17g} {r64.delta_norm[c]:.17g}\n")
        for c in cps:
            a = r64.snapshots[c]
            dev = np.linalg.norm(r32.snapshots[c].astype(np.float64) - a) / np.linalg.norm(a)
            f.write(f"checkpoint {c} {np.linalg.norm(a):.17g} {dev:.17g} "
                    + " ".join(f"{v:.17g}" for v in a[idx]) + "\n")
    last = cps[-1]
    np.savez_compressed(FULL_OUT, commit=np.int64(last),
                        theta64=r64.snapshots[last].astype(np.float32),
                        theta32=r32.snapshots[last].astype(np.float32))
    print("wrote", OUT, FULL_OUT)


def load():
    """Parse the golden file: (indices, loss[C], dnorm[C], {c: (norm, dev32, values)})."""
    idx, loss, dn, cps = None, [], [], {}
    with open(OUT) as f:
        for line in f:
            if line.startswith("#"):
                continue
            p = line.split()
            if p[0] == "indices":
                idx = np.array([int(v) for v in p[1:]])
            elif p[0] == "commit":
                loss.append(float(p[2]))
                dn.append(float(p[3]))
            elif p[0] == "checkpoint":
                cps[int(p[1])] = (float(p[2]), float(p[3]), np.array([float(v) for v in p[4:]]))
    return idx, np.array(loss), np.array(dn), cps


def load_full():
    """(commit index, float64 oracle's theta~, float32 oracle's theta~) after
    the last commit, both as float32 arrays of P values in flat order."""
    z = np.load(FULL_OUT)
    return int(z["commit"]), z["theta64"], z["theta32"]


if __name__ == "__main__":
    main()
