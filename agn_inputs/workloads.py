"""The five AGN workloads, as plain data (no arithmetic of the method).

Each MLP workload names: layer dims, n workers, lambda local steps, eta,
minibatch m per worker, dataset size N and distribution, teacher dims, the
staleness range of the round-robin schedule, the number of commits and the
compute precision.  `commit_pull` is the standalone commit+pull workload.
Shapes follow the paper's setting (Section 4: m=128, MNIST-shaped 784-dim
inputs with 10 classes, n and lambda in the tens); the rest is synthetic.
"""

from __future__ import annotations

from dataclasses import dataclass, field

from . import DIST_NORMAL, DIST_UNIFORM

PREC_FP32 = 0
PREC_BF16 = 1


@dataclass(frozen=True)
class MLPWorkload:
    name: str
    dims: tuple
    n: int
    lam: int
    eta: float
    batch: int
    n_samples: int
    dist: int
    teacher_dims: tuple
    tau_lo: int
    tau_hi: int
    commits: int
    precision: int
    normalize: int = 1
    lam_sweep: tuple = field(default=())

    @property
    def shard(self) -> int:
        return self.n_samples // self.n


@dataclass(frozen=True)
class CommitWorkload:
    name: str
    sizes: tuple          # P values
    n: int                # accumulators / replicas
    lam: int
    eta: float
    pulls_per_commit: int


# n=4, lambda=5, 784-128-10, fp32, m=32, 2048 samples, teacher 784-64-10,
# tau ~ U{0,1,2}, 50 commits.
SMALL = MLPWorkload(
    name="agn-784-128-10-n4-lam5-m32-fp32", dims=(784, 128, 10), n=4, lam=5,
    eta=0.05, batch=32, n_samples=2048, dist=DIST_UNIFORM,
    teacher_dims=(784, 64, 10), tau_lo=0, tau_hi=2, commits=50,
    precision=PREC_FP32)

# n=16, lambda=15, 784-1000-1000-10, fp32, m=128, 60k samples,
# staleness up to n-1, 2000 commits.
MNIST_SHAPED = MLPWorkload(
    name="agn-784-1000-1000-10-n16-lam15-m128-fp32", dims=(784, 1000, 1000, 10),
    n=16, lam=15, eta=0.01, batch=128, n_samples=60000, dist=DIST_UNIFORM,
    teacher_dims=(784, 64, 10), tau_lo=0, tau_hi=15, commits=2000,
    precision=PREC_FP32)

# n=32, lambda=10, 3072-2048-2048-2048-10, bf16 with fp32 master, m=256,
# 50k N(0,1) samples, homogeneous round robin (tau = n-1), 1000 commits.
WIDE_BF16 = MLPWorkload(
    name="agn-3072-2048x3-10-n32-lam10-m256-bf16", dims=(3072, 2048, 2048, 2048, 10),
    n=32, lam=10, eta=0.01, batch=256, n_samples=50000, dist=DIST_NORMAL,
    teacher_dims=(3072, 64, 10), tau_lo=31, tau_hi=31, commits=1000,
    precision=PREC_BF16)

# commit+pull alone: P in {1M,16M,64M,256M}, 64 accumulators, lambda=10,
# eta=0.01, each commit followed by 4 pulls.
COMMIT_PULL = CommitWorkload(
    name="agn-commit-pull-n64", sizes=(1 << 20, 1 << 24, 1 << 26, 1 << 28), n=64,
    lam=10, eta=0.01, pulls_per_commit=4)

# n=64, lambda in {1,5,10,20,40}, 784-4096-4096-10 bf16/fp32 master, m=64,
# 100k samples, tau = n-1, 5000 commits; ablation without the 1/lambda.
LARGE_BF16 = MLPWorkload(
    name="agn-784-4096-4096-10-n64-lam10-m64-bf16", dims=(784, 4096, 4096, 10),
    n=64, lam=10, eta=0.01, batch=64, n_samples=100000, dist=DIST_UNIFORM,
    teacher_dims=(784, 64, 10), tau_lo=63, tau_hi=63, commits=5000,
    precision=PREC_BF16, lam_sweep=(1, 5, 10, 20, 40))

MLP_WORKLOADS = {w.name: w for w in (SMALL, MNIST_SHAPED, WIDE_BF16, LARGE_BF16)}

__all__ = ["MLPWorkload", "CommitWorkload", "SMALL", "MNIST_SHAPED", "WIDE_BF16",
           "COMMIT_PULL", "LARGE_BF16", "MLP_WORKLOADS", "PREC_FP32", "PREC_BF16",
           "DIST_UNIFORM", "DIST_NORMAL"]
