"""Benchmark of the AGN hot path on GB300 (one JSON line on rank 0).

Workload (default): 16 workers, lambda = 15, eta = 0.01, MLP 784-1000-1000-10
fp32, minibatch 128 per worker, 60k synthetic MNIST-shaped samples, seeded
round-robin schedule with staleness uniform in {0..15}; 2000 commits in all.
A step is 100 consecutive commits of that schedule: every row of the path
(pull, minibatch fetch, forward, softmax-CE, dX, dW with the fused local
update and accumulation, commit + normalisation, pulls).  Metric:
worker-samples/s = commits * lambda * m / time.

--impl reference times the CPU oracle (the plain NumPy restatement of the
method) on a bounded sample of the same workload instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import select
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import agn_inputs as I  # noqa: E402
from agn_inputs import workloads as WL  # noqa: E402

METRIC = "worker-samples/s (fwd+bwd+AGN commit) on 1 GB300; % tensor-pipe peak; commit HBM GB/s"
UNIT = "worker-samples/s"
# commits per step: whole waves where the schedule allows (n or 2n commits)
COMMITS_PER_STEP = {"mnist": 100, "small": 50, "wide": 64, "large": 128}
GEMMS = {"auto": 0, "simt": 1, "tcgen05": 2}
WORKLOADS = {"mnist": WL.MNIST_SHAPED, "small": WL.SMALL, "wide": WL.WIDE_BF16,
             "large": WL.LARGE_BF16}
# FP32 FMA peak of the CUDA cores: 152 SMs x 128 lanes x 2 flop x 2.07 GHz.
FP32_FMA_PEAK_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12
BF16_OVER_FP32_NOMINAL = 1.0


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained"), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def max_over_ranks(values, device):
    """Each value's maximum over the ranks of the default process group (every
    rank receives it): the slowest rank's time is the job's time."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def whole_job_value(world_size, steps, commits_per_step, lam, batch, ms):
    """Worker-samples per second of the whole job: every rank runs its own
    replica of the workload (weak scaling), so the units add up over ranks,
    divided by the slowest rank's time."""
    return world_size * steps * commits_per_step * lam * batch / (ms / 1e3)


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 100 ms."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return self
        # the sampler's start-up must not eat the timed region: wait (3 s at
        # most) for its first sample, which is taken before the region and
        # not counted
        ready, _, _ = select.select([self.proc.stdout], [], [], 3.0)
        if ready:
            self.proc.stdout.readline()
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in getattr(self, "lines", []):
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def _traffic_for(kernel_class, workload, on_tc):
    """ncu DRAM bytes per launch of a kernel class, if a summary for the current
    source of that kernel exists under profiles/ (else None)."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    if on_tc:
        src = {"forward": "mlp_tc.cu", "backward_dx": "mlp_tc.cu", "backward_dw": "mlp_tc_dw.cu",
               "softmax": "mlp_head.cu", "commit": "commit_pull.cu"}.get(kernel_class)
    else:
        src = {"forward": "mlp_simt.cu", "backward_dx": "mlp_simt.cu",
               "backward_dw": "mlp_simt.cu", "commit": "commit_pull.cu"}.get(kernel_class)
    if src is None:
        return None
    digest = hashlib.sha256(open(os.path.join(ROOT, "paper_1710_02368_gb300", "csrc", src),
                                 "rb").read()).hexdigest()[:12]
    for line in open(path):
        f = line.split()
        if len(f) >= 4 and not line.startswith("#") and f[0] == kernel_class and f[1] == workload \
                and f[3] == digest:
            return float(f[2])
    return None


def cpu_baseline(wl, seconds=15.0):
    """The oracle (as it stands) on the first commits of the workload, fp64."""
    import oracle as O
    seed = I.DEFAULT_SEED
    w, tau = I.make_schedule(wl.n, wl.commits, wl.tau_lo, wl.tau_hi, seed)
    ds = I.workload_dataset(wl, seed)
    th0 = I.init_params(seed, wl.dims)
    dtype = np.float64 if wl.precision == WL.PREC_FP32 else np.float32
    mlp = O.MLP(wl.dims, dtype)
    # warm the dataset cache outside the timing
    for k in range(wl.n):
        ds(np.array([k * wl.shard]))
    t0 = time.perf_counter()
    O.agn_run(mlp, th0, wl.n, wl.lam, wl.eta, w[:1], tau[:1], ds, wl.batch, wl.shard,
              dtype=dtype)
    per_commit = time.perf_counter() - t0
    n_commits = max(1, min(wl.commits, int(seconds / max(per_commit, 1e-6))))
    t0 = time.perf_counter()
    O.agn_run(mlp, th0, wl.n, wl.lam, wl.eta, w[:n_commits], tau[:n_commits], ds, wl.batch,
              wl.shard, dtype=dtype)
    dt = time.perf_counter() - t0
    return {"value": n_commits * wl.lam * wl.batch / dt, "unit": UNIT, "cores": os.cpu_count(),
            "kind": "oracle",
            "sample": f"first {n_commits} commits of the workload ({n_commits * wl.lam} "
                      f"worker-steps of m={wl.batch}), NumPy {np.dtype(dtype).name}, "
                      f"{dt:.1f} s"}


def run_reference(args, wl):
    ws, rank, _ = _dist()
    if rank != 0:
        return 0
    import oracle as O
    seed = I.DEFAULT_SEED
    w, tau = I.make_schedule(wl.n, wl.commits, wl.tau_lo, wl.tau_hi, seed)
    ds = I.workload_dataset(wl, seed)
    th0 = I.init_params(seed, wl.dims)
    dtype = np.float64 if wl.precision == WL.PREC_FP32 else np.float32
    mlp = O.MLP(wl.dims, dtype)
    per_step = max(1, args.ref_commits)

    def step():
        O.agn_run(mlp, th0, wl.n, wl.lam, wl.eta, w[:per_step], tau[:per_step], ds, wl.batch,
                  wl.shard, dtype=dtype, staleness_scaled=args.commit_rule == "dynsgd",
                  elide_accumulator=args.elide_accumulator, optimizer=args.optimizer)
    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    value = args.steps * per_step * wl.lam * wl.batch / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64" if dtype == np.float64 else "f32", "data": "synthetic",
        "config": {"workload": wl.name, "commits_per_step": per_step,
                   "commit_rule": args.commit_rule,
                   "sample": f"each step re-runs the first {per_step} commits on the CPU"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(),
                         "kind": "oracle",
                         "sample": f"{per_step} commits ({per_step * wl.lam} worker-steps) "
                                   "of the workload per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def commit_kernel_bench(agn, torch, dev, P=1 << 28, reps=3):
    """The standalone commit+pull kernel: 64 accumulators, the seeded order,
    4 pulls after each commit (one pass = 64 commits)."""
    wl = WL.COMMIT_PULL
    n = wl.n
    theta = torch.empty(P, device=dev)
    acc = torch.empty(n, P, device=dev)
    reps_t = torch.empty(n, P, device=dev)
    agn.agn_fill_commit_inputs(theta, acc, reps_t, P, P, n, I.DEFAULT_SEED)
    order, pulls = I.commit_bench_order(I.DEFAULT_SEED, n, wl.pulls_per_commit)
    offs = np.cumsum([0] + [len(p) for p in pulls]).astype(np.int32)
    flat = np.concatenate(pulls).astype(np.int32)
    st = torch.cuda.current_stream()

    def one():
        agn.agn_commit_pull(theta, acc, reps_t, None, P, P, n, order, offs, flat, wl.eta, wl.lam,
                            stream=st.cuda_stream)
    one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(reps):
        one()
    e1.record(st)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    bytes_ = P * 4.0 * (2 + 2 * n + n * wl.pulls_per_commit)
    del theta, acc, reps_t
    torch.cuda.empty_cache()
    return {"P": P, "commits": n, "pulls_per_commit": wl.pulls_per_commit,
            "ms_per_pass": ms, "GB/s": bytes_ / ms / 1e6, "launches_per_pass": 2 * ((n + 15) // 16)}


def run_agn(args, wl):
    import torch
    import paper_1710_02368_gb300 as agn
    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    st = torch.cuda.current_stream()
    seed = I.DEFAULT_SEED
    per_step = args.commits_per_step or (
        COMMITS_PER_STEP[args.workload] if not args.workers else 2 * wl.n)
    total = (args.warmup + 3 * args.steps) * per_step + wl.n
    w, tau = agn.agn_make_schedule(wl.n, total, wl.tau_lo, wl.tau_hi, seed)
    h = agn.AGN(wl.dims, wl.n, wl.lam, wl.eta, seed, precision=wl.precision, batch=wl.batch,
                n_samples=wl.n_samples, input_dist=wl.dist, teacher_dims=wl.teacher_dims,
                normalize=wl.normalize, gemm=GEMMS[args.gemm], stream=st.cuda_stream,
                commit_rule=agn.AGN_COMMIT_DYNSGD if args.commit_rule == "dynsgd"
                else agn.AGN_COMMIT_AGN, elide_accumulator=int(args.elide_accumulator),
                local_optimizer=agn.AGN_OPT_ADAM if args.optimizer == "adam" else agn.AGN_OPT_SGD)

    def barrier():
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    def step(i, e2e=False):
        a = i * per_step
        h.run(per_step, w[a:], tau[a:])
        if e2e:
            return h.loss()
        return None

    for i in range(args.warmup):
        step(i)
    # timed region 1: device-resident inputs, no per-kernel events (the
    # headline value)
    launches = 0
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        e0.record(st)
        for i in range(args.warmup, args.warmup + args.steps):
            step(i)
            launches += int(h.last_run_stats()["launches"])
        e1.record(st)
        barrier()
    ms = e0.elapsed_time(e1)
    # timed region 2: the next steps of the same run with CUDA events around
    # every kernel launch on the launching stream (per-kernel durations for
    # the roofline and the shares; the events themselves cost some time, so
    # this region is not the headline)
    h.profile(2)
    h.profile(1)
    barrier()
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    p0.record(st)
    for i in range(args.warmup + args.steps, args.warmup + 2 * args.steps):
        step(i)
    p1.record(st)
    barrier()
    h.profile(0)
    prof_ms = p0.elapsed_time(p1)
    kst = h.kernel_stats()
    tc_ok = wl.batch <= 256 and all(d % 8 == 0 for d in wl.dims[:-1])
    if args.gemm != "simt" and tc_ok:
        gemm_used = ("tcgen05 bf16" if wl.precision == WL.PREC_BF16 else
                     "tcgen05 fp32 as three exact bf16 pieces") + \
                    " (hidden layers); fused output layer on CUDA cores"
    else:
        gemm_used = "CUDA-core GEMMs; fused output layer"
    # timed region 2: end to end through the public API with host buffers
    barrier()
    t0 = time.perf_counter()
    e2 = torch.cuda.Event(enable_timing=True)
    e3 = torch.cuda.Event(enable_timing=True)
    e2.record(st)
    d2h = 0
    for i in range(args.warmup + 2 * args.steps, args.warmup + 3 * args.steps):
        losses = step(i, e2e=True)
        d2h += losses.nbytes
    e3.record(st)
    barrier()
    e2e_ms = max(e2.elapsed_time(e3), 1e3 * (time.perf_counter() - t0))
    h2d = 2 * 4 * (per_step + wl.n)           # the schedule window of each step
    if ws > 1:
        ms, e2e_ms = max_over_ranks([ms, e2e_ms], dev)
    value = whole_job_value(ws, args.steps, per_step, wl.lam, wl.batch, ms)
    e2e_value = whole_job_value(ws, args.steps, per_step, wl.lam, wl.batch, e2e_ms)

    hbm, bf16, bf16_sus, peak_src = _peaks()
    dom = max(("forward", "backward_dx", "backward_dw", "commit", "softmax", "gather"),
              key=lambda k: kst[k]["ms"])
    d = kst[dom]
    on_tc = args.gemm != "simt" and tc_ok
    if dom in ("forward", "backward_dx", "backward_dw"):
        if wl.precision == WL.PREC_FP32 and not on_tc:
            roof = {"bound": "alu", "achieved": d["flops"] / d["ms"] / 1e9,
                    "peak": FP32_FMA_PEAK_TFLOPS, "unit": "TFLOP/s",
                    "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 x 2.07 GHz"}
        else:
            # bf16 GEMMs: the bound is set by the arithmetic intensity against
            # the ridge point of the measured peaks (bf16 TFLOP/s / HBM GB/s)
            ai = d["flops"] / max(d["bytes"], 1.0)
            if ai >= bf16 * 1e12 / (hbm * 1e9):
                roof = {"bound": "tensor", "achieved": d["flops"] / d["ms"] / 1e9, "peak": bf16,
                        "unit": "TFLOP/s", "peak_source": f"{peak_src} bf16 burst"}
            else:
                roof = {"bound": "hbm", "achieved": d["bytes"] / d["ms"] / 1e6, "peak": hbm,
                        "unit": "GB/s", "peak_source": f"{peak_src} copy bandwidth"}
            # fp32 mode on tensor cores issues six bf16 piece products per fp32 product
            mma_per_flop = 6.0 if wl.precision == WL.PREC_FP32 else 1.0
            roof["tensor_pipe_frac_of_bf16_peak"] = mma_per_flop * d["flops"] / d["ms"] / 1e9 / bf16
            roof["arithmetic_intensity_flop_per_byte"] = ai
    else:
        roof = {"bound": "hbm", "achieved": d["bytes"] / d["ms"] / 1e6, "peak": hbm,
                "unit": "GB/s", "peak_source": f"{peak_src} copy bandwidth"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    tr = _traffic_for(dom, wl.name, on_tc)
    roof["traffic"] = tr
    roof["kernel"] = dom
    roof["avg_launch_us"] = 1e3 * d["ms"] / max(d["launches"], 1)
    roof["events_region_ms_per_step"] = prof_ms / args.steps
    roof["algorithmic_per_launch"] = {"flops": d["flops"] / max(d["launches"], 1),
                                      "bytes": d["bytes"] / max(d["launches"], 1)}
    kernels = {k: {"launches": int(v["launches"]), "ms": round(v["ms"], 3),
                   "share": round(v["ms"] / max(sum(x["ms"] for x in kst.values()), 1e-9), 4)}
               for k, v in kst.items() if v["launches"]}
    h.close()
    commit = None
    if rank == 0 and not args.no_commit_bench:
        commit = commit_kernel_bench(agn, torch, dev)
        commit["frac_of_measured_hbm"] = commit["GB/s"] / hbm
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "f32" if wl.precision == WL.PREC_FP32 else "bf16",
        "data": "synthetic (seeded MNIST-shaped teacher-labelled set; MNIST itself unavailable)",
        "config": {"workload": wl.name, "commits_per_step": per_step,
                   "commit_rule": args.commit_rule,
                   "accumulator": "elided" if args.elide_accumulator else "kept",
                   "local_optimizer": args.optimizer,
                   "parallelism": "replicas" if ws > 1 else "single GPU",
                   "l2": "inputs larger than L2 (dataset 188 MB + replicas and accumulators "
                         "230 MB vs 129 MB L2)" if args.workload == "mnist" else
                         "inputs larger than L2 (replicas and accumulators of all workers)",
                   "gemm": gemm_used},
        "roofline": roof,
        "kernels": kernels,
        "commit_pull_kernel": commit,
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h // max(args.steps, 1)},
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, args.cpu_seconds)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="agn", choices=["agn", "reference"])
    ap.add_argument("--workload", default="mnist", choices=sorted(WORKLOADS))
    ap.add_argument("--commits-per-step", type=int, default=0)
    ap.add_argument("--gemm", default="auto", choices=sorted(GEMMS))
    ap.add_argument("--commit-rule", default="agn", choices=["agn", "dynsgd"],
                    help="AGN's commit (Eq. 1) or the DynSGD-style staleness-scaled commit")
    ap.add_argument("--elide-accumulator", action="store_true",
                    help="keep no gradient accumulator; commit from the pulled parameters")
    ap.add_argument("--optimizer", default="sgd", choices=["sgd", "adam"],
                    help="the local optimizer of the workers (Algorithm 1's gradient line)")
    ap.add_argument("--workers", type=int, default=0,
                    help="override n (profiling captures of a smaller case)")
    ap.add_argument("--ref-commits", type=int, default=2)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-commit-bench", action="store_true")
    args = ap.parse_args()
    wl = WORKLOADS[args.workload]
    if args.workers:
        # a smaller copy of the workload (fewer workers, same shapes), for
        # profiler captures that must stay small; not a benchmark line
        import dataclasses
        wl = dataclasses.replace(wl, name=f"{wl.name}-workers{args.workers}", n=args.workers,
                                 n_samples=wl.shard * args.workers,
                                 tau_lo=min(wl.tau_lo, args.workers - 1),
                                 tau_hi=min(wl.tau_hi, args.workers - 1))
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_agn(args, wl)


if __name__ == "__main__":
    sys.exit(main())
