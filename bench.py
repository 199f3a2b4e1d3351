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
        src = {"forward": "mlp_tc.cu", "forward_head": "mlp_tc.cu", "backward_dx": "mlp_tc.cu",
               "backward_dw": "mlp_tc_dw.cu", "softmax": "mlp_head.cu",
               "commit": "commit_pull.cu"}.get(kernel_class)
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
              normalize=bool(wl.normalize),
              dtype=dtype)
    per_commit = time.perf_counter() - t0
    n_commits = max(1, min(wl.commits, int(seconds / max(per_commit, 1e-6))))
    t0 = time.perf_counter()
    O.agn_run(mlp, th0, wl.n, wl.lam, wl.eta, w[:n_commits], tau[:n_commits], ds, wl.batch,
              wl.shard, normalize=bool(wl.normalize), dtype=dtype)
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
                  wl.shard, normalize=bool(wl.normalize), dtype=dtype,
                  staleness_scaled=args.commit_rule == "dynsgd",
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
                   "sample": f"{per_step}-commit {'fp64' if dtype == np.float64 else 'fp32'} "
                             f"sample: each step re-runs the first {per_step} commits of the "
                             "workload on the CPU"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(),
                         "kind": "oracle",
                         "sample": f"{per_step} commits ({per_step * wl.lam} worker-steps) "
                                   "of the workload per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def commit_plan_launches(order, pulls, max_commits=16, max_pulls=256):
    """Commit launches the library makes for one pass: runs of at most 16
    consecutive commits, cut early at a repeated worker or when the pulls of
    the run would exceed 256 (the grouping of agn_commit_pull)."""
    launches, cur, npulls = 0, set(), 0
    for k, p in zip(order, pulls):
        if cur and (len(cur) == max_commits or int(k) in cur or npulls + len(p) > max_pulls):
            launches += 1
            cur, npulls = set(), 0
        cur.add(int(k))
        npulls += len(p)
    return launches + (1 if cur else 0)


def commit_pass_bytes(P, n_commits, n_pulls, launches):
    """Bytes one pass of the standalone commit workload must move: theta~ read
    and written once per launch (8P), each commit's accumulator read and
    zeroed (8P), each pull's replica written (4P)."""
    return float(P) * (8.0 * launches + 8.0 * n_commits + 4.0 * n_pulls)


def commit_kernel_bench(agn, torch, dev, P, min_ms=200.0):
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
    for _ in range(3):
        one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    one()
    e1.record(st)
    torch.cuda.synchronize()
    reps = max(3, int(min_ms / max(e0.elapsed_time(e1), 1e-3)))
    e0.record(st)
    for _ in range(reps):
        one()
    e1.record(st)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    launches = commit_plan_launches(order, pulls)
    bytes_ = commit_pass_bytes(P, n, len(flat), launches)
    del theta, acc, reps_t
    torch.cuda.empty_cache()
    return {"P": P, "commits": n, "pulls_per_commit": wl.pulls_per_commit, "passes_timed": reps,
            "ms_per_pass": ms, "GB/s": bytes_ / ms / 1e6, "bytes_per_pass": bytes_,
            "launches_per_pass": launches,
            "inputs": f"{(2 * n + 1) * P * 4 / 1e9:.2f} GB of accumulators, replicas and theta~ "
                      "(larger than L2)"}


def method_bytes_per_worker_step(wl, cls, fused_head=False):
    """Bytes the method itself moves per worker-step (one local step of one
    worker) in a kernel class: each local step reads and writes the fp32
    replica theta_k and accumulator a_k of every parameter (Algorithm 1: 16 B
    per parameter; 18 with the bf16 working copy the bf16 mode refreshes),
    plus the GEMM operands at the mode's element size (fp32 4 B, bf16 2 B).
    The fp32 mode's tensor-core pieces (6 B per operand element) are this
    implementation's cost and are left out.  None for classes without a
    per-step formula."""
    es = 4.0 if wl.precision == WL.PREC_FP32 else 2.0
    d, m = wl.dims, wl.batch
    L = len(d) - 1
    P = I.num_params(d)
    if cls == "backward_dw":
        return P * (16.0 if wl.precision == WL.PREC_FP32 else 18.0) + sum(
            m * (d[l] + d[l - 1]) * es for l in range(1, L + 1))
    if cls == "forward":        # the hidden layers (the last one not, when the output
        # layer rides in its epilogue: that launch is the forward_head class)
        return sum(d[l] * d[l - 1] * es + 4.0 * d[l] + m * (d[l - 1] + d[l]) * es
                   for l in range(1, L - 1 if fused_head else L))
    if cls == "backward_dx":    # layers L-1 .. 2 (the head writes layer L's dX)
        return sum(d[l] * d[l - 1] * es + m * d[l] * es + 2.0 * m * d[l - 1] * es
                   for l in range(2, L))
    if cls == "forward_head":   # the last hidden layer's forward and the output layer
        return (d[L - 1] * d[L - 2] * es + 4.0 * d[L - 1] + m * (d[L - 2] + 2.0 * d[L - 1]) * es
                + d[L] * d[L - 1] * es + 4.0 * d[L] + m * d[L] * es + 4.0 * m)
    if cls == "softmax":        # output layer: forward, softmax-CE, dX
        return (d[L] * d[L - 1] * es + 4.0 * d[L] + 2.0 * m * d[L - 1] * es + m * d[L] * es
                + 4.0 * m)
    if cls == "gather":
        return m * (2.0 * d[0] * es + 8.0)
    return None


GEMM_CLASSES = ("forward", "forward_head", "backward_dx", "backward_dw", "softmax")


def roofline(wl, kst, worker_steps, on_tc, hbm, bf16, peak_src):
    """Roofline of the dominant kernel class (by device time) from the CUDA
    events of the profiled region: achieved = method bytes (or flops) per
    launch / average launch time."""
    dom = max(("forward", "forward_head", "backward_dx", "backward_dw", "commit", "softmax",
               "gather"), key=lambda k: kst[k]["ms"])
    d = kst[dom]
    launches = max(d["launches"], 1)
    sec = d["ms"] / 1e3 / launches
    impl_bytes = d["bytes"] / launches
    mb = method_bytes_per_worker_step(wl, dom, fused_head=kst["forward_head"]["launches"] > 0)
    method_bytes = mb * worker_steps / launches if mb is not None else impl_bytes
    flops = d["flops"] / launches
    # fp32 mode on the tensor cores issues six bf16 piece products per fp32 product
    mma_per_flop = 6.0 if (wl.precision == WL.PREC_FP32 and on_tc) else 1.0
    if wl.precision == WL.PREC_FP32 and not on_tc and dom in GEMM_CLASSES:
        roof = {"bound": "alu", "achieved": flops / sec / 1e12, "peak": FP32_FMA_PEAK_TFLOPS,
                "unit": "TFLOP/s",
                "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 x 2.07 GHz"}
    elif flops * mma_per_flop / max(method_bytes, 1.0) >= bf16 * 1e12 / (hbm * 1e9):
        roof = {"bound": "tensor", "achieved": flops * mma_per_flop / sec / 1e12, "peak": bf16,
                "unit": "TFLOP/s", "peak_source": f"{peak_src} bf16 burst"}
    else:
        roof = {"bound": "hbm", "achieved": method_bytes / sec / 1e9, "peak": hbm,
                "unit": "GB/s", "peak_source": f"{peak_src} copy bandwidth"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["kernel"] = dom
    roof["avg_launch_us"] = 1e6 * sec
    roof["bytes_basis"] = ("method: fp32 theta_k and a_k read-modify-write per parameter and "
                           "local step (16 B; 18 B with the bf16 copy) plus the GEMM operands at "
                           "the mode's element size" if dom == "backward_dw" else
                           "method: the class's weights and activations at the mode's element "
                           "size" if mb is not None else "implementation bytes")
    roof["method_bytes_per_launch"] = method_bytes
    roof["impl_bytes_per_launch"] = impl_bytes
    roof["impl_frac"] = impl_bytes / sec / 1e9 / hbm
    roof["flops_per_launch"] = flops
    if dom in GEMM_CLASSES and on_tc:
        roof["tensor_pipe_frac_of_bf16_peak"] = mma_per_flop * flops / sec / 1e12 / bf16
    roof["traffic"] = _traffic_for(dom, wl.name, on_tc)
    return roof


def tensor_summary(wl, kst, ms_step, worker_steps_step, on_tc, bf16):
    """Tensor-pipe use of the GEMM classes: their method flops over their own
    device time, and over the whole step, against the bf16 burst peak (issued
    = six bf16 piece products per fp32 product in the fp32 mode)."""
    mma = 6.0 if (wl.precision == WL.PREC_FP32 and on_tc) else 1.0
    fl = sum(kst[k]["flops"] for k in GEMM_CLASSES)
    t = sum(kst[k]["ms"] for k in GEMM_CLASSES) / 1e3
    d, m = wl.dims, wl.batch
    W_f = sum(d[l] * d[l - 1] for l in range(1, len(d)))
    W_x = sum(d[l] * d[l - 1] for l in range(2, len(d)))
    step_flops = worker_steps_step * m * (4.0 * W_f + 2.0 * W_x)
    return {"gemm_method_tflops": fl / max(t, 1e-12) / 1e12,
            "gemm_issued_frac_of_bf16_peak": mma * fl / max(t, 1e-12) / 1e12 / bf16,
            "step_method_tflops": step_flops / (ms_step / 1e3) / 1e12,
            "step_issued_frac_of_bf16_peak": mma * step_flops / (ms_step / 1e3) / 1e12 / bf16}


def measure_workload(args, wl, agn, torch, dev, per_step, ws, clock_index=None):
    """Three timed regions over consecutive steps of one run of the workload:
    (1) device-resident inputs, no per-kernel events (the value); (2) CUDA
    events around every launch (per-kernel durations for the roofline and the
    shares); (3) end to end through the public API with the step's schedule
    from host memory and its losses read back."""
    st = torch.cuda.current_stream()
    seed = I.DEFAULT_SEED
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
        return h.loss() if e2e else None

    for i in range(args.warmup):
        step(i)
    launches = 0
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk = ClockSampler(clock_index) if clock_index is not None else None
    if clk is not None:
        clk.__enter__()
    e0.record(st)
    for i in range(args.warmup, args.warmup + args.steps):
        step(i)
        launches += int(h.last_run_stats()["launches"])
    e1.record(st)
    barrier()
    if clk is not None:
        clk.__exit__(None, None, None)
    ms = e0.elapsed_time(e1)
    h.profile(2)
    h.profile(1)
    barrier()
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if args.profile_region:
        torch.cuda.profiler.start()
    p0.record(st)
    for i in range(args.warmup + args.steps, args.warmup + 2 * args.steps):
        step(i)
    p1.record(st)
    barrier()
    if args.profile_region:
        torch.cuda.profiler.stop()
    h.profile(0)
    prof_ms = p0.elapsed_time(p1)
    kst = h.kernel_stats()
    barrier()
    t0 = time.perf_counter()
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2.record(st)
    d2h = 0
    for i in range(args.warmup + 2 * args.steps, args.warmup + 3 * args.steps):
        d2h += step(i, e2e=True).nbytes
    e3.record(st)
    barrier()
    e2e_ms = max(e2.elapsed_time(e3), 1e3 * (time.perf_counter() - t0))
    h.close()
    return {"ms": ms, "prof_ms": prof_ms, "e2e_ms": e2e_ms, "kst": kst, "launches": launches,
            "clk": clk, "d2h": d2h, "h2d": 2 * 4 * (per_step + wl.n)}


def tc_eligible(wl, gemm):
    return (gemm != "simt" and wl.batch <= 256 and len(wl.dims) >= 3
            and all(d % 8 == 0 for d in wl.dims[:-1]))


def workload_record(args, wl, r, per_step, ws, hbm, bf16, peak_src):
    on_tc = tc_eligible(wl, args.gemm)
    ms_step = r["ms"] / args.steps
    ws_step = per_step * wl.lam
    value = whole_job_value(ws, args.steps, per_step, wl.lam, wl.batch, r["ms"])
    rec = {
        "value": value, "unit": UNIT, "ms_per_step": ms_step,
        "dtype": "f32" if wl.precision == WL.PREC_FP32 else "bf16",
        "config": {"workload": wl.name, "commits_per_step": per_step,
                   "l2": "inputs larger than L2 (replicas and accumulators of all workers: "
                         f"{2 * wl.n * I.num_params(wl.dims) * 4 / 1e6:.0f} MB vs 129 MB L2)",
                   "gemm": ("tcgen05 bf16" if wl.precision == WL.PREC_BF16 else
                            "tcgen05 fp32 as three exact bf16 pieces") +
                           " (hidden layers); fused output layer on CUDA cores" if on_tc else
                           "CUDA-core GEMMs; fused output layer"},
        "roofline": roofline(wl, r["kst"], args.steps * ws_step, on_tc, hbm, bf16, peak_src),
        "tensor": tensor_summary(wl, r["kst"], r["prof_ms"] / args.steps, ws_step, on_tc, bf16),
        "events_region_ms_per_step": r["prof_ms"] / args.steps,
        "kernels": {k: {"launches": int(v["launches"]), "ms": round(v["ms"], 3),
                        "share": round(v["ms"] / max(sum(x["ms"] for x in r["kst"].values()),
                                                     1e-9), 4)}
                    for k, v in r["kst"].items() if v["launches"]},
        "e2e": {"value": whole_job_value(ws, args.steps, per_step, wl.lam, wl.batch,
                                         r["e2e_ms"]),
                "unit": UNIT, "h2d_bytes_per_step": r["h2d"],
                "d2h_bytes_per_step": r["d2h"] // max(args.steps, 1)},
        "gpu_launches": r["launches"],
    }
    return rec


def commit_sizes(args):
    """P values of the standalone commit workload (all four by default)."""
    if args.commit_log2p:
        return [1 << int(v) for v in args.commit_log2p.split(",")]
    return list(WL.COMMIT_PULL.sizes)


def run_commit_only(args):
    """Only the standalone commit+pull kernel (profiler captures of small P)."""
    import torch
    import paper_1710_02368_gb300 as agn
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    hbm, _, _, _ = _peaks()
    out = {}
    for P in commit_sizes(args):
        cr = commit_kernel_bench(agn, torch, dev, P)
        cr["frac_of_measured_hbm"] = cr["GB/s"] / hbm
        out[str(P)] = cr
    print(json.dumps({"commit_pull_kernel": out}), flush=True)
    return 0


def run_agn(args, wl):
    import torch
    import paper_1710_02368_gb300 as agn
    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    per_step = args.commits_per_step or (
        COMMITS_PER_STEP[args.workload] if not args.workers else 2 * wl.n)
    hbm, bf16, _, peak_src = _peaks()
    r = measure_workload(args, wl, agn, torch, dev, per_step, ws, clock_index=local)
    if ws > 1:
        r["ms"], r["e2e_ms"] = max_over_ranks([r["ms"], r["e2e_ms"]], dev)
    head = workload_record(args, wl, r, per_step, ws, hbm, bf16, peak_src)
    # the other MLP workloads of the benchmark, each measured the same way
    # (sub-records; the headline stays the workload above)
    subs = {}
    if rank == 0 and ws == 1 and not args.no_sub_workloads and args.workload == "mnist":
        for key in ("wide", "large"):
            swl = WORKLOADS[key]
            sr = measure_workload(args, swl, agn, torch, dev, COMMITS_PER_STEP[key], 1)
            subs[swl.name] = workload_record(args, swl, sr, COMMITS_PER_STEP[key], 1, hbm, bf16,
                                             peak_src)
    commit = None
    if rank == 0 and not args.no_commit_bench:
        commit = {}
        for P in commit_sizes(args):
            cr = commit_kernel_bench(agn, torch, dev, P)
            cr["frac_of_measured_hbm"] = cr["GB/s"] / hbm
            commit[str(P)] = cr
    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": head["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": head["dtype"],
        "data": "synthetic (seeded MNIST-shaped teacher-labelled set; MNIST itself unavailable)",
        "config": dict(head["config"], commit_rule=args.commit_rule,
                       accumulator="elided" if args.elide_accumulator else "kept",
                       local_optimizer=args.optimizer,
                       parallelism="replicas" if ws > 1 else "single GPU"),
        "roofline": head["roofline"],
        "tensor": head["tensor"],
        "events_region_ms_per_step": head["events_region_ms_per_step"],
        "kernels": head["kernels"],
        "gpu_launches": head["gpu_launches"],
        "clocks": r["clk"].summary() if r["clk"] is not None else None,
        "e2e": head["e2e"],
        "workloads": subs,
        "commit_pull_kernel": commit,
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
    ap.add_argument("--commit-log2p", default="",
                    help="comma-separated log2 P of the commit kernel runs (default: 20,24,26,28)")
    ap.add_argument("--commit-only", action="store_true",
                    help="time only the standalone commit+pull kernel")
    ap.add_argument("--lam", type=int, default=0,
                    help="local steps per commit (lambda) instead of the workload's own: the "
                         "lambda sweep of the 64-worker workload (1, 5, 10, 20, 40)")
    ap.add_argument("--profile-region", action="store_true",
                    help="bracket the per-kernel timing region with cudaProfilerStart/Stop, so "
                         "that ncu --profile-from-start off captures the launches the roofline "
                         "figures come from")
    ap.add_argument("--no-sub-workloads", action="store_true",
                    help="time only the headline workload (not the two bf16 workloads)")
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
    if args.lam:
        import dataclasses
        name = wl.name.replace(f"-lam{wl.lam}-", f"-lam{args.lam}-")
        wl = dataclasses.replace(wl, name=name if name != wl.name else f"{wl.name}-lam{args.lam}",
                                 lam=args.lam)
    if args.impl == "reference":
        return run_reference(args, wl)
    if args.commit_only:
        return run_commit_only(args)
    return run_agn(args, wl)


if __name__ == "__main__":
    sys.exit(main())
