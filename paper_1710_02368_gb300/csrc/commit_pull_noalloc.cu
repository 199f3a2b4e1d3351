// agn_commit_pull_noalloc: the standalone commit + pull for callers that may
// not allocate device memory.
//
// Some callers cannot call cudaMalloc on this path: a host framework that owns
// every byte of device memory through its own pool and forbids allocations
// outside it, or a latency-bound loop in which an allocation (which can
// synchronise the device or fail under memory pressure) is not allowed.  This
// entry point computes exactly what agn_commit_pull computes, with the same
// kernels, but takes its scratch memory (the per-block partial sums of the
// per-commit norms) from a fixed array in device global memory that the
// library reserves when it is loaded, instead of from the stream-ordered
// allocator.
#include <mutex>
#include <string>

#include "mlp.cuh"

namespace agn {
void set_global_error(const std::string& msg);   // agn_api.cu: agn_last_error(NULL)
}

namespace {

// Blocks of the commit kernel this entry point launches at most (the kernel
// loops over P, so any P works with a capped grid).
constexpr int kNoAllocMaxGrid = 1024;
constexpr size_t kScratchDoubles = (size_t)agn::kMaxCommitsPerLaunch * kNoAllocMaxGrid;

// 16 x 1024 doubles = 128 KiB, held by every GPU that loads the library
// until the process exits.  Shared by every call: see the header.
static __device__ __align__(256) double g_commit_scratch[kScratchDoubles];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
double* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device.  In host code
// the name g_commit_scratch is only a host-side stand-in, so the address is
// looked up once per device (with that device current) and cached.
agn::Status scratch_on_current_device(double** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return agn::cuda_status(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices)
    return agn::Status::Err(AGN_E_UNSUPPORTED, "device ordinal beyond 63");
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_commit_scratch);
    if (e != cudaSuccess) return agn::cuda_status(e, "cudaGetSymbolAddress(scratch)");
    g_scratch_ptr[dev] = static_cast<double*>(p);
  }
  *out = g_scratch_ptr[dev];
  return agn::Status::Ok();
}

agn::Status commit_pull_noalloc(float* theta_c, float* acc, float* reps, void* reps_b, int64_t P,
                                int64_t ld, int n, int C, const int32_t* cw, const int32_t* po,
                                const int32_t* pw, double eta, int lambda, int normalize,
                                float* dnorm, cudaStream_t st) {
  using agn::Status;
  if (P < 1 || ld < P || ld % 4 != 0 || n < 1 || C < 0 || lambda < 1 || !(eta > 0.0))
    return Status::Err(AGN_E_INVALID, "bad sizes (need P >= 1, ld >= P, ld % 4 == 0, n >= 1)");
  if (!theta_c || !acc || (C > 0 && (!cw || !po)))
    return Status::Err(AGN_E_INVALID, "null pointer");
  auto misaligned = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) != 0; };
  if (misaligned(theta_c) || misaligned(acc) || (reps && misaligned(reps)) ||
      (reps_b && (reinterpret_cast<uintptr_t>(reps_b) & 7) != 0))
    return Status::Err(AGN_E_INVALID, "device buffers must be 16-byte aligned");
  if (C == 0) return Status::Ok();
  if (po[0] != 0) return Status::Err(AGN_E_INVALID, "pull_offsets[0] must be 0");
  // offsets first (they bound every later read), then the pointers the pulls need
  for (int c = 0; c < C; ++c)
    if (po[c + 1] < po[c]) return Status::Err(AGN_E_INVALID, "pull_offsets must not decrease");
  if (po[C] > 0 && (!reps || !pw)) return Status::Err(AGN_E_INVALID, "pulls need replicas");
  for (int c = 0; c < C; ++c) {
    if (cw[c] < 0 || cw[c] >= n) return Status::Err(AGN_E_INVALID, "commit worker out of range");
    if (po[c + 1] - po[c] > agn::kMaxPullsPerLaunch)
      return Status::Err(AGN_E_INVALID,
                         "commit " + std::to_string(c) + " has " + std::to_string(po[c + 1] - po[c]) +
                             " pulls; this entry point takes at most " +
                             std::to_string(agn::kMaxPullsPerLaunch) + " per commit");
    for (int p = po[c]; p < po[c + 1]; ++p)
      if (pw[p] < 0 || pw[p] >= n) return Status::Err(AGN_E_INVALID, "pull worker out of range");
  }
  double* scratch = nullptr;
  AGN_TRY(scratch_on_current_device(&scratch));
  const float scale = (float)(normalize ? -(eta / (double)lambda) : -eta);
  const int grid = std::min(agn::commit_grid(P), kNoAllocMaxGrid);
  // bounds-checked build: the caller's buffers and the scratch array are known
  // for this call (nothing is allocated; in the normal build this is empty)
  struct CallBuffers {
    const void* p[6] = {};
    int k = 0;
    void add(const void* q, size_t b) {
      if (q) {
        agn::bounds_add(q, b);
        p[k++] = q;
      }
    }
    ~CallBuffers() {
      for (int i = 0; i < k; ++i) agn::bounds_remove(p[i]);
    }
  } call;
  call.add(theta_c, (size_t)P * sizeof(float));
  call.add(acc, (size_t)n * ld * sizeof(float));
  call.add(reps, (size_t)n * ld * sizeof(float));
  call.add(reps_b, (size_t)n * ld * sizeof(agn::bf16));
  call.add(dnorm, (size_t)C * sizeof(float));
  call.add(scratch, kScratchDoubles * sizeof(double));
  AGN_TRY(agn::bounds_upload(st));
  agn::CommitPlan cp{};
  auto flush = [&]() -> Status {
    if (cp.n_commits > 0)
      AGN_TRY(agn::launch_commit_pull(cp, theta_c, acc, reps, static_cast<agn::bf16*>(reps_b), P,
                                      ld, scale, true, dnorm ? scratch : nullptr, grid, dnorm,
                                      nullptr, st));
    cp = agn::CommitPlan{};
    return Status::Ok();
  };
  for (int c = 0; c < C; ++c) {
    bool dup = false;
    for (int i = 0; i < cp.n_commits; ++i) dup |= cp.worker[i] == cw[c];
    const int np = po[c + 1] - po[c];
    if (cp.n_commits == agn::kMaxCommitsPerLaunch || dup ||
        cp.pull_begin[cp.n_commits] + np > agn::kMaxPullsPerLaunch)
      AGN_TRY(flush());
    const int i = cp.n_commits;
    cp.worker[i] = cw[c];
    cp.norm_slot[i] = c;
    int pb = cp.pull_begin[i];
    for (int p = po[c]; p < po[c + 1]; ++p) cp.pull_worker[pb++] = pw[p];
    cp.pull_begin[i + 1] = pb;
    cp.n_commits = i + 1;
  }
  AGN_TRY(flush());
  return agn::bounds_collect(st);   // bounds-checked build only
}

}  // namespace

extern "C" int agn_commit_pull_noalloc(float* theta_c, float* acc, float* replicas,
                                       void* replicas_bf16, int64_t P, int64_t ld, int32_t n,
                                       int32_t C, const int32_t* commit_worker,
                                       const int32_t* pull_offsets, const int32_t* pull_workers,
                                       double eta, int32_t lambda, int32_t normalize,
                                       float* delta_norm, void* stream) {
  agn::Status s = commit_pull_noalloc(theta_c, acc, replicas, replicas_bf16, P, ld, n, C,
                                      commit_worker, pull_offsets, pull_workers, eta, lambda,
                                      normalize, delta_norm, static_cast<cudaStream_t>(stream));
  if (!s.ok()) agn::set_global_error(s.msg);
  return s.code;
}
