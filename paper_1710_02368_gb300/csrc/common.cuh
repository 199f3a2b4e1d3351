// Shared definitions of the AGN CUDA library (not part of the C ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstdio>
#include <string>
#include <utility>

#include "../../include/agn.h"
#include "bounds.cuh"

namespace agn {

// Programmatic dependent launch: every kernel of the library is launched with
// programmatic stream serialisation and starts with pdl_begin(), which waits
// for the preceding kernel of the stream to complete (and its memory to be
// visible) before touching global memory, then lets the next kernel launch.
// The next kernel's launch and CTA dispatch thereby overlap this kernel's run;
// the order of memory accesses is that of plain stream order.
__device__ __forceinline__ void pdl_begin() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
// The tensor-core forward and dX request their first weight stages before
// their dependency wait.  That is safe for weights written two or more
// kernels back (the preceding kernel let them launch only after its own
// wait).  The kernels that write replicas the very next kernel may read so
// (the dW local step, pulls, the Adam step) therefore wait without letting
// the next kernel launch early (pdl_wait_only): it launches when all their
// CTAs have exited, and every thread fences its writes before it exits
// (pdl_fence_exit), so they are visible to those early reads.
__device__ __forceinline__ void pdl_wait_only() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_fence_exit() { __threadfence(); }

// Handles that time each kernel with CUDA events (agn_profile) turn the
// overlap off while they do, so that an event pair brackets one kernel only.
inline std::atomic<int> g_pdl_off{0};

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_pdl_off.load(std::memory_order_relaxed) > 0 ? 0 : 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

using bf16 = __nv_bfloat16;

// Error carried from an internal call up to the C ABI.
struct Status {
  int code = AGN_OK;
  std::string msg;
  bool ok() const { return code == AGN_OK; }
  static Status Ok() { return Status{}; }
  static Status Err(int c, std::string m) { return Status{c, std::move(m)}; }
};

inline Status cuda_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return Status::Ok();
  return Status::Err(e == cudaErrorMemoryAllocation ? AGN_E_OOM : AGN_E_CUDA,
                     std::string(what) + ": " + cudaGetErrorString(e));
}

#define AGN_TRY_CUDA(expr)                                  \
  do {                                                      \
    cudaError_t e__ = (expr);                               \
    if (e__ != cudaSuccess) return ::agn::cuda_status(e__, #expr); \
  } while (0)

#define AGN_TRY(expr)             \
  do {                            \
    ::agn::Status s__ = (expr);   \
    if (!s__.ok()) return s__;    \
  } while (0)

// The host's table of device buffers for the bounds-checked build
// (bounds.cuh): buffers are added when allocated (or, for a standalone call,
// for its duration), the table is uploaded to every kernel translation unit
// before kernels run and the units' refusal counts are collected after.  In
// the normal build these do nothing.
#ifdef AGN_BOUNDS_CHECK
void bounds_add(const void* p, size_t bytes);
void bounds_remove(const void* p);
bool bounds_host_ok(const void* p, size_t bytes);
Status bounds_upload(cudaStream_t st);
Status bounds_collect(cudaStream_t st);
#else
inline void bounds_add(const void*, size_t) {}
inline void bounds_remove(const void*) {}
inline bool bounds_host_ok(const void*, size_t) { return true; }
inline Status bounds_upload(cudaStream_t) { return Status::Ok(); }
inline Status bounds_collect(cudaStream_t) { return Status::Ok(); }
#endif

constexpr int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }
constexpr int64_t ceil_div(int64_t x, int64_t a) { return (x + a - 1) / a; }

// Algorithm 1's local step on one parameter, in its two steps: the update
// g = -eta grad rounded to fp32, then theta + g rounded to fp32 (no fused
// multiply-add; the L2-add form of the dW kernel performs the same two
// roundings, so every path agrees bit for bit).
__device__ __forceinline__ float local_step(float theta, float eta, float grad) {
  return __fadd_rn(theta, __fmul_rn(-eta, grad));
}

// Padded shards (the tensor-core path's layer-1 operand and labels): worker
// w's shard of S dataset rows is stored as S + m rows, row r holding dataset
// row w S + (r mod S), so that the minibatch of local step `step` of slot z,
// rows (t m + j) mod S for j < m (t = slot_t0[z] + step, Algorithm 1's
// FetchNextMiniBatch), is the m consecutive rows starting at this row.
__device__ __forceinline__ int64_t batch_row0(const long long* slot_t0, int slot, int step,
                                              int m, int64_t S) {
  const unsigned long long t = (unsigned long long)(AGN_LD(slot_t0 + slot) + step);
  return (int64_t)((t * (unsigned long long)m) % (unsigned long long)S);
}

// x = q0 + q1 + q2 exactly, each a bf16 (round to nearest even): q0 keeps the
// leading 8 significant bits of x, q1 the next 8, q2 the last 8.  The two
// residuals are exact float subtractions (Sterbenz); x must not be so small
// that a piece falls below the smallest normal float.  The fp32 mode feeds
// the tensor cores with these pieces.
__device__ __forceinline__ void split3(float x, bf16& q0, bf16& q1, bf16& q2) {
  q0 = __float2bfloat16_rn(x);
  const float r1 = __fsub_rn(x, __bfloat162float(q0));
  q1 = __float2bfloat16_rn(r1);
  const float r2 = __fsub_rn(r1, __bfloat162float(q1));
  q2 = __float2bfloat16_rn(r2);
}

// ---------------------------------------------------------------------------
// Standalone commit + pull (kernel c)
// ---------------------------------------------------------------------------

// Commits handled by one launch of the fused commit+pull kernel: theta~ stays
// in registers across them and each keeps a per-thread norm accumulator.
constexpr int kMaxCommitsPerLaunch = 16;
// Pulls one launch may do in total.
constexpr int kMaxPullsPerLaunch = 256;

struct CommitPlan {
  int32_t n_commits;                       // <= kMaxCommitsPerLaunch
  int32_t worker[kMaxCommitsPerLaunch];    // accumulator committed by commit c
  int32_t pull_begin[kMaxCommitsPerLaunch + 1];
  int32_t pull_worker[kMaxPullsPerLaunch];
  int32_t norm_slot[kMaxCommitsPerLaunch]; // index of commit c in the norm output
  int32_t per_commit_scale;                // 1: commit c uses scale[c], else the launch's
  float scale[kMaxCommitsPerLaunch];
};

// Queue one fused launch for the commits of `plan` plus the partial-norm
// reduction.  partials: device double [kMaxCommitsPerLaunch * grid] (null: no
// norms); delta_norm: device float indexed by norm_slot (may be null).
// flag: device int set to 1 when a Delta is not finite (may be null).
Status launch_commit_pull(const CommitPlan& plan, float* theta_c, float* acc, float* replicas,
                          bf16* replicas_bf16, int64_t P, int64_t ld, float scale,
                          bool zero_acc, double* partials, int grid, float* delta_norm,
                          int* flag, cudaStream_t stream, bool norms = true,
                          int64_t piece_plane = 0,   // > 0: pulls write 3 pieces
                          bool elide = false);       // acc holds pull snapshots (no accumulators)
// The per-commit norm reduction of one launch of launch_commit_pull (when
// that launch was queued with norms = false).
Status launch_commit_norms(const CommitPlan& plan, const double* partials, int grid,
                           float* delta_norm, int* flag, cudaStream_t stream);

// Grid size used by the commit kernel for P parameters (a multiple of the SM
// count, capped by the work).
int commit_grid(int64_t P);

}  // namespace agn
