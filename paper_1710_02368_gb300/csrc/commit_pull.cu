// Kernel (c): fused commit + pull of the parameter server.
//
// For a run of consecutive commits (FIFO order, Eq. 2) the kernel streams the
// parameter vector once: each thread keeps its slice of theta~ in registers,
// and for every commit c of the launch takes the committing worker's
// accumulator, forms Delta = fp32(a * s) with s = fp32(-eta/lambda) (Eq. 1;
// the normalisation step of Algorithm 1; or a per-commit s = fp32(-eta /
// (tau_c + 1)) for the DynSGD rule), adds it to theta~ with a plain
// round-to-nearest add (no FMA, so the sequence is bit-reproducible), zeroes
// the accumulator (Algorithm 1 restarts a at 0) and writes theta~ into every
// replica that pulls at the new version (Pull).  theta~ is written back once.
// Bytes per launch: 8P (theta~) + C (4P read a + 4P zero a) + pulls * 4P
// (+ 2P per pull for the bf16 working copy).
//
// Per-commit ||Delta||_2: per-thread double partial sums, a warp-shuffle
// tree, a fixed-order sum over the warps of the block, one partial per block,
// then a second kernel sums the block partials in a fixed order.  The result
// is deterministic for a given grid size.
#include "generator.cuh"
#include "mlp.cuh"

namespace agn {

namespace {

constexpr int kThreads = 256;
// Two shapes of the same loop.  Long vectors (many float4 per thread): two
// float4 per thread and commit by commit, registers kept low for occupancy.
// Short vectors (a few float4 per thread, the MLP workloads' commits): one
// float4 per thread and the accumulator loads of eight commits in flight.
constexpr int kLongUnroll = 2, kLongGroup = 1;
constexpr int kShortUnroll = 1, kShortGroup = 8;

__device__ __forceinline__ float4 ld_stream(const float4* p) { return AGN_LDCS(p); }
__device__ __forceinline__ void st_stream(float4* p, float4 v) { AGN_STCS(p, v); }

__device__ __forceinline__ uint2 pack_bf16x4(float4 v) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y);
  __nv_bfloat162 hi = __floats2bfloat162_rn(v.z, v.w);
  uint2 r;
  r.x = *reinterpret_cast<uint32_t*>(&lo);
  r.y = *reinterpret_cast<uint32_t*>(&hi);
  return r;
}

// Three exact bf16 pieces of four floats, one uint2 per piece plane.
__device__ __forceinline__ void pack_pieces_x4(float4 v, uint2& p0, uint2& p1, uint2& p2) {
  const float x[4] = {v.x, v.y, v.z, v.w};
  bf16 q[3][4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    q[0][i] = __float2bfloat16_rn(x[i]);
    const float r1 = __fsub_rn(x[i], __bfloat162float(q[0][i]));
    q[1][i] = __float2bfloat16_rn(r1);
    q[2][i] = __float2bfloat16_rn(__fsub_rn(r1, __bfloat162float(q[1][i])));
  }
  uint2* out[3] = {&p0, &p1, &p2};
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    __nv_bfloat162 lo = __halves2bfloat162(q[k][0], q[k][1]);
    __nv_bfloat162 hi = __halves2bfloat162(q[k][2], q[k][3]);
    out[k]->x = *reinterpret_cast<uint32_t*>(&lo);
    out[k]->y = *reinterpret_cast<uint32_t*>(&hi);
  }
}

// kCopy: 0 = fp32 replicas only, 1 = plus a bf16 copy, 3 = plus the three
// exact bf16 pieces (planes `plane` elements apart) of the fp32 mode's
// tensor-core operands.
// kElide: no accumulators.  `acc` then holds each worker's snapshot theta_pull
// of its last pull, the committed quantity is fp32(theta_k - theta_pull) (the
// sum of the local updates) with s = fp32(1/lambda) (or fp32(1/(tau_c + 1)),
// or 1), and every pull also refreshes the snapshot.
template <int kCopy, bool kElide, int kUnroll, int kGroup>
__global__ void __launch_bounds__(kThreads)
commit_pull_kernel(const __grid_constant__ CommitPlan plan, float* __restrict__ theta_c,
                   float* __restrict__ acc, float* __restrict__ replicas,
                   bf16* __restrict__ rep_bf16, int64_t P, int64_t ld, float s, int zero_acc,
                   double* __restrict__ partials, int64_t plane) {
  pdl_begin();
  const int nc = plan.n_commits;
  double sq[kMaxCommitsPerLaunch];
#pragma unroll
  for (int c = 0; c < kMaxCommitsPerLaunch; ++c) sq[c] = 0.0;

  const int64_t n4 = P / 4;
  const int64_t stride = (int64_t)gridDim.x * kThreads * kUnroll;
  float4* th4 = reinterpret_cast<float4*>(theta_c);
  for (int64_t base = (int64_t)blockIdx.x * kThreads * kUnroll + threadIdx.x; base < n4;
       base += stride) {
    int64_t idx[kUnroll];
    bool live[kUnroll];
    float4 th[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      idx[u] = base + (int64_t)u * kThreads;
      live[u] = idx[u] < n4;
      if (live[u]) th[u] = AGN_LD(th4 + idx[u]);
    }
    // commits in groups of kGroup: every accumulator load of a group is in
    // flight before the group's dependent chain of adds (theta~ must see the
    // commits in FIFO order, the loads need not wait for each other)
#pragma unroll
    for (int c0 = 0; c0 < kMaxCommitsPerLaunch; c0 += kGroup) {
      if (c0 >= nc) break;
      float4 a[kGroup][kUnroll];
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        const int c = c0 + j;
        if (c >= nc) break;
        const int64_t row = (int64_t)plan.worker[c] * ld;
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          if (!live[u]) continue;
          if (kElide) {   // theta_k - theta_pull, the sum of the local updates
            const float4 tk = ld_stream(reinterpret_cast<const float4*>(replicas + row) + idx[u]);
            const float4 tp = ld_stream(reinterpret_cast<const float4*>(acc + row) + idx[u]);
            a[j][u] = make_float4(__fsub_rn(tk.x, tp.x), __fsub_rn(tk.y, tp.y),
                                  __fsub_rn(tk.z, tp.z), __fsub_rn(tk.w, tp.w));
          } else {
            a[j][u] = ld_stream(reinterpret_cast<const float4*>(acc + row) + idx[u]);
          }
        }
      }
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        const int c = c0 + j;
        if (c >= nc) break;
        const float sc = plan.per_commit_scale ? plan.scale[c] : s;
        const int64_t arow = (int64_t)plan.worker[c] * ld;
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          if (!live[u]) continue;
          float4 d;
          d.x = __fmul_rn(a[j][u].x, sc);
          d.y = __fmul_rn(a[j][u].y, sc);
          d.z = __fmul_rn(a[j][u].z, sc);
          d.w = __fmul_rn(a[j][u].w, sc);
          th[u].x = __fadd_rn(th[u].x, d.x);
          th[u].y = __fadd_rn(th[u].y, d.y);
          th[u].z = __fadd_rn(th[u].z, d.z);
          th[u].w = __fadd_rn(th[u].w, d.w);
          const float q = d.x * d.x + d.y * d.y + d.z * d.z + d.w * d.w;
          sq[c] += (double)q;
          if (!kElide && zero_acc)
            st_stream(reinterpret_cast<float4*>(acc + arow) + idx[u],
                      make_float4(0.f, 0.f, 0.f, 0.f));
        }
        for (int p = plan.pull_begin[c]; p < plan.pull_begin[c + 1]; ++p) {
          const int64_t row = (int64_t)plan.pull_worker[p] * ld;
#pragma unroll
          for (int u = 0; u < kUnroll; ++u) {
            if (!live[u]) continue;
            AGN_ST(reinterpret_cast<float4*>(replicas + row) + idx[u], th[u]);
            if (kElide) AGN_ST(reinterpret_cast<float4*>(acc + row) + idx[u], th[u]);
            if (kCopy == 1)
              AGN_ST(reinterpret_cast<uint2*>(rep_bf16 + row) + idx[u], pack_bf16x4(th[u]));
            if (kCopy == 3) {
              uint2 q0, q1, q2;
              pack_pieces_x4(th[u], q0, q1, q2);
              AGN_ST(reinterpret_cast<uint2*>(rep_bf16 + row) + idx[u], q0);
              AGN_ST(reinterpret_cast<uint2*>(rep_bf16 + plane + row) + idx[u], q1);
              AGN_ST(reinterpret_cast<uint2*>(rep_bf16 + 2 * plane + row) + idx[u], q2);
            }
          }
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (live[u]) AGN_ST(th4 + idx[u], th[u]);
  }

  // Tail of P % 4 elements: block 0, one element per thread.
  if (blockIdx.x == 0 && threadIdx.x < (int)(P - n4 * 4)) {
    const int64_t i = n4 * 4 + threadIdx.x;
    float t = AGN_LD(theta_c + i);
    for (int c = 0; c < nc; ++c) {
      float* ap = acc + (int64_t)plan.worker[c] * ld + i;
      const float av = kElide ? __fsub_rn(AGN_LD(replicas + (int64_t)plan.worker[c] * ld + i),
                                          AGN_LD(ap))
                              : AGN_LD(ap);
      float d = __fmul_rn(av, plan.per_commit_scale ? plan.scale[c] : s);
      t = __fadd_rn(t, d);
#pragma unroll
      for (int cc = 0; cc < kMaxCommitsPerLaunch; ++cc)
        if (cc == c) sq[cc] += (double)(d * d);
      if (!kElide && zero_acc) AGN_ST(ap, 0.f);
      for (int p = plan.pull_begin[c]; p < plan.pull_begin[c + 1]; ++p) {
        const int64_t row = (int64_t)plan.pull_worker[p] * ld;
        AGN_ST(replicas + row + i, t);
        if (kElide) AGN_ST(acc + row + i, t);
        if (kCopy == 1) AGN_ST(rep_bf16 + row + i, __float2bfloat16_rn(t));
        if (kCopy == 3) {
          const bf16 q0 = __float2bfloat16_rn(t);
          const float r1 = __fsub_rn(t, __bfloat162float(q0));
          const bf16 q1 = __float2bfloat16_rn(r1);
          AGN_ST(rep_bf16 + row + i, q0);
          AGN_ST(rep_bf16 + plane + row + i, q1);
          AGN_ST(rep_bf16 + 2 * plane + row + i,
                 __float2bfloat16_rn(__fsub_rn(r1, __bfloat162float(q1))));
        }
      }
    }
    AGN_ST(theta_c + i, t);
  }

  if (partials == nullptr) return;
  __shared__ double red[kThreads / 32][kMaxCommitsPerLaunch];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int c = 0; c < kMaxCommitsPerLaunch; ++c) {
    if (c < nc) {
      double v = sq[c];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (lane == 0) red[warp][c] = v;
    }
  }
  __syncthreads();
  if (threadIdx.x < nc) {
    double v = 0.0;
    for (int w = 0; w < kThreads / 32; ++w) v += red[w][threadIdx.x];
    AGN_ST(partials + (int64_t)threadIdx.x * gridDim.x + blockIdx.x, v);
  }
}

// norm[slot] = sqrt(sum_b partials[slot][b]) in a fixed order; one block per commit.
__global__ void __launch_bounds__(kThreads)
reduce_norms_kernel(const double* __restrict__ partials, int grid, const __grid_constant__ CommitPlan plan,
                    float* __restrict__ norms, int* __restrict__ flag) {
  pdl_begin();
  const int c = blockIdx.x;
  const int slot = plan.norm_slot[c];
  const double* row = partials + (int64_t)c * grid;
  double v = 0.0;
  for (int b = threadIdx.x; b < grid; b += kThreads) v += AGN_LD(row + b);
  __shared__ double red[kThreads];
  red[threadIdx.x] = v;
  __syncthreads();
  for (int w = kThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    float nrm = (float)sqrt(red[0]);
    if (norms) AGN_ST(norms + slot, nrm);
    if (flag && !isfinite(nrm)) atomicExch(flag, 1);
  }
}

int g_num_sms = 0;

}  // namespace

int commit_grid(int64_t P) {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_num_sms <= 0) g_num_sms = 148;
  }
  const int64_t need = ceil_div(std::max<int64_t>(P / 4, 1), (int64_t)kThreads * kLongUnroll);
  const int64_t cap = (int64_t)g_num_sms * 4;
  return (int)std::max<int64_t>(1, std::min(need, cap));
}

Status launch_commit_pull(const CommitPlan& plan, float* theta_c, float* acc, float* replicas,
                          bf16* replicas_bf16, int64_t P, int64_t ld, float scale, bool zero_acc,
                          double* partials, int grid, float* delta_norm, int* flag,
                          cudaStream_t stream, bool norms, int64_t piece_plane, bool elide) {
  if (plan.n_commits <= 0) return Status::Ok();
  const int z = zero_acc ? 1 : 0;
  auto go = [&](auto kern, bf16* rb, int64_t plane) {
    return launch_pdl(kern, grid, kThreads, 0, stream, plan, theta_c, acc, replicas, rb, P, ld,
                      scale, z, partials, plane);
  };
  // short vectors: at most 8 float4 per thread over the grid
  const bool shrt = P / 4 <= (int64_t)grid * kThreads * 8;
  cudaError_t e;
#define AGN_COMMIT_GO(C, E, RB, PL)                                                            \
  (shrt ? go(commit_pull_kernel<C, E, kShortUnroll, kShortGroup>, RB, PL)                       \
        : go(commit_pull_kernel<C, E, kLongUnroll, kLongGroup>, RB, PL))
  if (replicas_bf16 && piece_plane > 0)
    e = elide ? AGN_COMMIT_GO(3, true, replicas_bf16, piece_plane)
              : AGN_COMMIT_GO(3, false, replicas_bf16, piece_plane);
  else if (replicas_bf16)
    e = elide ? AGN_COMMIT_GO(1, true, replicas_bf16, 0) : AGN_COMMIT_GO(1, false, replicas_bf16, 0);
  else
    e = elide ? AGN_COMMIT_GO(0, true, nullptr, 0) : AGN_COMMIT_GO(0, false, nullptr, 0);
#undef AGN_COMMIT_GO
  AGN_TRY_CUDA(e);
  if (norms && partials && (delta_norm || flag))
    return launch_commit_norms(plan, partials, grid, delta_norm, flag, stream);
  return Status::Ok();
}

Status launch_commit_norms(const CommitPlan& plan, const double* partials, int grid,
                           float* delta_norm, int* flag, cudaStream_t stream) {
  if (plan.n_commits <= 0) return Status::Ok();
  {
    auto kf = reduce_norms_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, plan.n_commits, kThreads, 0, stream, partials,
                            grid, plan, delta_norm, flag));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

// ---------------------------------------------------------------------------
// Pulls outside a commit (version 0 at create, or at the start of a run)
// ---------------------------------------------------------------------------

namespace {

__global__ void __launch_bounds__(kThreads)
pull_kernel(const float* __restrict__ theta_c, float* __restrict__ replicas,
            bf16* __restrict__ rep_bf16, int64_t P, int64_t ld, const int* __restrict__ workers,
            int64_t plane, float* __restrict__ snapshot) {
  pdl_wait_only();   // the next forward may read the replicas before its own wait
  const int k = AGN_LD(workers + blockIdx.y);
  float* dst = replicas + (int64_t)k * ld;
  float* snap = snapshot ? snapshot + (int64_t)k * ld : nullptr;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < P; i += stride) {
    const float t = AGN_LD(theta_c + i);
    AGN_ST(dst + i, t);
    if (snap) AGN_ST(snap + i, t);
    if (rep_bf16) {
      const int64_t o = (int64_t)k * ld + i;
      if (plane > 0) {
        bf16 q0, q1, q2;
        split3(t, q0, q1, q2);
        AGN_ST(rep_bf16 + o, q0);
        AGN_ST(rep_bf16 + plane + o, q1);
        AGN_ST(rep_bf16 + 2 * plane + o, q2);
      } else {
        AGN_ST(rep_bf16 + o, __float2bfloat16_rn(t));
      }
    }
  }
  pdl_fence_exit();
}

__global__ void reduce_losses_kernel(const float* __restrict__ parts, int lambda, int q_per,
                                     int count, float* __restrict__ loss) {
  pdl_begin();
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= count) return;
  float s = 0.f;
  for (int i = 0; i < lambda; ++i) {
    const float* p = parts + ((int64_t)c * lambda + i) * q_per;
    float st = AGN_LD(p);
    for (int q = 1; q < q_per; ++q) st += AGN_LD(p + q);
    s += st;
  }
  AGN_ST(loss + c, s / (float)lambda);
}

}  // namespace

Status pull_replicas(const float* theta_c, float* replicas, bf16* replicas_bf16, int64_t P,
                     int64_t ld, const int* workers, int count, cudaStream_t st,
                     int64_t piece_plane, float* snapshot) {
  if (count <= 0) return Status::Ok();
  dim3 grid((unsigned)std::max(1, commit_grid(P) / std::max(1, count) + 1), (unsigned)count);
  {
    auto kf = pull_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kThreads, 0, st, theta_c,
                            replicas, replicas_bf16, P, ld, workers, piece_plane, snapshot));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

Status reduce_losses(const float* parts, int lambda, int q_per, int count, float* loss,
                     cudaStream_t st) {
  if (count <= 0) return Status::Ok();
  {
    auto kf = reduce_losses_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, (unsigned)ceil_div(count, 128), 128, 0, st, parts,
                            lambda, q_per, count, loss));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

// ---------------------------------------------------------------------------
// Inputs of the standalone commit workload, on the device (float32 variates)
// ---------------------------------------------------------------------------

namespace {

constexpr int kLnTermsF32 = 6;
constexpr int kCosTermsF32 = 12;

__device__ __forceinline__ float normal_f32(uint64_t k, uint64_t i) {
  using namespace gen;
  const float u1 = uniform_f32(draw(k, 2 * i));
  const float u2 = uniform_f32(draw(k, 2 * i + 1));
  const float x = __fsub_rn(1.0f, u1);
  int e;
  float f = frexpf(x, &e);
  if (f < (float)kSqrtHalf) {
    f = __fmul_rn(f, 2.0f);
    e -= 1;
  }
  const float s = __fdiv_rn(__fsub_rn(f, 1.0f), __fadd_rn(f, 1.0f));
  const float s2 = __fmul_rn(s, s);
  float p = __fdiv_rn(1.0f, (float)(2 * (kLnTermsF32 - 1) + 1));
  for (int j = kLnTermsF32 - 2; j >= 0; --j)
    p = __fadd_rn(__fmul_rn(p, s2), __fdiv_rn(1.0f, (float)(2 * j + 1)));
  const float ln = __fadd_rn(__fmul_rn((float)e, (float)kLn2), __fmul_rn(__fmul_rn(2.0f, s), p));
  const float r = __fsqrt_rn(__fmul_rn(-2.0f, ln));
  float c[kCosTermsF32];
  c[0] = 1.0f;
  for (int j = 1; j < kCosTermsF32; ++j) c[j] = __fdiv_rn(-c[j - 1], (float)((2 * j - 1) * (2 * j)));
  const float th = __fsub_rn(__fmul_rn(u2, (float)kTwoPi), (float)kPi);
  const float th2 = __fmul_rn(th, th);
  float q = c[kCosTermsF32 - 1];
  for (int j = kCosTermsF32 - 2; j >= 0; --j) q = __fadd_rn(__fmul_rn(q, th2), c[j]);
  return __fmul_rn(r, -q);
}

__global__ void fill_commit_inputs_kernel(float* __restrict__ theta_c, float* __restrict__ acc,
                                          float* __restrict__ replicas, int64_t P, int64_t ld,
                                          int n, uint64_t key_theta, uint64_t key_acc) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < P; i += stride) {
    const float t = normal_f32(key_theta, (uint64_t)i);
    theta_c[i] = t;
    for (int k = 0; k < n; ++k) {
      acc[(int64_t)k * ld + i] = __fmul_rn(normal_f32(key_acc, (uint64_t)k * (uint64_t)P + i), 0.1f);
      if (replicas) replicas[(int64_t)k * ld + i] = t;
    }
  }
}

}  // namespace

Status fill_commit_inputs(float* theta_c, float* acc, float* replicas, int64_t P, int64_t ld,
                          int n, uint64_t seed, cudaStream_t stream) {
  const int grid = commit_grid(P) * 2;
  {
    auto kf = fill_commit_inputs_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kThreads, 0, stream, theta_c,
                            acc, replicas, P, ld, n, gen::key(seed, gen::kCommitTheta),
                            gen::key(seed, gen::kCommitAcc)));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

AGN_BOUNDS_UNIT(commit)

}  // namespace agn
