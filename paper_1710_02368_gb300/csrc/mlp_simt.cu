// Kernels (a) and (b) on CUDA cores: the batched-over-workers MLP forward,
// softmax cross-entropy, and backward with the fused local SGD step and
// gradient accumulation of Algorithm 1 (g = grad L; theta_k -= eta g; a_k += g).
//
// One launch covers every worker of a wave: grid.z indexes the wave's slots,
// and slot z reads and updates the replica of worker slot_worker[z].  All
// three GEMM shapes use one tiled kernel (64x64 tile, 16-deep k slices, 4x4
// outputs per thread); the element type T is float (fp32 mode) or bf16 (bf16
// mode: operands bf16, accumulation fp32, master weights fp32).
#include <algorithm>

#include "mlp.cuh"

namespace agn {

namespace {

constexpr int kBM = 64, kBN = 64, kBK = 16, kTM = 4, kTN = 4;
constexpr int kThreads = (kBM / kTM) * (kBN / kTN);   // 256

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<bf16>(bf16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// The low-precision copy of an updated weight: one bf16, or its three exact
// pieces (fp32 mode on tensor cores).
__device__ __forceinline__ void write_copy(bf16* tb, int64_t plane, int64_t p, float t) {
  if (plane > 0) {
    bf16 q0, q1, q2;
    split3(t, q0, q1, q2);
    AGN_ST(tb + p, q0);
    AGN_ST(tb + plane + p, q1);
    AGN_ST(tb + 2 * plane + p, q2);
  } else {
    AGN_ST(tb + p, __float2bfloat16_rn(t));
  }
}

// C[M x N] (+)= sum_k A(m, k) B(k, n) for one slot; see GemmArgs for layouts.
template <typename T, typename TO, bool kAKMajor, bool kBKMajor, int kEpi>
__global__ void __launch_bounds__(kThreads) gemm_simt_kernel(const GemmArgs g) {
  pdl_begin();
  __shared__ float As[kBK][kBM + 1];
  __shared__ float Bs[kBK][kBN + 1];
  const int z = blockIdx.z;
  const int w = AGN_LD(g.slot_worker + z);
  const int64_t m0 = (int64_t)blockIdx.y * kBM, n0 = (int64_t)blockIdx.x * kBN;
  const T* A = reinterpret_cast<const T*>(g.a) + (g.a_by_worker ? (int64_t)w : z) * g.a_bstride;
  const T* B = reinterpret_cast<const T*>(g.b) + (g.b_by_worker ? (int64_t)w : z) * g.b_bstride;
  const int tid = threadIdx.x;
  const int tx = tid % (kBN / kTN), ty = tid / (kBN / kTN);

  float acc[kTM][kTN];
#pragma unroll
  for (int i = 0; i < kTM; ++i)
#pragma unroll
    for (int j = 0; j < kTN; ++j) acc[i][j] = 0.f;
  float bsum = 0.f;   // bias gradient (kEpi == kEpiDW, first column tile)
  const bool do_bias = (kEpi == kEpiDW) && blockIdx.x == 0 && tid < kBM;

  for (int64_t k0 = 0; k0 < g.K; k0 += kBK) {
#pragma unroll
    for (int r = 0; r < (kBM * kBK) / kThreads; ++r) {
      const int e = tid + r * kThreads;
      int mm, kk;
      if (kAKMajor) { mm = e / kBK; kk = e % kBK; } else { kk = e / kBM; mm = e % kBM; }
      const int64_t gm = m0 + mm, gk = k0 + kk;
      float v = 0.f;
      if (gm < g.M && gk < g.K)
        v = to_f(AGN_LD(kAKMajor ? A + gm * g.lda + gk : A + gk * g.lda + gm));
      As[kk][mm] = v;
    }
#pragma unroll
    for (int r = 0; r < (kBN * kBK) / kThreads; ++r) {
      const int e = tid + r * kThreads;
      int nn, kk;
      if (kBKMajor) { nn = e / kBK; kk = e % kBK; } else { kk = e / kBN; nn = e % kBN; }
      const int64_t gn = n0 + nn, gk = k0 + kk;
      float v = 0.f;
      if (gn < g.N && gk < g.K)
        v = to_f(AGN_LD(kBKMajor ? B + gn * g.ldb + gk : B + gk * g.ldb + gn));
      Bs[kk][nn] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kBK; ++kk) {
      float a[kTM], b[kTN];
#pragma unroll
      for (int i = 0; i < kTM; ++i) a[i] = As[kk][ty + i * (kBM / kTM)];
#pragma unroll
      for (int j = 0; j < kTN; ++j) b[j] = Bs[kk][tx + j * (kBN / kTN)];
#pragma unroll
      for (int i = 0; i < kTM; ++i)
#pragma unroll
        for (int j = 0; j < kTN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (do_bias) {
#pragma unroll
      for (int kk = 0; kk < kBK; ++kk) bsum += As[kk][tid];
    }
    __syncthreads();
  }

  // Epilogues.
  float* theta = g.theta + (int64_t)w * g.ld_param;
  if (kEpi == kEpiFwd) {
    const float* bias = theta + g.boff;
    TO* out = reinterpret_cast<TO*>(g.out) + (int64_t)z * g.out_bstride;
#pragma unroll
    for (int i = 0; i < kTM; ++i) {
      const int64_t m = m0 + ty + i * (kBM / kTM);
      if (m >= g.M) continue;
#pragma unroll
      for (int j = 0; j < kTN; ++j) {
        const int64_t n = n0 + tx + j * (kBN / kTN);
        if (n >= g.N) continue;
        float v = acc[i][j] + AGN_LD(bias + n);
        if (g.relu) v = fmaxf(v, 0.f);
        AGN_ST(out + m * g.ldo + n, from_f<TO>(v));
      }
    }
  } else if (kEpi == kEpiDX) {
    const T* mask = reinterpret_cast<const T*>(g.mask) + (int64_t)z * g.mask_bstride;
    TO* out = reinterpret_cast<TO*>(g.out) + (int64_t)z * g.out_bstride;
#pragma unroll
    for (int i = 0; i < kTM; ++i) {
      const int64_t m = m0 + ty + i * (kBM / kTM);
      if (m >= g.M) continue;
#pragma unroll
      for (int j = 0; j < kTN; ++j) {
        const int64_t n = n0 + tx + j * (kBN / kTN);
        if (n >= g.N) continue;
        const float h = to_f(AGN_LD(mask + m * g.ldo + n));
        AGN_ST(out + m * g.ldo + n, from_f<TO>(h > 0.f ? acc[i][j] : 0.f));
      }
    }
  } else if (g.grad_out) {   // kEpiDW, raw gradient out (the optimizer runs after)
    float* go = g.grad_out + (int64_t)w * g.ld_param;
#pragma unroll
    for (int i = 0; i < kTM; ++i) {
      const int64_t m = m0 + ty + i * (kBM / kTM);
      if (m >= g.M) continue;
#pragma unroll
      for (int j = 0; j < kTN; ++j) {
        const int64_t n = n0 + tx + j * (kBN / kTN);
        if (n < g.N) AGN_ST(go + g.woff + m * g.N + n, acc[i][j]);
      }
    }
    if (do_bias && m0 + tid < g.M) AGN_ST(go + g.boff + m0 + tid, bsum);
  } else {   // kEpiDW: theta_k -= eta g, a_k += g (unless elided), bf16 copy refresh
    const bool has_a = g.acc != nullptr;
    float* a = has_a ? g.acc + (int64_t)w * g.ld_param : theta;
    bf16* tb = g.theta_bf16 ? g.theta_bf16 + (int64_t)w * g.ld_param : nullptr;
    // loads of all 16 outputs first, then the updates (memory-level parallelism)
    const float* __restrict__ th_in = theta;
    const float* __restrict__ a_in = a;
    float th[kTM][kTN], av[kTM][kTN];
#pragma unroll
    for (int i = 0; i < kTM; ++i) {
      const int64_t m = m0 + ty + i * (kBM / kTM);
#pragma unroll
      for (int j = 0; j < kTN; ++j) {
        const int64_t n = n0 + tx + j * (kBN / kTN);
        if (m < g.M && n < g.N) {
          const int64_t p = g.woff + m * g.N + n;
          th[i][j] = AGN_LDCS(th_in + p);
          av[i][j] = has_a ? AGN_LDCS(a_in + p) : 0.f;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < kTM; ++i) {
      const int64_t m = m0 + ty + i * (kBM / kTM);
      if (m >= g.M) continue;
#pragma unroll
      for (int j = 0; j < kTN; ++j) {
        const int64_t n = n0 + tx + j * (kBN / kTN);
        if (n >= g.N) continue;
        const int64_t p = g.woff + m * g.N + n;
        const float gr = acc[i][j];
        const float t = local_step(th[i][j], g.eta, gr);
        AGN_ST(theta + p, t);
        if (has_a) AGN_ST(a + p, av[i][j] + gr);
        if (tb) write_copy(tb, g.piece_plane, p, t);
      }
    }
    if (do_bias && m0 + tid < g.M) {
      const int64_t p = g.boff + m0 + tid;
      const float t = local_step(AGN_LD(theta + p), g.eta, bsum);
      AGN_ST(theta + p, t);
      if (has_a) AGN_ST(a + p, AGN_LD(a + p) + bsum);
      if (tb) write_copy(tb, g.piece_plane, p, t);
    }
  }
}

// Softmax cross-entropy on Z [m][C] (fp32) per slot: dZ = (softmax - onehot)/m,
// loss = mean_j (logsumexp(z_j) - z_j[y_j]), summed over the block in a fixed
// order.  One block per slot.
template <typename T>
__global__ void __launch_bounds__(128) softmax_xent_kernel(const float* __restrict__ Z,
                                                           const int* __restrict__ yb, T* dZ,
                                                           int m, int C, float* loss_parts,
                                                           const int* slot_commit, int lam,
                                                           int step, int* flag) {
  pdl_begin();
  const int z = blockIdx.x;
  const float* Zs = Z + (int64_t)z * m * C;
  T* dZs = dZ + (int64_t)z * m * C;
  const int* ys = yb + (int64_t)z * m;
  const float inv_m = 1.0f / (float)m;
  float part = 0.f;
  for (int j = threadIdx.x; j < m; j += blockDim.x) {
    const float* zr = Zs + (int64_t)j * C;
    float mx = AGN_LD(zr);
    for (int c = 1; c < C; ++c) mx = fmaxf(mx, AGN_LD(zr + c));
    float s = 0.f;
    for (int c = 0; c < C; ++c) s += expf(AGN_LD(zr + c) - mx);
    const int y = AGN_LD(ys + j);
    part += (logf(s) + mx) - AGN_LD(zr + y);
    const float inv_s = 1.0f / s;
    for (int c = 0; c < C; ++c) {
      float p = expf(AGN_LD(zr + c) - mx) * inv_s;
      if (c == y) p -= 1.0f;
      AGN_ST(dZs + (int64_t)j * C + c, from_f<T>(p * inv_m));
    }
  }
  __shared__ float red[128];
  red[threadIdx.x] = part;
  __syncthreads();
  for (int s = 64; s > 0; s >>= 1) {
    if (threadIdx.x < s) red[threadIdx.x] += red[threadIdx.x + s];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const float loss = red[0] * inv_m;
    AGN_ST(loss_parts + (int64_t)AGN_LD(slot_commit + z) * lam + step, loss);
    if (!isfinite(loss)) atomicExch(flag, 1);
  }
}

// Minibatch gather (FetchNextMiniBatch of Algorithm 1): slot z, row j reads
// dataset row k S + ((t0 + i) m + j) mod S of worker k = slot_worker[z].
// With `pieces` (fp32 mode on tensor cores) the rows are also written as three
// exact bf16 pieces, planes `plane` apart.
template <typename T>
__global__ void gather_kernel(const T* __restrict__ X, const int* __restrict__ y, T* Xb, int* yb,
                              int d0, int m, int64_t S, const int* slot_worker,
                              const long long* slot_t0, int step, bf16* pieces, int64_t plane) {
  pdl_begin();
  const int z = blockIdx.y, j = blockIdx.x;
  const int w = AGN_LD(slot_worker + z);
  const long long t = AGN_LD(slot_t0 + z) + step;
  const int64_t row = (int64_t)w * S + (int64_t)(((unsigned long long)t * m + j) % (unsigned long long)S);
  const T* src = X + row * d0;
  const int64_t o = ((int64_t)z * m + j) * d0;
  T* dst = Xb + o;
  for (int c = threadIdx.x; c < d0; c += blockDim.x) {
    const T v = AGN_LD(src + c);
    AGN_ST(dst + c, v);
    if (pieces) {
      bf16 q0, q1, q2;
      split3(to_f(v), q0, q1, q2);
      AGN_ST(pieces + o + c, q0);
      AGN_ST(pieces + plane + o + c, q1);
      AGN_ST(pieces + 2 * plane + o + c, q2);
    }
  }
  if (threadIdx.x == 0) AGN_ST(yb + (int64_t)z * m + j, AGN_LD(y + row));
}

// The same gather, four consecutive elements per thread (d_0 a multiple of
// 4): a block per minibatch row, one 16-byte (fp32) or 8-byte (bf16) load and
// store per thread and group, and 8-byte piece stores.
//
// early = 1: the destination buffers are not read by the preceding kernel
// (the tensor-core operand alternates between two buffers by local step, and
// the labels' last reader finished before this launch could start), so the
// rows are copied before waiting for the preceding kernel; the wait at the
// end keeps this launch's completion ordered after it for the next kernel.
template <typename T>
__global__ void __launch_bounds__(256) gather4_kernel(const T* __restrict__ X,
                                                      const int* __restrict__ y, T* Xb, int* yb,
                                                      int d0, int m, int64_t S,
                                                      const int* slot_worker,
                                                      const long long* slot_t0, int step,
                                                      bf16* pieces, int64_t plane, int early) {
  if (early) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  else pdl_begin();
  struct alignas(4 * sizeof(T)) Vec { T v[4]; };
  struct alignas(8) Piece4 { bf16 v[4]; };
  const int r = blockIdx.x;                 // slot * m + j
  const int z = r / m, j = r - z * m;
  const int w = AGN_LD(slot_worker + z);
  const long long t = AGN_LD(slot_t0 + z) + step;
  const int64_t row =
      (int64_t)w * S + (int64_t)(((unsigned long long)t * m + j) % (unsigned long long)S);
  const T* src = X + row * d0;
  const int64_t o = (int64_t)r * d0;
  for (int c = threadIdx.x * 4; c < d0; c += blockDim.x * 4) {
    const Vec v = AGN_LD(reinterpret_cast<const Vec*>(src + c));
    if (Xb) AGN_ST(reinterpret_cast<Vec*>(Xb + o + c), v);
    if (pieces) {
      Piece4 p0, p1, p2;
#pragma unroll
      for (int e = 0; e < 4; ++e) split3(to_f(v.v[e]), p0.v[e], p1.v[e], p2.v[e]);
      AGN_ST(reinterpret_cast<Piece4*>(pieces + o + c), p0);
      AGN_ST(reinterpret_cast<Piece4*>(pieces + plane + o + c), p1);
      AGN_ST(reinterpret_cast<Piece4*>(pieces + 2 * plane + o + c), p2);
    }
  }
  if (threadIdx.x == 0) AGN_ST(yb + r, AGN_LD(y + row));
  if (early) asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <typename T, typename TO, bool kAK, bool kBK, int kEpi>
Status launch_gemm(const GemmArgs& g, int slots, cudaStream_t st) {
  dim3 grid((unsigned)ceil_div(g.N, kBN), (unsigned)ceil_div(g.M, kBM), (unsigned)slots);
  {
    auto kf = gemm_simt_kernel<T, TO, kAK, kBK, kEpi>;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kThreads, 0, st, g));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

}  // namespace

template <typename T>
Status simt_forward(const GemmArgs& g, bool last, int slots, cudaStream_t st) {
  if (last) return launch_gemm<T, float, true, true, kEpiFwd>(g, slots, st);
  return launch_gemm<T, T, true, true, kEpiFwd>(g, slots, st);
}
template <typename T>
Status simt_backward_dx(const GemmArgs& g, int slots, cudaStream_t st) {
  return launch_gemm<T, T, true, false, kEpiDX>(g, slots, st);
}
template <typename T>
Status simt_backward_dw(const GemmArgs& g, int slots, cudaStream_t st) {
  return launch_gemm<T, T, false, false, kEpiDW>(g, slots, st);
}
template <typename T>
Status softmax_xent(const float* Z, const int* yb, T* dZ, int m, int C, float* loss_parts,
                    const int* slot_commit, int lam, int step, int* flag, int slots,
                    cudaStream_t st) {
  {
    auto kf = softmax_xent_kernel<T>;
    AGN_TRY_CUDA(launch_pdl(kf, slots, 128, 0, st, Z,
                            yb, dZ, m, C, loss_parts, slot_commit, lam, step, flag));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}
template <typename T>
Status gather_batch(const T* X, const int* y, T* Xb, int* yb, int d0, int m, int64_t S,
                    const int* slot_worker, const long long* slot_t0, int step, int slots,
                    cudaStream_t st, bf16* pieces, int64_t plane, int early) {
  const bool vec = d0 % 4 == 0 && plane % 4 == 0 &&
                   ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(Xb) |
                     reinterpret_cast<uintptr_t>(pieces)) & 15) == 0;
  if (slots <= 0 || m <= 0) return Status::Ok();
  if (vec) {
    const int threads = (int)std::min<int64_t>(256, round_up((int64_t)d0 / 4, 32));
    {
      auto kf = gather4_kernel<T>;
      AGN_TRY_CUDA(launch_pdl(kf, slots * m, threads, 0, st, X,
                              y, Xb, yb, d0, m, S, slot_worker, slot_t0, step, pieces, plane,
                              early));
    }
  } else {
    if (early) return Status::Err(AGN_E_INVALID, "internal: early gather needs d_0 % 4 == 0");
    dim3 grid((unsigned)m, (unsigned)slots);
    {
      auto kf = gather_kernel<T>;
      AGN_TRY_CUDA(launch_pdl(kf, grid, 128, 0, st, X,
                              y, Xb, yb, d0, m, S, slot_worker, slot_t0, step, pieces, plane));
    }
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

#define AGN_INST(T)                                                                          \
  template Status simt_forward<T>(const GemmArgs&, bool, int, cudaStream_t);                 \
  template Status simt_backward_dx<T>(const GemmArgs&, int, cudaStream_t);                   \
  template Status simt_backward_dw<T>(const GemmArgs&, int, cudaStream_t);                   \
  template Status softmax_xent<T>(const float*, const int*, T*, int, int, float*, const int*, \
                                  int, int, int*, int, cudaStream_t);                        \
  template Status gather_batch<T>(const T*, const int*, T*, int*, int, int, int64_t,          \
                                  const int*, const long long*, int, int, cudaStream_t,       \
                                  bf16*, int64_t, int);
AGN_INST(float)
AGN_INST(bf16)
#undef AGN_INST

AGN_BOUNDS_UNIT(simt)

}  // namespace agn
