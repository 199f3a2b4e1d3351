// The output layer in one kernel: forward z = h W_L^T + b_L (Eq. 1 inner
// term), softmax cross-entropy (loss and dZ_L = (softmax(z) - onehot(y)) / m)
// and the output layer's dX, dZ_{L-1} = (dZ_L W_L) [h > 0].
//
// The output layer is narrow (d_L classes, at most 16 here), so a GEMM tile
// would leave the GPU idle.  Instead a block takes two samples with four warps
// each: it first stages W_L and the two input rows in shared memory with
// asynchronous 16-byte copies (all in flight at once); warp q of a sample then
// takes the inputs k = 32 q + lane (mod 128), keeps one partial dot product
// per class and folds it with a fixed shuffle tree; the four partials of a
// class are added in a fixed order by every warp of the sample, so all four
// hold the same z, softmax and dZ_L, and each writes its own inputs of
// dZ_{L-1}.  Results are deterministic.  The per-slot loss (mean over the
// minibatch) is summed in a fixed order by the last block of the slot to
// finish.
#include <mutex>
#include <set>
#include <utility>

#include "mlp.cuh"

namespace agn {

namespace {

constexpr int kHeadSplit = 4;                          // warps per sample
constexpr int kHeadSmemCap = 200 * 1024;               // dynamic shared memory per block
constexpr int kHeadThreads = 32 * kHeadSplit * kHeadSamples;

__device__ __forceinline__ float cvt(float v) { return v; }
__device__ __forceinline__ float cvt(bf16 v) { return __bfloat162float(v); }
template <typename T>
__device__ __forceinline__ T st_f(float v);
template <>
__device__ __forceinline__ float st_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ bf16 st_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// Start copying `count` elements of T from global to shared memory: 16-byte
// asynchronous copies (cp.async, no register round trip, so every row of the
// block is in flight at once) where both ends are aligned, element copies
// elsewhere.  The caller waits with cp.async.wait_all before its barrier.
template <typename T>
__device__ __forceinline__ void stage(T* dst, const T* src, int64_t count) {
  // bounds-checked build: a source row outside every known buffer is not copied
  if (!AGN_BOUNDS_OK(src, (unsigned int)(count * sizeof(T)))) {
    if (threadIdx.x == 0) AGN_BOUNDS_FAIL(src);
    return;
  }
  constexpr int kVec = 16 / sizeof(T);
  const bool aligned = ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0;
  if (aligned) {
    const int64_t nv = count / kVec;
    const uint4* s = reinterpret_cast<const uint4*>(src);
    uint4* d = reinterpret_cast<uint4*>(dst);
    for (int64_t i = threadIdx.x; i < nv; i += blockDim.x)
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                       static_cast<uint32_t>(__cvta_generic_to_shared(d + i))),
                   "l"(s + i)
                   : "memory");
    for (int64_t i = nv * kVec + threadIdx.x; i < count; i += blockDim.x) dst[i] = src[i];
  } else {
    for (int64_t i = threadIdx.x; i < count; i += blockDim.x) dst[i] = src[i];
  }
}
__device__ __forceinline__ void stage_wait() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// Eight consecutive elements (16-byte aligned) as floats: one 16-byte shared
// load of bf16 (a bf16 is the upper half of the float it stands for), two of
// floats.  st8 rounds eight floats to T and stores them (16 or 32 bytes).
__device__ __forceinline__ void ld8(const bf16* p, float (&v)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(w[i] << 16);
    v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
__device__ __forceinline__ void ld8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
__device__ __forceinline__ uint32_t bf16x2_bits(float lo, float hi) {
  const __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&t);
}
__device__ __forceinline__ void st8(bf16* p, const float (&v)[8]) {
  AGN_ST(reinterpret_cast<uint4*>(p),
         make_uint4(bf16x2_bits(v[0], v[1]), bf16x2_bits(v[2], v[3]), bf16x2_bits(v[4], v[5]),
                    bf16x2_bits(v[6], v[7])));
}
__device__ __forceinline__ void st8(float* p, const float (&v)[8]) {
  AGN_ST(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
  AGN_ST(reinterpret_cast<float4*>(p + 4), make_float4(v[4], v[5], v[6], v[7]));
}

template <typename T, int kMaxC>
__global__ void __launch_bounds__(kHeadThreads) head_kernel(const HeadArgs a) {
  extern __shared__ __align__(16) uint8_t head_smem[];
  __shared__ float red[kHeadSamples][kHeadSplit][kMaxC];
  __shared__ float ce_s[kHeadSamples];
  const int z = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sj = warp / kHeadSplit, q = warp % kHeadSplit;   // sample in block, input quarter
  const int j0 = blockIdx.x * kHeadSamples;
  const int K = a.K, C = a.C, m = a.m;
  const int nj = min(kHeadSamples, m - j0);
  const int w = AGN_LD(a.slot_worker + z);
  const int64_t Kp = (K + 7) / 8 * 8;   // padded row length in shared memory
  T* Ws = reinterpret_cast<T*>(head_smem);                  // [C][Kp]
  T* Hs = Ws + (int64_t)C * Kp;                             // [kHeadSamples][Kp]
  const T* Wg = static_cast<const T*>(a.W) + (int64_t)w * a.ld_param + a.woff;
  const T* Hg = static_cast<const T*>(a.H) + ((int64_t)z * m + j0) * K;
  // W_L was last written two or more launches back (this slot's output-layer
  // update of the previous local step, or a pull), so its copy starts before
  // waiting for the preceding kernel (programmatic dependent launch); the
  // input rows come from the preceding forward and wait for it
  for (int c = 0; c < C; ++c) stage(Ws + c * Kp, Wg + (int64_t)c * K, K);
  pdl_begin();
  for (int r = 0; r < nj; ++r) stage(Hs + r * Kp, Hg + (int64_t)r * K, K);
  stage_wait();
  __syncthreads();

  const bool active = sj < nj;
  const T* h = Hs + (int64_t)sj * Kp;
  constexpr int kStride = 32 * kHeadSplit;
  // K % 8 == 0: each lane takes eight consecutive inputs at a time (16-byte
  // shared loads, 16- or 32-byte global stores); else one input at a time
  const bool vec = K % 8 == 0;
  if (active) {
    float part[kMaxC];
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) part[c] = 0.f;
    if (vec) {
      for (int k0 = 8 * (32 * q + lane); k0 < K; k0 += 8 * kStride) {
        float hv[8];
        ld8(h + k0, hv);
#pragma unroll
        for (int c = 0; c < kMaxC; ++c) {
          if (c < C) {
            float wv[8];
            ld8(Ws + (int64_t)c * Kp + k0, wv);
#pragma unroll
            for (int i = 0; i < 8; ++i) part[c] = fmaf(hv[i], wv[i], part[c]);
          }
        }
      }
    } else {
      for (int k = 32 * q + lane; k < K; k += kStride) {
        const float hv = cvt(h[k]);
#pragma unroll
        for (int c = 0; c < kMaxC; ++c)
          if (c < C) part[c] = fmaf(hv, cvt(Ws[(int64_t)c * Kp + k]), part[c]);
      }
    }
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) {
      float v = part[c];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (lane == 0) red[sj][q][c] = v;
    }
  }
  __syncthreads();

  float ce = 0.f;
  if (active) {
    const int j = j0 + sj;
    const float* bias = a.theta + (int64_t)w * a.ld_param + a.boff;
    float zc[kMaxC];
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) {
      float v = 0.f;
#pragma unroll
      for (int r = 0; r < kHeadSplit; ++r) v += red[sj][r][c < C ? c : 0];
      zc[c] = c < C ? v + AGN_LD(bias + c) : -INFINITY;
    }
    const int y = a.x_shard > 0
                      ? AGN_LD(a.yb + (int64_t)w * (a.x_shard + m) +
                               batch_row0(a.slot_t0, z, a.step, m, a.x_shard) + j)
                      : AGN_LD(a.yb + (int64_t)z * m + j);
    float mx = zc[0];
#pragma unroll
    for (int c = 1; c < kMaxC; ++c) mx = fmaxf(mx, zc[c]);
    float s = 0.f, zy = 0.f;
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) {
      if (c < C) s += expf(zc[c] - mx);
      if (c == y) zy = zc[c];
    }
    ce = (logf(s) + mx) - zy;
    const float inv_s = 1.0f / s, inv_m = 1.0f / (float)m;
    float g[kMaxC];
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) {
      float p = c < C ? expf(zc[c] - mx) * inv_s : 0.f;
      if (c == y) p -= 1.0f;
      g[c] = p * inv_m;
    }
    if (q == 0) {
      T* dzl = static_cast<T*>(a.dZL) + ((int64_t)z * m + j) * a.ldz;
      bf16* dzp = a.dZL_pieces ? a.dZL_pieces + ((int64_t)z * m + j) * a.ldz : nullptr;
#pragma unroll
      for (int c = 0; c < kMaxC; ++c)
        if (c < C && lane == c) {
          const T gv = st_f<T>(g[c]);
          AGN_ST(dzl + c, gv);
          if (dzp) {
            bf16 q0, q1, q2;
            split3(cvt(gv), q0, q1, q2);
            AGN_ST(dzp + c, q0);
            AGN_ST(dzp + a.dZL_plane + c, q1);
            AGN_ST(dzp + 2 * a.dZL_plane + c, q2);
          }
        }
    }
    // dZ_{L-1}[j][k] = sum_c dZ_L[j][c] W_L[c][k], masked by h > 0 (W before its
    // update); skipped when the output layer is the only layer (dH null)
    T* dh = a.dH ? static_cast<T*>(a.dH) + ((int64_t)z * m + j) * K : nullptr;
    bf16* dp = a.dH_pieces ? a.dH_pieces + ((int64_t)z * m + j) * K : nullptr;
    for (int k0 = 8 * (32 * q + lane); vec && dh && k0 < K; k0 += 8 * kStride) {
      float v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = 0.f;
#pragma unroll
      for (int c = 0; c < kMaxC; ++c) {
        if (c < C) {
          float wv[8];
          ld8(Ws + (int64_t)c * Kp + k0, wv);
#pragma unroll
          for (int i = 0; i < 8; ++i) v[i] = fmaf(g[c], wv[i], v[i]);
        }
      }
      float hv[8], o[8];
      ld8(h + k0, hv);
#pragma unroll
      for (int i = 0; i < 8; ++i) o[i] = cvt(st_f<T>(hv[i] > 0.f ? v[i] : 0.f));
      st8(dh + k0, o);
      if (dp) {   // (fp32 mode: o holds the stored floats themselves)
        float q0[8], q1[8], q2[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          bf16 b0, b1, b2;
          split3(o[i], b0, b1, b2);
          q0[i] = __bfloat162float(b0);
          q1[i] = __bfloat162float(b1);
          q2[i] = __bfloat162float(b2);
        }
        st8(dp + k0, q0);
        st8(dp + a.dH_plane + k0, q1);
        st8(dp + 2 * a.dH_plane + k0, q2);
      }
    }
    for (int k = 32 * q + lane; !vec && dh && k < K; k += kStride) {
      float v0 = 0.f, v1 = 0.f;   // two chains: even and odd classes
#pragma unroll
      for (int c = 0; c < kMaxC; c += 2) {
        if (c < C) v0 = fmaf(g[c], cvt(Ws[(int64_t)c * Kp + k]), v0);
        if (c + 1 < C && c + 1 < kMaxC) v1 = fmaf(g[c + 1], cvt(Ws[(int64_t)(c + 1) * Kp + k]), v1);
      }
      const float v = v0 + v1;
      const T out = st_f<T>(cvt(h[k]) > 0.f ? v : 0.f);
      AGN_ST(dh + k, out);
      if (dp) {
        bf16 q0, q1, q2;
        split3(cvt(out), q0, q1, q2);
        AGN_ST(dp + k, q0);
        AGN_ST(dp + a.dH_plane + k, q1);
        AGN_ST(dp + 2 * a.dH_plane + k, q2);
      }
    }
  }
  if (q == 0 && lane == 0) ce_s[sj] = ce;
  __syncthreads();
  // per-slot loss: the last block of the slot to finish sums the blocks'
  // partials with a fixed assignment (thread t takes blocks t, t + 256, ...)
  // and a fixed shuffle tree, so the result does not depend on timing
  __shared__ int s_last;
  __shared__ float warp_sum[kHeadThreads / 32];
  const int nblk = gridDim.x;
  if (threadIdx.x == 0) {
    float part = 0.f;
    for (int r = 0; r < kHeadSamples; ++r) part += ce_s[r];
    AGN_ST(a.ce_partial + (int64_t)z * nblk + blockIdx.x, part);
    __threadfence();
    if (AGN_BOUNDS_OK(a.counter + z, 4)) {
      s_last = atomicAdd(a.counter + z, 1) == nblk - 1;
    } else {
      AGN_BOUNDS_FAIL(a.counter + z);
      s_last = 0;
    }
  }
  __syncthreads();
  if (!s_last) return;   // uniform across the block
  __threadfence();
  float v = 0.f;
  for (int b = threadIdx.x; b < nblk; b += blockDim.x)
    v += AGN_LDCG(a.ce_partial + (int64_t)z * nblk + b);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  if (lane == 0) warp_sum[warp] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float tot = 0.f;
    for (int q = 0; q < kHeadThreads / 32; ++q) tot += warp_sum[q];
    const float loss = tot / (float)m;
    float* lp = a.loss_parts + ((int64_t)AGN_LD(a.slot_commit + z) * a.lam + a.step) * a.loss_q;
    AGN_ST(lp, loss);
    for (int q = 1; q < a.loss_q; ++q) AGN_ST(lp + q, 0.f);
    if (!isfinite(loss)) atomicExch(a.flag, 1);
    AGN_ST(a.counter + z, 0);
  }
}

// The output layer's weight gradient and local update:
//   g[c][k] = sum_j dZ_L[j][c] h[j][k],   g_b[c] = sum_j dZ_L[j][c],
//   theta_k -= eta g, a_k += g, and the bf16 copy (or its three pieces).
// A block covers 32 inputs k of one slot with eight warps: dZ_L of the whole
// minibatch is staged in shared memory (asynchronous copies); warp w takes
// the samples j = w (mod 8), eight loads of h in flight per lane; the eight
// partials are added in a fixed order by the warp that owns the class
// (c = w mod 8), which then updates theta_k and a_k.  The bias gradient is
// summed by the last warp of the slot's first block (fixed shuffle tree).
constexpr int kDwGroups = 8;
template <typename T, int kMaxC>
__global__ void __launch_bounds__(32 * kDwGroups) head_dw_kernel(const HeadDwArgs a) {
  extern __shared__ __align__(16) uint8_t dw_smem[];
  float* red = reinterpret_cast<float*>(dw_smem);                      // [kDwGroups][kMaxC][32]
  T* dz = reinterpret_cast<T*>(red + kDwGroups * kMaxC * 32);           // [m][C]
  const int z = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = a.K, C = a.C, m = a.m;
  // dZ_L comes from the output head; when another launch ran in between
  // (a.dz_early), its copy starts before waiting for the preceding kernel
  if (a.dz_early) stage(dz, static_cast<const T*>(a.dZL) + (int64_t)z * m * C, (int64_t)m * C);
  pdl_begin();
  if (!a.dz_early) stage(dz, static_cast<const T*>(a.dZL) + (int64_t)z * m * C, (int64_t)m * C);
  stage_wait();
  __syncthreads();
  const int w = AGN_LD(a.slot_worker + z);
  const int k = blockIdx.x * 32 + lane;
  const T* hg = static_cast<const T*>(a.H) + (int64_t)z * m * K + k;
  float g[kMaxC];
#pragma unroll
  for (int c = 0; c < kMaxC; ++c) g[c] = 0.f;
  if (k < K) {
    constexpr int kU = 8;   // loads in flight per lane
    int j = warp;
    for (; j + (kU - 1) * kDwGroups < m; j += kU * kDwGroups) {
      float hv[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) hv[u] = cvt(AGN_LD(hg + (int64_t)(j + u * kDwGroups) * K));
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const T* dzj = dz + (j + u * kDwGroups) * C;
#pragma unroll
        for (int c = 0; c < kMaxC; ++c)
          if (c < C) g[c] = fmaf(cvt(dzj[c]), hv[u], g[c]);
      }
    }
    for (; j < m; j += kDwGroups) {
      const float hv = cvt(AGN_LD(hg + (int64_t)j * K));
      const T* dzj = dz + j * C;
#pragma unroll
      for (int c = 0; c < kMaxC; ++c)
        if (c < C) g[c] = fmaf(cvt(dzj[c]), hv, g[c]);
    }
  }
#pragma unroll
  for (int c = 0; c < kMaxC; ++c) red[(warp * kMaxC + c) * 32 + lane] = g[c];
  __syncthreads();
  float* theta = a.theta + (int64_t)w * a.ld_param;
  float* acc = a.acc ? a.acc + (int64_t)w * a.ld_param : nullptr;   // null: elided
  bf16* tb = a.theta_b ? a.theta_b + (int64_t)w * a.ld_param : nullptr;
  auto update = [&](int64_t p, float gr, float th, float ac) {
    const float t = local_step(th, a.eta, gr);
    AGN_ST(theta + p, t);
    if (acc) AGN_ST(acc + p, ac + gr);
    if (tb) {
      if (a.piece_plane > 0) {
        bf16 q0, q1, q2;
        split3(t, q0, q1, q2);
        AGN_ST(tb + p, q0);
        AGN_ST(tb + a.piece_plane + p, q1);
        AGN_ST(tb + 2 * a.piece_plane + p, q2);
      } else {
        AGN_ST(tb + p, __float2bfloat16_rn(t));
      }
    }
  };
  if (a.grad_out) {   // raw gradient out (the optimizer runs after)
    float* go = a.grad_out + (int64_t)w * a.ld_param;
    if (k < K) {
      for (int c = warp; c < C; c += kDwGroups) {
        float v = 0.f;
#pragma unroll
        for (int r = 0; r < kDwGroups; ++r) v += red[(r * kMaxC + c) * 32 + lane];
        AGN_ST(go + a.woff + (int64_t)c * K + k, v);
      }
    }
    if (blockIdx.x == 0 && warp == kDwGroups - 1) {
      for (int c = 0; c < C; ++c) {
        float v = 0.f;
        for (int j = lane; j < m; j += 32) v += cvt(dz[j * C + c]);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if (lane == 0) AGN_ST(go + a.boff + c, v);
      }
    }
    return;
  }
  if (k < K) {
    constexpr int kPer = (kMaxC + kDwGroups - 1) / kDwGroups;   // classes per warp
    float th[kPer], ac[kPer], gs[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) {   // loads first, all in flight
      const int c = warp + e * kDwGroups;
      if (c < C) {
        const int64_t p = a.woff + (int64_t)c * K + k;
        th[e] = AGN_LD(theta + p);
        ac[e] = acc ? AGN_LD(acc + p) : 0.f;
        float v = 0.f;
#pragma unroll
        for (int r = 0; r < kDwGroups; ++r) v += red[(r * kMaxC + c) * 32 + lane];
        gs[e] = v;
      }
    }
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int c = warp + e * kDwGroups;
      if (c < C) update(a.woff + (int64_t)c * K + k, gs[e], th[e], ac[e]);
    }
  }
  if (blockIdx.x == 0 && warp == kDwGroups - 1) {
    for (int c = 0; c < C; ++c) {
      float v = 0.f;
      for (int j = lane; j < m; j += 32) v += cvt(dz[j * C + c]);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (lane == 0)
        update(a.boff + c, v, AGN_LD(theta + a.boff + c), acc ? AGN_LD(acc + a.boff + c) : 0.f);
    }
  }
}

template <typename T>
size_t head_smem_bytes(int K, int C) {
  const size_t kp = (size_t)(K + 7) / 8 * 8;
  return (size_t)(C + kHeadSamples) * kp * sizeof(T);
}

// Opt a kernel in to the full dynamic shared-memory budget of the fused
// head (static shared memory comes on top, so the 48 KB default can fail
// even below 48 KB of dynamic memory); once per kernel and device.
Status allow_smem(const void* kern) {
  static std::mutex mu;
  static std::set<std::pair<int, const void*>> done;
  int dev = 0;
  AGN_TRY_CUDA(cudaGetDevice(&dev));
  std::lock_guard<std::mutex> lock(mu);
  if (done.count({dev, kern})) return Status::Ok();
  AGN_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kHeadSmemCap));
  done.insert({dev, kern});
  return Status::Ok();
}

}  // namespace

template <typename T>
bool head_fits(int K, int C) {
  return C <= kHeadMaxClasses && head_smem_bytes<T>(K, C) <= (size_t)kHeadSmemCap;
}

template <typename T>
Status head_forward_backward(const HeadArgs& a, int slots, cudaStream_t st) {
  if (!head_fits<T>(a.K, a.C)) return Status::Err(AGN_E_UNSUPPORTED, "output layer too wide");
  const size_t smem = head_smem_bytes<T>(a.K, a.C);
  // ten classes (the MNIST-shaped workloads) get an exact instantiation
  auto kern = a.C == 10 ? head_kernel<T, 10> : head_kernel<T, kHeadMaxClasses>;
  AGN_TRY(allow_smem(reinterpret_cast<const void*>(kern)));
  dim3 grid((unsigned)ceil_div(a.m, kHeadSamples), (unsigned)slots);
  {
    auto kf = kern;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kHeadThreads, smem, st, a));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

template <typename T>
Status head_backward_dw(const HeadDwArgs& a, int slots, cudaStream_t st) {
  if (a.C > kHeadMaxClasses) return Status::Err(AGN_E_UNSUPPORTED, "output layer too wide");
  const size_t smem = (size_t)kDwGroups * kHeadMaxClasses * 32 * sizeof(float) +
                      (size_t)a.m * a.C * sizeof(T);
  if (smem > (size_t)kHeadSmemCap)
    return Status::Err(AGN_E_UNSUPPORTED, "minibatch too large for the output dW");
  auto kern = a.C == 10 ? head_dw_kernel<T, 10> : head_dw_kernel<T, kHeadMaxClasses>;
  AGN_TRY(allow_smem(reinterpret_cast<const void*>(kern)));
  dim3 grid((unsigned)ceil_div(a.K, 32), (unsigned)slots);
  {
    auto kf = kern;
    AGN_TRY_CUDA(launch_pdl(kf, grid, 32 * kDwGroups, smem, st, a));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

template bool head_fits<float>(int, int);
template bool head_fits<bf16>(int, int);
template Status head_forward_backward<float>(const HeadArgs&, int, cudaStream_t);
template Status head_forward_backward<bf16>(const HeadArgs&, int, cudaStream_t);
template Status head_backward_dw<float>(const HeadDwArgs&, int, cudaStream_t);
template Status head_backward_dw<bf16>(const HeadDwArgs&, int, cudaStream_t);

AGN_BOUNDS_UNIT(head)

}  // namespace agn
