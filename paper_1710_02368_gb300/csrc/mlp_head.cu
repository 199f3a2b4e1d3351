// The output layer in one kernel: forward z = h W_L^T + b_L (Eq. 1 inner
// term), softmax cross-entropy (loss and dZ_L = (softmax(z) - onehot(y)) / m)
// and the output layer's dX, dZ_{L-1} = (dZ_L W_L) [h > 0].
//
// The output layer is narrow (d_L classes, at most 16 here), so a GEMM tile
// would leave the GPU idle; instead one warp takes one sample.  A block first
// stages W_L and its samples' input rows in shared memory with asynchronous
// 16-byte copies (all in flight at once), then each warp's lanes stride over the d_{L-1}
// inputs, keep one partial dot product per class and combine them with a
// fixed shuffle tree, so results are deterministic.  The per-slot loss (mean
// over the minibatch) is summed in a fixed order by the last block of the
// slot to finish.
#include "mlp.cuh"

namespace agn {

namespace {

constexpr int kHeadWarps = 8;   // samples per block

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

template <typename T, int kMaxC>
__global__ void __launch_bounds__(kHeadWarps * 32) head_kernel(const HeadArgs a) {
  extern __shared__ __align__(16) uint8_t head_smem[];
  const int z = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j0 = blockIdx.x * kHeadWarps;
  const int K = a.K, C = a.C, m = a.m;
  const int nj = min(kHeadWarps, m - j0);
  const int w = a.slot_worker[z];
  const int64_t Kp = (K + 7) / 8 * 8;   // padded row length in shared memory
  T* Ws = reinterpret_cast<T*>(head_smem);                  // [C][Kp]
  T* Hs = Ws + (int64_t)C * Kp;                             // [kHeadWarps][Kp]
  const T* Wg = static_cast<const T*>(a.W) + (int64_t)w * a.ld_param + a.woff;
  const T* Hg = static_cast<const T*>(a.H) + ((int64_t)z * m + j0) * K;
  for (int c = 0; c < C; ++c) stage(Ws + c * Kp, Wg + (int64_t)c * K, K);
  for (int q = 0; q < nj; ++q) stage(Hs + q * Kp, Hg + (int64_t)q * K, K);
  stage_wait();
  __syncthreads();

  const float* bias = a.theta + (int64_t)w * a.ld_param + a.boff;
  __shared__ float ce_warp[kHeadWarps];
  float ce = 0.f;
  const int j = j0 + warp;
  if (warp < nj) {
    const T* h = Hs + (int64_t)warp * Kp;
    float part[kMaxC];
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) part[c] = 0.f;
    for (int k = lane; k < K; k += 32) {
      const float hv = cvt(h[k]);
#pragma unroll
      for (int c = 0; c < kMaxC; ++c)
        if (c < C) part[c] = fmaf(hv, cvt(Ws[(int64_t)c * Kp + k]), part[c]);
    }
    float zc[kMaxC];
#pragma unroll
    for (int c = 0; c < kMaxC; ++c) {
      float v = part[c];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      zc[c] = c < C ? v + bias[c] : -INFINITY;
    }
    const int y = a.yb[(int64_t)z * m + j];
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
    T* dzl = static_cast<T*>(a.dZL) + ((int64_t)z * m + j) * C;
#pragma unroll
    for (int c = 0; c < kMaxC; ++c)
      if (c < C && lane == c) dzl[c] = st_f<T>(g[c]);
    // dZ_{L-1}[j][k] = sum_c dZ_L[j][c] W_L[c][k], masked by h > 0 (W before its
    // update); skipped when the output layer is the only layer (dH null)
    T* dh = a.dH ? static_cast<T*>(a.dH) + ((int64_t)z * m + j) * K : nullptr;
    bf16* dp = a.dH_pieces ? a.dH_pieces + ((int64_t)z * m + j) * K : nullptr;
    for (int k = lane; dh && k < K; k += 32) {
      float v = 0.f;
#pragma unroll
      for (int c = 0; c < kMaxC; ++c)
        if (c < C) v = fmaf(g[c], cvt(Ws[(int64_t)c * Kp + k]), v);
      const T out = st_f<T>(cvt(h[k]) > 0.f ? v : 0.f);
      dh[k] = out;
      if (dp) {
        bf16 q0, q1, q2;
        split3(cvt(out), q0, q1, q2);
        dp[k] = q0;
        dp[a.dH_plane + k] = q1;
        dp[2 * a.dH_plane + k] = q2;
      }
    }
  }
  if (lane == 0) ce_warp[warp] = ce;
  __syncthreads();
  if (threadIdx.x == 0) {
    float part = 0.f;
    for (int q = 0; q < kHeadWarps; ++q) part += ce_warp[q];
    const int nblk = gridDim.x;
    a.ce_partial[(int64_t)z * nblk + blockIdx.x] = part;
    __threadfence();
    const int done = atomicAdd(a.counter + z, 1);
    if (done == nblk - 1) {   // last block of this slot: fixed-order sum
      __threadfence();
      float tot = 0.f;
      for (int b = 0; b < nblk; ++b) tot += *(volatile float*)(a.ce_partial + (int64_t)z * nblk + b);
      const float loss = tot / (float)m;
      a.loss_parts[(int64_t)a.slot_commit[z] * a.lam + a.step] = loss;
      if (!isfinite(loss)) atomicExch(a.flag, 1);
      a.counter[z] = 0;
    }
  }
}

template <typename T>
size_t head_smem_bytes(int K, int C) {
  const size_t kp = (size_t)(K + 7) / 8 * 8;
  return (size_t)(C + kHeadWarps) * kp * sizeof(T);
}

}  // namespace

template <typename T>
bool head_fits(int K, int C) {
  return C <= kHeadMaxClasses && head_smem_bytes<T>(K, C) <= 200 * 1024;
}

template <typename T>
Status head_forward_backward(const HeadArgs& a, int slots, cudaStream_t st) {
  if (!head_fits<T>(a.K, a.C)) return Status::Err(AGN_E_UNSUPPORTED, "output layer too wide");
  const size_t smem = head_smem_bytes<T>(a.K, a.C);
  auto kern = head_kernel<T, kHeadMaxClasses>;
  if (smem > 48 * 1024)
    AGN_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  dim3 grid((unsigned)ceil_div(a.m, kHeadWarps), (unsigned)slots);
  kern<<<grid, kHeadWarps * 32, smem, st>>>(a);
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

template bool head_fits<float>(int, int);
template bool head_fits<bf16>(int, int);
template Status head_forward_backward<float>(const HeadArgs&, int, cudaStream_t);
template Status head_forward_backward<bf16>(const HeadArgs&, int, cudaStream_t);

}  // namespace agn
