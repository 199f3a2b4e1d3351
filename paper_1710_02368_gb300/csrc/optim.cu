// Adam as the local optimizer of Algorithm 1 (its gradient line names Adam as
// an example of where g comes from): per worker and parameter, from the raw
// minibatch gradient gr of the local step t = 1, 2, ... (the worker's step
// counter, never reset),
//   m = beta1 m + (1 - beta1) gr,   v = beta2 v + (1 - beta2) gr^2,
//   g = -eta (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps),
//   a += g (unless the accumulator is elided),  theta_k += g,
// then the bf16 copy (or the three pieces) of theta_k.  m and v belong to the
// worker and persist across its commits.  One pass over the replica, 16-byte
// accesses; the bias corrections are computed once per block in double.
#include "mlp.cuh"

namespace agn {

namespace {

constexpr int kOptThreads = 256;

__device__ __forceinline__ void write_copy4(bf16* tb, int64_t plane, int64_t p, const float (&t)[4]) {
  if (plane > 0) {
    bf16 q[3][4];
#pragma unroll
    for (int e = 0; e < 4; ++e) split3(t[e], q[0][e], q[1][e], q[2][e]);
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      const __nv_bfloat162 lo = __halves2bfloat162(q[k][0], q[k][1]);
      const __nv_bfloat162 hi = __halves2bfloat162(q[k][2], q[k][3]);
      AGN_ST(reinterpret_cast<uint2*>(tb + k * plane + p),
             make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                        *reinterpret_cast<const uint32_t*>(&hi)));
    }
  } else {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(t[0], t[1]);
    const __nv_bfloat162 hi = __floats2bfloat162_rn(t[2], t[3]);
    AGN_ST(reinterpret_cast<uint2*>(tb + p),
           make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi)));
  }
}

__global__ void __launch_bounds__(kOptThreads) adam_kernel(const AdamArgs a) {
  pdl_wait_only();   // the next forward may read theta_k before its own wait
  const int z = blockIdx.y;
  const int w = AGN_LD(a.slot_worker + z);
  __shared__ float s_c1, s_c2;
  if (threadIdx.x == 0) {
    const double t = (double)(AGN_LD(a.slot_t0 + z) + a.step + 1);
    s_c1 = (float)(1.0 / (1.0 - pow((double)a.beta1, t)));
    s_c2 = (float)(1.0 / (1.0 - pow((double)a.beta2, t)));
  }
  __syncthreads();
  const float c1 = s_c1, c2 = s_c2;
  const float b1 = a.beta1, b2 = a.beta2, ob1 = 1.0f - a.beta1, ob2 = 1.0f - a.beta2;
  const int64_t base = (int64_t)w * a.ld;
  const int64_t n4 = a.P / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const int64_t p = base + 4 * i;
    const float4 g4 = AGN_LD(reinterpret_cast<const float4*>(a.grad + p));
    const float4 t4 = AGN_LD(reinterpret_cast<const float4*>(a.theta + p));
    float4 m4 = AGN_LD(reinterpret_cast<const float4*>(a.m + p));
    float4 v4 = AGN_LD(reinterpret_cast<const float4*>(a.v + p));
    const float gr[4] = {g4.x, g4.y, g4.z, g4.w};
    float mm[4] = {m4.x, m4.y, m4.z, m4.w}, vv[4] = {v4.x, v4.y, v4.z, v4.w};
    float th[4] = {t4.x, t4.y, t4.z, t4.w}, u[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      mm[e] = b1 * mm[e] + ob1 * gr[e];
      vv[e] = b2 * vv[e] + ob2 * (gr[e] * gr[e]);
      u[e] = -a.eta * (mm[e] * c1) / (sqrtf(vv[e] * c2) + a.eps);
      th[e] = th[e] + u[e];
    }
    AGN_ST(reinterpret_cast<float4*>(a.m + p), make_float4(mm[0], mm[1], mm[2], mm[3]));
    AGN_ST(reinterpret_cast<float4*>(a.v + p), make_float4(vv[0], vv[1], vv[2], vv[3]));
    AGN_ST(reinterpret_cast<float4*>(a.theta + p), make_float4(th[0], th[1], th[2], th[3]));
    if (a.acc) {
      const float4 c4 = AGN_LD(reinterpret_cast<const float4*>(a.acc + p));
      AGN_ST(reinterpret_cast<float4*>(a.acc + p),
             make_float4(c4.x + u[0], c4.y + u[1], c4.z + u[2], c4.w + u[3]));
    }
    if (a.theta_b) write_copy4(a.theta_b, a.piece_plane, p, th);
  }
  pdl_fence_exit();
}

}  // namespace

Status adam_step(const AdamArgs& a, int slots, int num_sms, cudaStream_t st) {
  if (slots <= 0) return Status::Ok();
  if (a.P % 4 || a.ld % 4) return Status::Err(AGN_E_INVALID, "Adam step needs P and ld % 4 == 0");
  const int64_t n4 = a.P / 4;
  const int per_slot = (int)std::max<int64_t>(
      1, std::min<int64_t>(ceil_div(n4, kOptThreads), ceil_div((int64_t)num_sms * 8, slots)));
  dim3 grid((unsigned)per_slot, (unsigned)slots);
  {
    auto kf = adam_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kOptThreads, 0, st, a));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

AGN_BOUNDS_UNIT(optim)

}  // namespace agn
