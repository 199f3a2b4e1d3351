// Evaluation of the central variable on a held-out set (the accuracy-versus-
// time curves of the paper's experiments, Section 4) and the temporal
// efficiency of two such curves (Eq. 4).
//
// The forward pass reuses the CUDA-core fp32 GEMMs with theta~ as the weight
// operand of every row block (evaluation is not on the training hot path;
// theta~ has no bf16 copy).  Per sample: log-sum-exp with max subtraction,
// loss = lse - z_y, prediction = argmax with the lowest index on ties, as the
// teacher labels are defined.  Sums are taken in a fixed order (deterministic).
#include "mlp.cuh"

namespace agn {

namespace {

constexpr int kEvalThreads = 256;

__global__ void __launch_bounds__(kEvalThreads)
eval_logits_kernel(const float* __restrict__ Z, const int* __restrict__ y, int rows, int C,
                   float* __restrict__ loss, int* __restrict__ correct, int* __restrict__ pred) {
  pdl_begin();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= rows) return;
  const float* z = Z + (int64_t)i * C;
  float mx = AGN_LD(z);
  int am = 0;
  for (int c = 1; c < C; ++c) {
    const float zc = AGN_LD(z + c);
    if (zc > mx) {   // strict: the lowest index wins ties
      mx = zc;
      am = c;
    }
  }
  float s = 0.f;
  for (int c = 0; c < C; ++c) s += expf(AGN_LD(z + c) - mx);
  const int yi = AGN_LD(y + i);
  AGN_ST(loss + i, (logf(s) + mx) - AGN_LD(z + yi));
  AGN_ST(correct + i, am == yi ? 1 : 0);
  if (pred) AGN_ST(pred + i, am);
}

// out[0] = mean loss, out[1] = accuracy over E samples: thread t sums samples
// t, t + 256, ... in order (double), then a fixed shuffle / warp tree.
__global__ void __launch_bounds__(kEvalThreads)
eval_reduce_kernel(const float* __restrict__ loss, const int* __restrict__ correct, int64_t E,
                   float* __restrict__ out) {
  pdl_begin();
  __shared__ double ws[kEvalThreads / 32][2];
  double l = 0.0, c = 0.0;
  for (int64_t i = threadIdx.x; i < E; i += blockDim.x) {
    l += (double)AGN_LD(loss + i);
    c += (double)AGN_LD(correct + i);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    l += __shfl_xor_sync(0xffffffffu, l, off);
    c += __shfl_xor_sync(0xffffffffu, c, off);
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) {
    ws[warp][0] = l;
    ws[warp][1] = c;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double L = 0.0, Cc = 0.0;
    for (int w = 0; w < kEvalThreads / 32; ++w) {
      L += ws[w][0];
      Cc += ws[w][1];
    }
    AGN_ST(out, (float)(L / (double)E));
    AGN_ST(out + 1, (float)(Cc / (double)E));
  }
}

}  // namespace

Status eval_logits(const float* Z, const int* y, int rows, int C, float* loss, int* correct,
                   int* pred, cudaStream_t st) {
  if (rows <= 0) return Status::Ok();
  {
    auto kf = eval_logits_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, (unsigned)ceil_div(rows, kEvalThreads), kEvalThreads, 0, st, Z,
                            y, rows, C, loss, correct, pred));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

Status eval_reduce(const float* loss, const int* correct, int64_t E, float* out,
                   cudaStream_t st) {
  if (E <= 0) return Status::Err(AGN_E_INVALID, "empty evaluation set");
  {
    auto kf = eval_reduce_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, 1, kEvalThreads, 0, st, loss, correct, E, out));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

// Eq. 4: E(a, b) = int_0^m f_a dt / int_0^m f_b dt, m the shorter of the two
// curves' end times.  Each curve is the piecewise-linear interpolation of its
// samples (t non-decreasing, t >= 0), constant at its first value on
// [0, t_0]; the integrals are exact for that interpolation (trapezoids, the
// last one cut at m).
namespace {
double integral_to(const double* t, const double* f, int64_t n, double m) {
  double s = t[0] > 0.0 ? f[0] * std::min(t[0], m) : 0.0;
  for (int64_t i = 0; i + 1 < n && t[i] < m; ++i) {
    const double t0 = t[i], t1 = std::min(t[i + 1], m);
    if (t1 <= t0) continue;
    const double f1 = t[i + 1] > t0
                          ? f[i] + (f[i + 1] - f[i]) * ((t1 - t0) / (t[i + 1] - t0))
                          : f[i + 1];
    s += 0.5 * (f[i] + f1) * (t1 - t0);
  }
  return s;
}
}  // namespace

Status temporal_efficiency(const double* ta, const double* fa, int64_t na, const double* tb,
                           const double* fb, int64_t nb, double* out) {
  if (!ta || !fa || !tb || !fb || !out || na < 1 || nb < 1)
    return Status::Err(AGN_E_INVALID, "temporal efficiency needs two non-empty curves");
  for (int k = 0; k < 2; ++k) {
    const double* t = k ? tb : ta;
    const int64_t n = k ? nb : na;
    if (t[0] < 0.0) return Status::Err(AGN_E_INVALID, "negative time");
    for (int64_t i = 1; i < n; ++i)
      if (!(t[i] >= t[i - 1])) return Status::Err(AGN_E_INVALID, "times must not decrease");
  }
  const double m = std::min(ta[na - 1], tb[nb - 1]);
  if (!(m > 0.0)) return Status::Err(AGN_E_INVALID, "no shared training time");
  const double ib = integral_to(tb, fb, nb, m);
  if (ib == 0.0) return Status::Err(AGN_E_INVALID, "the second curve integrates to zero");
  *out = integral_to(ta, fa, na, m) / ib;
  return Status::Ok();
}

AGN_BOUNDS_UNIT(eval)

}  // namespace agn
