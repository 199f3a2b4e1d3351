// Batched MLP kernels (forward, softmax cross-entropy, backward with the
// fused local update) shared by the host scheduler.
#pragma once

#include "common.cuh"

namespace agn {

enum { kEpiFwd = 0, kEpiDX = 1, kEpiDW = 2, kEpiFwdHead = 3 };

// One batched GEMM over the slots of a wave: C[M x N] = sum_k A(m,k) B(k,n).
// Slot z reads operand X at X + (X_by_worker ? slot_worker[z] : z) * X_bstride.
//   forward : A = H_{l-1} [m][d_{l-1}] (k-major), B = W_l [d_l][d_{l-1}]
//             (k-major), M = m, N = d_l, K = d_{l-1};
//             out[j][f] = act(C + b_l[f])                       (Eq. 1 inner term)
//   dX      : A = dZ_l [m][d_l] (k-major), B = W_l (n-major), M = m,
//             N = d_{l-1}, K = d_l; out = C * [H_{l-1} > 0]
//   dW      : A = dZ_l (m-major: A(f,j) = dZ_l[j][f]), B = H_{l-1} (n-major),
//             M = d_l, N = d_{l-1}, K = m; theta_k -= eta C, a_k += C
//             (Algorithm 1's local step and accumulation; the bias gradient
//             sum_j dZ_l[j][f] is folded into the first column tile)
struct GemmArgs {
  int64_t M, N, K;
  const void* a;
  int64_t lda, a_bstride;
  int a_by_worker;
  const void* b;
  int64_t ldb, b_bstride;
  int b_by_worker;
  const int* slot_worker;
  // epilogue
  void* out;             // forward / dX output
  int64_t ldo, out_bstride;
  const void* mask;      // dX: H_{l-1}
  int64_t mask_bstride;
  int relu;
  float* theta;          // fp32 master replicas [n][ld_param]
  float* acc;            // accumulators [n][ld_param], or null (accumulator elided)
  bf16* theta_bf16;      // bf16 working copies or null
  int64_t piece_plane;   // > 0: theta_bf16 holds three exact bf16 pieces, planes this far apart
  int64_t ld_param;
  int64_t woff, boff;    // offsets of W_l and b_l in a replica
  float eta;
  float* grad_out;       // dW: store the raw gradient here ([n][ld_param]) instead of
                         // taking the local step; null = fused local step
};

template <typename T>
Status simt_forward(const GemmArgs& g, bool last, int slots, cudaStream_t st);
template <typename T>
Status simt_backward_dx(const GemmArgs& g, int slots, cudaStream_t st);
template <typename T>
Status simt_backward_dw(const GemmArgs& g, int slots, cudaStream_t st);
// Loss of slot z at local step `step` goes to loss_parts[slot_commit[z] * lam + step].
template <typename T>
Status softmax_xent(const float* Z, const int* yb, T* dZ, int m, int C, float* loss_parts,
                    const int* slot_commit, int lam, int step, int* flag, int slots,
                    cudaStream_t st);
template <typename T>
Status gather_batch(const T* X, const int* y, T* Xb, int* yb, int d0, int m, int64_t S,
                    const int* slot_worker, const long long* slot_t0, int step, int slots,
                    cudaStream_t st, bf16* pieces = nullptr, int64_t plane = 0,
                    int early = 0);

// Output layer fused (mlp_head.cu): forward, softmax cross-entropy and dX of
// layer L for d_L <= kHeadMaxClasses; kHeadSamples samples per block.
constexpr int kHeadMaxClasses = 16;
constexpr int kHeadSamples = 2;
struct HeadArgs {
  const void* H;           // H_{L-1} [slots][m][K] (T)
  const void* W;           // replica operand base [n][ld_param] (T); W_L at woff, [C][K]
  const float* theta;      // fp32 masters (bias b_L at boff)
  int64_t ld_param, woff, boff;
  int K, C, m;
  const int* slot_worker;
  const int* yb;           // labels [slots][m]
  void* dZL;               // out: dZ_L [slots][m][ldz] (T), ldz >= C
  int ldz;                 // row stride of dZ_L (columns C .. ldz - 1 are left alone)
  bf16* dZL_pieces;        // fp32 T only: also dZ_L's three exact bf16 pieces (planes
  int64_t dZL_plane;       // dZL_plane apart, same layout) for the tensor-core dW; null = no
  void* dH;                // out: dZ_{L-1} [slots][m][K] (T)
  bf16* dH_pieces;         // fp32 T only: also its three exact bf16 pieces (planes
  int64_t dH_plane;        // dH_plane apart) for tensor-core GEMMs; null = no
  float* ce_partial;       // [slots][ceil(m / kHeadSamples)] scratch
  int* counter;            // [slots], zero between launches
  float* loss_parts;       // [commit][lam][loss_q]: the step's loss in slot 0, zeros after
  int loss_q;
  const int* slot_commit;
  int lam, step;
  int* flag;
  // padded labels (batch_row0): x_shard = S > 0 reads yb [n][S + m] at the
  // slot's minibatch rows instead of yb [slots][m]
  const long long* slot_t0;
  int64_t x_shard;
};
template <typename T>
Status head_forward_backward(const HeadArgs& a, int slots, cudaStream_t st);
// dW of the output layer with its local update and accumulation (mlp_head.cu).
struct HeadDwArgs {
  const void* H;           // H_{L-1} [slots][m][K] (T)
  const void* dZL;         // dZ_L [slots][m][C] (T)
  const int* slot_worker;
  float* theta;            // fp32 master replicas [n][ld_param]
  float* acc;              // accumulators [n][ld_param], or null (accumulator elided)
  bf16* theta_b;           // bf16 copies (or piece 0 of three planes), or null
  int64_t piece_plane;     // > 0: three piece planes this far apart
  int64_t ld_param, woff, boff;
  int K, C, m;
  float eta;
  float* grad_out;         // store the raw gradient here instead of updating; null = update
  int dz_early;            // 1: dZ_L was written two or more launches back (may be read
                           // before the preceding launch completes)
};
template <typename T>
Status head_backward_dw(const HeadDwArgs& a, int slots, cudaStream_t st);
// The fused head takes this output layer (classes and shared-memory staging fit).
template <typename T>
bool head_fits(int K, int C);

// Adam as the local optimizer (optim.cu): from the raw gradients grad of the
// wave's slots, the moments m, v and theta_k (a_k += the step, unless acc is
// null; the bf16 copy or pieces of theta_k, unless theta_b is null).
struct AdamArgs {
  const float* grad;       // [n][ld] raw minibatch gradients of this local step
  float* theta;            // [n][ld] fp32 replicas
  float* acc;              // [n][ld] accumulators (of the steps), or null
  float* m;                // [n][ld] first moments
  float* v;                // [n][ld] second moments
  bf16* theta_b;           // bf16 copies / piece 0 of three planes, or null
  int64_t piece_plane;     // > 0: three pieces, planes this far apart
  int64_t P, ld;           // elements updated per replica (multiple of 4), row stride
  const int* slot_worker;
  const long long* slot_t0;   // the worker's step counter before this wave
  int step;                   // local step index within the wave
  float eta, beta1, beta2, eps;
};
Status adam_step(const AdamArgs& a, int slots, int num_sms, cudaStream_t st);

// Evaluation (mlp_eval.cu): per-sample loss / correctness / prediction of
// fp32 logits Z [rows][C] against labels y, and their fixed-order means
// (out[0] loss, out[1] accuracy).
Status eval_logits(const float* Z, const int* y, int rows, int C, float* loss, int* correct,
                   int* pred, cudaStream_t st);
Status eval_reduce(const float* loss, const int* correct, int64_t E, float* out,
                   cudaStream_t st);
// Eq. 4 on two sampled curves (host).
Status temporal_efficiency(const double* ta, const double* fa, int64_t na, const double* tb,
                           const double* fb, int64_t nb, double* out);

// Pull: copy theta~ into the replicas of `workers` (device list) and their bf16 copies.
// piece_plane > 0: replicas_bf16 holds three piece planes (fp32 mode on tensor cores).
// snapshot (accumulator elided): also copy theta~ into the workers' rows there.
Status pull_replicas(const float* theta_c, float* replicas, bf16* replicas_bf16, int64_t P,
                     int64_t ld, const int* workers, int count, cudaStream_t st,
                     int64_t piece_plane = 0, float* snapshot = nullptr);
// loss[c] = mean_i parts[c * lambda + i] for c < count.
// loss[c] = (1/lambda) sum_i sum_q parts[(c lambda + i) q_per + q] (fixed order).
Status reduce_losses(const float* parts, int lambda, int q_per, int count, float* loss,
                     cudaStream_t st);
// Device-side standalone-commit input generator.
Status fill_commit_inputs(float* theta_c, float* acc, float* replicas, int64_t P, int64_t ld,
                          int n, uint64_t seed, cudaStream_t stream);

}  // namespace agn
