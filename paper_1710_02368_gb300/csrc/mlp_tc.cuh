// tcgen05 GEMMs of the bf16 mode (see mlp_tc.cu).
#pragma once

#include <cuda.h>

#include "mlp.cuh"

namespace agn {

// Arguments of one batched tcgen05 GEMM.  M, N, K are the per-slot GEMM
// sizes in the orientation of mlp_tc.cu; the A / B tensor maps are 3D
// (inner, rows, batch) with batch coordinate slot_worker[z] (by_worker) or z.
struct TcArgs {
  int M, N, K;
  const int* slot_worker;
  int a_by_worker, b_by_worker;
  int* err;                // set to 1 when a bounded wait gives up
  void* out;               // forward / dX output (bf16) [slots][N rows][ldo]
  int64_t ldo, out_bstride;
  const bf16* mask;        // dX: H_{l-1}, same layout as out
  int64_t mask_bstride;
  int relu;
  float* theta;            // fp32 master replicas [n][ld_param]
  float* acc;              // accumulators [n][ld_param]
  bf16* theta_b;           // bf16 working copies [n][ld_param]
  int64_t ld_param, woff, boff;
  float eta;
};

// Column tile used for an N: the tensor map of the operand that spans N
// must have this many rows (K-major) or 64-element chunks summing to it.
inline int tc_bn(int N) { return N <= 64 ? 64 : N <= 128 ? 128 : 256; }
constexpr int kTcDwBN = 256;

Status tc_init();
// 3D bf16 tensor map (inner, rows, batch), 128-byte swizzle, zero fill.
Status make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                         uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                         uint32_t box_inner, uint32_t box_rows);

// forward: w_k box {64, 128} over W (K-major); h_k box {64, tc_bn(m)} over H_{l-1}.
Status tc_forward(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args, int slots,
                  cudaStream_t st);
// dX: w_mn box {64, 64} over W (MN-major view); dz_k box {64, tc_bn(m)} over dZ_l.
Status tc_backward_dx(const CUtensorMap& w_mn, const CUtensorMap& dz_k, const TcArgs& args,
                      int slots, cudaStream_t st);
// dW: h_mn box {64, 64} over H_{l-1}; dz_mn box {64, 64} over dZ_l.
Status tc_backward_dw(const CUtensorMap& h_mn, const CUtensorMap& dz_mn, const TcArgs& args,
                      int slots, cudaStream_t st);
// Bias gradient of a hidden layer and its local update.
Status bias_update(const bf16* dz, int m, int d, int64_t dz_bstride, const int* slot_worker,
                   float* theta, float* acc, bf16* theta_b, int64_t ld_param, int64_t boff,
                   float eta, int slots, cudaStream_t st);

}  // namespace agn
