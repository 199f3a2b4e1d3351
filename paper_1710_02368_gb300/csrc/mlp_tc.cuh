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
  const void* mask;        // dX: H_{l-1}, same layout and type as out
  int64_t mask_bstride;
  int relu;
  float* theta;            // fp32 master replicas [n][ld_param]
  float* acc;              // accumulators [n][ld_param]
  bf16* theta_b;           // bf16 working copies [n][ld_param] (split mode: piece 0 of
                           // three planes [3][n][ld_param])
  int64_t ld_param, woff, boff;
  int64_t piece_plane;     // split mode: elements between weight piece planes
  float eta;
  bf16* out_pieces;        // split mode, forward / dX: also write the output's three
  int64_t out_plane;       // pieces here (same index, planes out_plane apart); null = no
  // forward / dX split K: ksplit CTAs share an output tile, each a contiguous
  // range of ceil(KT / ksplit) k steps (none empty); each stores its partial
  // sums to part ([tile][rank][BN][128] fp32) and the last to arrive (counter
  // per tile, zero between launches) adds them in rank order and runs the
  // epilogue.  ksplit <= 1: one CTA per tile.
  int ksplit;
  float* part;
  int* counter;
  // The per-tile arrival counters (and the fused output layer's) alternate
  // between two arrays by launch: CTA 0 of a launch clears, after its
  // dependency wait, the array the previous launch used (null = none), so no
  // launch has to count its CTAs out to reset its own.
  int* counter_clear;
  int counter_clear_n;
  // dW: store the raw gradient at grad_out [n][ld_param] (same layout as the
  // replicas) instead of taking the local step (the optimizer runs after);
  // null = fused local step
  float* grad_out;
  // Forward of the last hidden layer with the output layer fused into its
  // epilogue (tc_forward_head): the d_L <= 16 logits of every sample from the
  // CTAs' partial sums over their 128 features, softmax cross-entropy, dZ_L and
  // dZ_{L-1} = (dZ_L W_L) [H_{L-1} > 0].
  int64_t head_woff, head_boff;   // W_L [C][M] and b_L [C] in the fp32 replicas
  int head_C;
  const int* yb;                  // labels [slots][m]
  void* dzl;                      // out: dZ_L [slots][m][ldz] (activation type)
  int ldz;
  bf16* dzl_pieces;               // split mode: its pieces, planes dzl_plane apart
  int64_t dzl_plane;
  void* dh;                       // out: dZ_{L-1} [slots][m][M]
  bf16* dh_pieces;                // split mode: its pieces, planes dh_plane apart
  int64_t dh_plane;
  float* head_part;               // [slots][ceil(m / 32)][M tiles][32][16] partial logits
  int* head_counter;              // [slots][ceil(m / 32)], zero at launch
  int* head_counter_clear;        // the other array, cleared by CTA 0 (null = none)
  int head_counter_clear_n;
  float* loss_parts;              // [commit][lambda][ceil(m / 32)]: per 32-sample chunk
                                  // its cross-entropy sum / m
  const int* slot_commit;
  int lam, step;
  int* nonfinite;                 // set to 1 for a non-finite loss
  // Test hook of the bounded waits (agn_debug_waits): wait_ns > 0 bounds the
  // split-K and output-layer waits by that many nanoseconds instead of 2 s;
  // withhold_rank = r + 1 makes split-K rank r withhold its arrival on the
  // tile counter (0 = none), so that the ranks waiting for it give up.
  uint64_t wait_ns;
  int withhold_rank;
  // Padded shards (batch_row0): x_shard = S > 0 makes the layer-1 operand
  // (the forward's B, dW's A of layer 1) rows of the padded-shard maps at the
  // slot's minibatch row, batch coordinate the worker; and labels come from
  // yb = the padded labels [n][S + m] at the same rows.  x_b_direct: this
  // launch's B operand is layer 1's (forward of layer 1).
  const long long* slot_t0;
  int64_t x_shard;
  int x_b_direct;
  // 1: one 128-row tile per CTA even where two would share the B stages
  // (the bf16 forward and dX of full waves)
  int one_row_tile;
  // dW: 1 reads a_k's chunks through the parameter ring and stores a_k + g;
  // 0 adds g to a_k in the L2 (red.add) and keeps the ring for theta_k
  int acc_ring;
  // forward / dX: 1 requests no weight stage before the dependency wait
  int no_a_prefetch;
};

// Column tile used for an N: the tensor map of the operand that spans N
// must have this many rows (K-major) or 64-element chunks summing to it.
inline int tc_bn(int N) { return N <= 64 ? 64 : N <= 128 ? 128 : 256; }
constexpr int kTcSplitBK = 32;      // forward / dX k per stage, split (fp32) mode
constexpr int kTcDwBN = 256;        // dW column tile, bf16 mode
constexpr int kTcDwBNSplit = 128;   // dW column tile, split (fp32) mode

Status tc_init();
// 3D bf16 tensor map (inner, rows, batch), 128-byte swizzle, zero fill.
Status make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                         uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                         uint32_t box_inner, uint32_t box_rows);
// 3D fp32 tensor map (inner, rows, batch), zero fill; no swizzle, or the
// 128-byte swizzle (box rows of 32 floats) when swizzle128.
Status make_tmap_f32_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                        uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                        uint32_t box_inner, uint32_t box_rows, bool swizzle128 = false);
// 4D bf16 tensor map (inner, rows, batch, piece) over three piece planes.
Status make_tmap_bf16_4d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                         uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                         uint64_t piece_stride_elems, uint32_t box_inner, uint32_t box_rows);

// split = false: bf16 operands (3D maps), bf16 activations.
// split = true : fp32 operands as three exact bf16 pieces (4D maps), fp32
//                activations; dW writes the three pieces of the new weights.
// forward: w_k box {64, 128} over W (K-major); h_k box {64, bn} over H_{l-1},
// bn = tc_bn(N) the column tile.  Small waves split K instead (args.ksplit).
Status tc_forward(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args, int slots,
                  cudaStream_t st, bool split, int bn);
// dX: w_mn box {64, 64} over W (MN-major view); dz_k box {64, bn} over dZ_l.
// The forward GEMM of the last hidden layer with the output layer fused
// (args.head_* set, args.relu = 1).  Needs every CTA of the launch resident at
// once; when the launch would exceed the SMs nothing is queued and *launched
// is false (the caller runs the forward and the output head separately).
Status tc_forward_head(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args,
                       int slots, cudaStream_t st, bool split, int bn, int num_sms,
                       bool* launched);
Status tc_backward_dx(const CUtensorMap& w_mn, const CUtensorMap& dz_k, const TcArgs& args,
                      int slots, cudaStream_t st, bool split, int bn);
// One hidden layer of a dW launch: h_mn box {64, kBK} over H_{l-1}; dz_mn box
// {64, kBK} over dZ_l (kBK = 64 samples, 32 in the split mode); theta / acc
// fp32 maps (d_{l-1}, d_l, n) over the
// layer's weights in the replicas and the accumulators, box {128, 32}, no
// swizzle.  M = d_{l-1}, N = d_l.
struct DwLayerMaps {
  const CUtensorMap *h_mn, *dz_mn, *theta, *acc;
  int M, N;
  int64_t woff, boff;
  int a_direct = 0;   // h_mn is a padded-shard map (layer 1; args.x_shard > 0)
};
// dW with the local step and accumulation of the weights and biases of all
// `layers` in one persistent launch (mlp_tc_dw.cu, grid min(tiles, num_sms)).
// args supplies slot_worker, err, theta, acc, theta_b, ld_param, piece_plane,
// eta and K = m; its per-layer fields are ignored.
Status tc_backward_dw(const DwLayerMaps* layers, int n_layers, const TcArgs& args, int slots,
                      cudaStream_t st, bool split, int num_sms);
// The earlier non-persistent dW kernel (mlp_tc.cu): one 128 x BN tile per CTA,
// two CTAs per SM, theta_k and a_k loaded into registers by the epilogue.
Status tc_backward_dw_tiled(const CUtensorMap& h_mn, const CUtensorMap& dz_mn, const TcArgs& args,
                            int slots, cudaStream_t st, bool split);
// Bias gradient of a hidden layer and its local update (dz: bf16, or fp32 when split).
Status bias_update(const void* dz, int m, int d, int64_t dz_bstride, const int* slot_worker,
                   float* theta, float* acc, bf16* theta_b, int64_t ld_param, int64_t boff,
                   float eta, int slots, cudaStream_t st, bool split, int64_t piece_plane);
// out[p * plane + i] = piece p of x[i], p < 3.
Status split_pieces(const float* x, bf16* out, int64_t count, int64_t plane, cudaStream_t st);

}  // namespace agn
