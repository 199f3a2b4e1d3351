// Kernel (b), weight-gradient half, on the tensor cores: D = H_{l-1}^T dZ_l
// for every slot of a wave and every hidden layer in one launch, fused with
// Algorithm 1's local step and accumulation (theta_k -= eta g, a_k += g, the
// bf16 copy of theta_k) for the weights and the biases.
//
// The GEMM is tiny next to its epilogue (K = m samples against 18-22 bytes
// of fp32 master weight and accumulator traffic per parameter), so the kernel
// is laid out around the parameter stream, not the MMA:
//
//   warp 0     operand producer: per tile, the GEMM operands (H^T and dZ^T
//              boxes, MN-major, 128-byte swizzle) into a ring of stages, as
//              fast as the MMA frees them, so the next tile's GEMM runs while
//              the current tile's epilogue drains.
//   warp 10    parameter producer: each tile's theta_k rows (and a_k's, for
//              waves whose accumulators exceed 64 MB), 32 output features x
//              128 inputs per chunk, into a second ring.  Each slot is
//              refilled as soon as it frees, so DRAM reads of the next chunks
//              (and of the next tile) are in flight while the current one is
//              updated.  Smaller waves add g to a_k in the L2 (red.add) and
//              keep twice the theta_k chunks in flight.
//   warp 1     MMA issuer (one thread) and TMEM owner.  Two accumulators
//              (double buffer): the GEMM of the next tile runs while the
//              epilogue drains this one.
//   warps 2-9  epilogue.  Warp w reads TMEM lanes 32 (w % 4) .. + 31, i.e.
//              32 consecutive inputs k of the tile, and 16 of the 32 features
//              of a chunk; it transposes them through shared memory so that
//              each lane updates four consecutive inputs of a feature at a
//              time (16-byte reads of theta_k and a_k from the chunk, 16-byte
//              coalesced stores).
//
// Bias gradients ride along: a layer with d_{l-1} = M inputs gets M + 1 GEMM
// rows, row M of H^T being all ones (written into the staged A tile by the
// MMA warp, over the zero fill of the out-of-range row), so D[M][f] =
// sum_j dZ_l[j][f] = g_b[f]; the epilogue updates b_l and its accumulator
// from that row, with their 32 values per chunk copied in by the producer.
//
// The local step rounds as Algorithm 1 computes it: g = fp32(-eta grad), then
// theta_k = fp32(theta_k + g) (local_step).
//
// The kernel is persistent (one CTA per SM: the rings take 210 KB of shared
// memory and the accumulators all 512 TMEM columns); tiles (layer, slot,
// feature tile, input tile) are dealt out round-robin with input tiles
// fastest, so neighbouring CTAs stream neighbouring parts of the same weight
// rows.  Every wait is bounded (2 s of global time): on expiry the CTA sets
// *err, stops issuing, drains its own copies and MMAs (bounded), frees TMEM
// and returns.
#include <cuda.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <set>

#include "mlp.cuh"
#include "mlp_tc.cuh"
#include "tc_ptx.cuh"

namespace agn {

namespace {

constexpr int kWarps = 11;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kCF = 32;                        // output features per parameter chunk
constexpr int kChunkBytes = kCF * 128 * 4;     // one fp32 chunk: 32 rows x 128 inputs
constexpr int kBiasHalf = kCF * 4;            // b_l (or its accumulator) for one chunk
constexpr uint64_t kWaitNs = 2000000000ull;    // 2 s
constexpr int kThrottleTiles = 8;              // tiles per CTA from which operands wait for chunks

// kBK samples per stage: one TMA box is 64 MN-elements x kBK samples of bf16
// (kBK rows of 128 bytes, 128-byte swizzle); A = two boxes (128 inputs),
// B = BN / 64 boxes.
// kMode: kDwUpdRed = the local step and accumulation, theta_k per chunk
// through the ring (6 slots in flight) and a_k += g as L2 adds (red.add,
// nothing read back into the SM); kDwUpdAcc = the same with a_k's chunk read
// through the ring beside theta_k's and stored back (3 slots); kDwUpd = the
// local step without accumulator (elided: commits from a pull snapshot),
// theta_k alone (6 slots); kDwGrad = the raw gradient only, stored for a
// separate optimizer kernel (no chunks).
enum { kDwUpdAcc = 0, kDwUpd = 1, kDwGrad = 2, kDwUpdRed = 3 };
template <int BN, int kSplit, int kStages, int kBKs, int kMode>
struct DwCfg {
  static constexpr bool kAcc = kMode == kDwUpdAcc || kMode == kDwUpdRed;   // a_k += g
  static constexpr bool kAccRing = kMode == kDwUpdAcc;                     // a_k via the ring
  static constexpr int kArrays = kAccRing ? 2 : 1;
  static constexpr int kSlotBytes = kArrays * (kChunkBytes + kBiasHalf);
  static constexpr int kRing = kAccRing ? 3 : 6;
  static constexpr int kBK = kBKs;
  static constexpr int kBox = kBK * 128;
  static constexpr int kABytes = 2 * kBox;
  static constexpr int kBBytes = (BN / 64) * kBox;
  static constexpr int kStageBytes = kSplit * (kABytes + kBBytes);
  // one accumulator: BN columns, or two of BN in the split mode (the leading
  // piece products and the five smaller pairs, kept apart for accuracy)
  static constexpr uint32_t kAccCols = (kSplit == 1 ? 1 : 2) * BN;
  static constexpr uint32_t kTmemCols = 2 * kAccCols;
  static constexpr int kChunks = BN / kCF;
  static constexpr size_t kRingOff = (size_t)kStages * kStageBytes;
  static constexpr size_t kGOff = kRingOff + (size_t)kRing * kSlotBytes;   // gradient staging
  static constexpr size_t kBarOff = kGOff + (size_t)kEpiWarps * 16 * 32 * 4;
  static constexpr size_t kSmem = kBarOff + 256 + 1024;   // barriers, alignment slack
};

// Four floats as four bf16 (round to nearest even), packed for one 8-byte store.
__device__ __forceinline__ uint2 bf16x4(const float (&x)[4]) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(x[0], x[1]);
  const __nv_bfloat162 hi = __floats2bfloat162_rn(x[2], x[3]);
  return make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
}
// Piece pairs (i, j), i + j <= 2, of the split product (pair 0 = a0 b0).
__device__ __forceinline__ int pair_a(int q) { return q == 2 || q == 4 ? 1 : q == 5 ? 2 : 0; }
__device__ __forceinline__ int pair_b(int q) { return q == 1 || q == 4 ? 1 : q == 3 ? 2 : 0; }

constexpr int kMaxDwLayers = 8;   // layers per launch (more are split into launches)
struct DwLayer {
  int M, N;          // inputs d_{l-1}, outputs d_l
  int mt, nt;        // input tiles (M / 128 + 1: the last holds the bias row), feature tiles
  int tile_begin;    // first tile of this layer in the launch
  int a_direct;      // A = the padded shards' rows of the slot's minibatch (layer 1)
  int64_t woff, boff;
};
struct DwBatch {
  CUtensorMap a[kMaxDwLayers], b[kMaxDwLayers], th[kMaxDwLayers], ac[kMaxDwLayers];
  DwLayer layer[kMaxDwLayers];
  int n_layers, total_tiles;
};

struct TileIdx {
  int layer, m_tile, n_tile, slot;
};
__device__ __forceinline__ TileIdx decode(const DwBatch& B, int t) {
  int i = 0;
  while (i + 1 < B.n_layers && t >= B.layer[i + 1].tile_begin) ++i;
  const DwLayer& L = B.layer[i];
  const int u = t - L.tile_begin;
  TileIdx r;
  r.layer = i;
  r.m_tile = u % L.mt;
  const int rest = u / L.mt;
  r.n_tile = rest % L.nt;
  r.slot = rest / L.nt;
  return r;
}

// Row r (< 128) of H^T set to one in every sample of an A stage: two 64-input
// boxes of kBK 128-byte rows (one per sample), 16-byte chunks swizzled by
// row % 8.
template <int kBK>
__device__ __forceinline__ void write_ones_row(uint8_t* sa, int r) {
  uint8_t* box = sa + (r >> 6) * (kBK * 128);
  const int i = r & 63;
  for (int j = 0; j < kBK; ++j) {
    const int off = j * 128 + ((((i >> 3) ^ (j & 7))) << 4) + (i & 7) * 2;
    *reinterpret_cast<uint16_t*>(box + off) = 0x3F80;   // bf16 1.0
  }
}

template <int BN, int kSplit, int kStages, int kBKs, int kMode>
__global__ void __launch_bounds__(kThreads, 1)
tc_dw_kernel(const __grid_constant__ DwBatch B, const TcArgs args) {
  using Cfg = DwCfg<BN, kSplit, kStages, kBKs, kMode>;
  constexpr bool kAcc = Cfg::kAcc, kAccRing = Cfg::kAccRing, kGrad = kMode == kDwGrad;
  constexpr int kRing = Cfg::kRing, kSlotBytes = Cfg::kSlotBytes;
  constexpr int kBK = Cfg::kBK, kABytes = Cfg::kABytes, kBox = Cfg::kBox;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Cfg::kBarOff);
  uint64_t* empty = full + kStages;
  uint64_t* cfull = empty + kStages;     // parameter chunk landed
  uint64_t* cempty = cfull + kRing;      // parameter chunk consumed (8 epilogue warps)
  uint64_t* tfull = cempty + kRing;      // accumulator b complete
  uint64_t* tempty = tfull + 2;          // accumulator b drained (8 epilogue warps)
  uint64_t* fin = tempty + 2;            // MMA drain on abort
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(fin + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
  volatile int* chunk_tiles = abort_flag + 1;   // tiles whose chunks are all requested

  __shared__ int s_skip;
  if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int*>(args.err);
  __syncthreads();
  if (s_skip != 0) return;   // an earlier launch gave up: uniform across the CTA

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int T = B.total_tiles;
  const int KT = (args.K + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int r = 0; r < kRing; ++r) {
      tc::mbar_init(&cfull[r], 1);
      tc::mbar_init(&cempty[r], kEpiWarps);
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(&tfull[b], 1);
      tc::mbar_init(&tempty[b], kEpiWarps);
    }
    tc::mbar_init(fin, 1);
    *abort_flag = 0;
    *chunk_tiles = 0;
    tc::fence_mbar_init();
    for (int i = 0; i < B.n_layers; ++i) {
      tc::tma_prefetch_desc(&B.a[i]);
      tc::tma_prefetch_desc(&B.b[i]);
      tc::tma_prefetch_desc(&B.th[i]);
      tc::tma_prefetch_desc(&B.ac[i]);
    }
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_holder, Cfg::kTmemCols);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  // programmatic dependent launch: the setup above overlapped the preceding
  // kernel; global memory is touched only after it has completed, except the
  // producer's first parameter chunks (below)

  // (the next forward may read theta_k before its own dependency wait: this
  // kernel lets it launch only when all CTAs have exited, writes fenced)
  if (!((warp == 0 || warp == kWarps - 1) && lane == 0)) pdl_wait_only();
  if (warp == 0 || warp == kWarps - 1) {
    if (warp == 0 && lane == 0) {
      // operand producer (warp 0): the GEMM operands of every tile into the
      // stage ring, as fast as the MMA frees stages
      pdl_wait_only();
      uint32_t ml = 0;   // stage fills issued
      bool ok = true;
      // On a long stream of tiles (bound by DRAM) the operands of a tile are
      // requested only once the previous tile's parameter chunks are, so
      // those stay first in line; on a short one they run ahead.
      const bool throttle = !kGrad && T >= kThrottleTiles * (int)gridDim.x;
      int itp = 0;
      for (int t = blockIdx.x; ok && t < T; t += gridDim.x, ++itp) {
        const TileIdx ti = decode(B, t);
        const CUtensorMap* tmA = &B.a[ti.layer];
        const CUtensorMap* tmB = &B.b[ti.layer];
        // layer 1's A from the padded shards: the worker's shard at the slot's
        // minibatch row (samples past m multiply dZ rows that are zero fill)
        const bool a_direct = B.layer[ti.layer].a_direct && args.x_shard > 0;
        const int a_row0 =
            a_direct ? (int)batch_row0(args.slot_t0, ti.slot, args.step, args.K, args.x_shard) : 0;
        const int a_z = a_direct ? AGN_LD(args.slot_worker + ti.slot) : ti.slot;
        if (throttle && itp > 0 && *chunk_tiles < itp) {
          const uint64_t t0 = tc::globaltimer_ns();
          while (*chunk_tiles < itp) {
            if (*abort_flag || tc::globaltimer_ns() - t0 > kWaitNs) {
              ok = false;
              break;
            }
            __nanosleep(64);
          }
          if (!ok) break;
        }
        for (int kt = 0; kt < KT; ++kt) {
          const int s = ml % kStages;
          if (ml >= kStages &&
              !tc::wait_or_abort(&empty[s], ((ml / kStages) - 1) & 1, abort_flag, kWaitNs)) {
            ok = false;
            break;
          }
          uint8_t* sa0 = smem + s * Cfg::kStageBytes;
          uint8_t* sb0 = sa0 + kSplit * kABytes;
          tc::mbar_arrive_expect_tx(&full[s], Cfg::kStageBytes);
  #pragma unroll
          for (int p = 0; p < kSplit; ++p) {
            uint8_t* sa = sa0 + p * kABytes;
            uint8_t* sb = sb0 + p * Cfg::kBBytes;
            if (kSplit == 1) {
              tc::tma_load_3d(sa, tmA, &full[s], ti.m_tile * 128, kt * kBK + a_row0, a_z);
              tc::tma_load_3d(sa + kBox, tmA, &full[s], ti.m_tile * 128 + 64, kt * kBK + a_row0,
                              a_z);
  #pragma unroll
              for (int c = 0; c < BN / 64; ++c)
                tc::tma_load_3d(sb + c * kBox, tmB, &full[s], ti.n_tile * BN + c * 64, kt * kBK,
                                ti.slot);
            } else {
              tc::tma_load_4d(sa, tmA, &full[s], ti.m_tile * 128, kt * kBK + a_row0, a_z, p);
              tc::tma_load_4d(sa + kBox, tmA, &full[s], ti.m_tile * 128 + 64, kt * kBK + a_row0,
                              a_z, p);
  #pragma unroll
              for (int c = 0; c < BN / 64; ++c)
                tc::tma_load_4d(sb + c * kBox, tmB, &full[s], ti.n_tile * BN + c * 64, kt * kBK,
                                ti.slot, p);
            }
          }
          ++ml;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        // drain (bounded) the copies armed but maybe not yet landed
        for (uint32_t j = ml > (uint32_t)kStages ? ml - kStages : 0; j < ml; ++j)
          tc::mbar_wait_bounded(&full[j % kStages], (j / kStages) & 1, kWaitNs);
      }
    } else if (lane == 0) {
      // parameter producer (the last warp): each tile's theta_k and a_k rows
      // into the chunk ring, as fast as the epilogue frees slots
      uint32_t ch = 0;   // chunk fills issued
      bool ok = true;
      // theta_k / a_k chunk c of tile ti into ring slot r
      auto issue_chunk = [&](const TileIdx& ti, int worker, int c, int r) {
        const DwLayer& L = B.layer[ti.layer];
        const bool bias_tile = ti.m_tile == L.M / 128;
        uint8_t* dst = smem + Cfg::kRingOff + (size_t)r * kSlotBytes;
        const int f0 = ti.n_tile * BN + c * kCF;
        constexpr int kA = Cfg::kArrays;
        tc::mbar_arrive_expect_tx(&cfull[r], kA * (kChunkBytes + (bias_tile ? kBiasHalf : 0)));
        tc::tma_load_3d(dst, &B.th[ti.layer], &cfull[r], ti.m_tile * 128, f0, worker);
        if (kAccRing)
          tc::tma_load_3d(dst + kChunkBytes, &B.ac[ti.layer], &cfull[r], ti.m_tile * 128, f0,
                          worker);
        if (bias_tile) {   // b_l[f0 .. f0 + 31] and its accumulator (within the replica)
          const int64_t pb = (int64_t)worker * args.ld_param + L.boff + f0;
          if (AGN_BOUNDS_OK(args.theta + pb, kBiasHalf)) {
            tc::bulk_load(dst + kA * kChunkBytes, args.theta + pb, kBiasHalf, &cfull[r]);
          } else {   // bounds-checked build: account for the bytes, skip the copy
            AGN_BOUNDS_FAIL(args.theta + pb);
            tc::mbar_complete_tx(&cfull[r], kBiasHalf);
          }
          if (kAccRing) {
            if (AGN_BOUNDS_OK(args.acc + pb, kBiasHalf)) {
              tc::bulk_load(dst + kA * kChunkBytes + kBiasHalf, args.acc + pb, kBiasHalf,
                            &cfull[r]);
            } else {
              AGN_BOUNDS_FAIL(args.acc + pb);
              tc::mbar_complete_tx(&cfull[r], kBiasHalf);
            }
          }
        }
      };
      // theta_k and a_k were last written by this kernel's previous launch or
      // a pull, two or more launches back: the first tile's first chunks are
      // requested before waiting for the preceding kernel
      int npre = 0;
      if (!kGrad && (int)blockIdx.x < T) {
        const TileIdx t0 = decode(B, blockIdx.x);
        const DwLayer& L0 = B.layer[t0.layer];
        npre = min(kRing, min(Cfg::kChunks, (L0.N - t0.n_tile * BN + kCF - 1) / kCF));
        const int w0 = AGN_LD(args.slot_worker + t0.slot);
        for (int c = 0; c < npre; ++c) {
          issue_chunk(t0, w0, c, (int)ch);
          ++ch;
        }
      }
      pdl_wait_only();
      for (int t = blockIdx.x; !kGrad && ok && t < T; t += gridDim.x) {
        const TileIdx ti = decode(B, t);
        const DwLayer& L = B.layer[ti.layer];
        const int worker = AGN_LD(args.slot_worker + ti.slot);
        const int nch = min(Cfg::kChunks, (L.N - ti.n_tile * BN + kCF - 1) / kCF);
        for (int c = t == (int)blockIdx.x ? npre : 0; c < nch; ++c) {
          const int r = ch % kRing;
          if (ch >= kRing &&
              !tc::wait_or_abort(&cempty[r], ((ch / kRing) - 1) & 1, abort_flag, kWaitNs)) {
            ok = false;
            break;
          }
          issue_chunk(ti, worker, c, r);
          ++ch;
        }
        *chunk_tiles = *chunk_tiles + 1;
      }
      if (!ok) {
        *abort_flag = 1;
        for (uint32_t j = ch > (uint32_t)kRing ? ch - kRing : 0; j < ch; ++j)
          tc::mbar_wait_bounded(&cfull[j % kRing], (j / kRing) & 1, kWaitNs);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t kIdesc = tc::idesc_bf16_f32(128, BN, true, true);
      uint32_t ml = 0;
      bool ok = true;
      int it = 0;
      for (int t = blockIdx.x; ok && t < T; t += gridDim.x, ++it) {
        const TileIdx ti = decode(B, t);
        const DwLayer& L = B.layer[ti.layer];
        const int b = it & 1;
        if (it >= 2 && !tc::wait_or_abort(&tempty[b], ((it >> 1) - 1) & 1, abort_flag, kWaitNs)) {
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const uint32_t dbase = tmem + (uint32_t)b * Cfg::kAccCols;
        const int ones_row = L.M - ti.m_tile * 128;   // < 128 on the bias tile
        for (int kt = 0; kt < KT; ++kt) {
          const int s = ml % kStages;
          if (!tc::wait_or_abort(&full[s], (ml / kStages) & 1, abort_flag, kWaitNs)) {
            ok = false;
            break;
          }
          tc::tc_fence_after();
          if (ones_row < 128) {   // piece 0 of the out-of-range row := 1 (pieces 1, 2 stay 0)
            write_ones_row<kBK>(smem + s * Cfg::kStageBytes, ones_row);
            tc::fence_proxy_async_smem();
          }
          const uint32_t sa0 = tc::smem_u32(smem + s * Cfg::kStageBytes);
          const uint32_t sb0 = sa0 + kSplit * kABytes;
          constexpr int kPairs = kSplit == 1 ? 1 : 6;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
#pragma unroll
            for (int q = 0; q < kPairs; ++q) {
              const uint32_t sa = sa0 + (kSplit == 1 ? 0 : pair_a(q)) * kABytes;
              const uint32_t sb = sb0 + (kSplit == 1 ? 0 : pair_b(q)) * Cfg::kBBytes;
              const uint64_t ad = tc::smem_desc_sw128(sa + kk * 2048, kBox, 1024);
              const uint64_t bd = tc::smem_desc_sw128(sb + kk * 2048, kBox, 1024);
              const uint32_t dcol = (kSplit == 3 && q > 0) ? (uint32_t)BN : 0u;
              const bool acc_on = kSplit == 1 ? (kt | kk | q) != 0
                                              : (q == 0 ? (kt | kk) != 0
                                                        : ((kt | kk) != 0 || q > 1));
              tc::mma_bf16(dbase + dcol, ad, bd, kIdesc, acc_on ? 1u : 0u);
            }
          }
          tc::mma_commit(&empty[s]);
          ++ml;
        }
        if (!ok) break;
        tc::mma_commit(&tfull[b]);
      }
      if (!ok) {
        *abort_flag = 1;
        tc::mma_commit(fin);   // every MMA issued so far has completed once fin flips
        tc::mbar_wait_bounded(fin, 0, kWaitNs);
      }
    }
  } else {
    // epilogue warps 2..9: warp w reads TMEM lane quadrant w % 4 (inputs
    // 32 (w % 4) .. + 31 of the tile) and columns 16 hf .. + 15 of each chunk,
    // hf = (w - 2) / 4.  It stages its 16 x 32 gradients in shared memory
    // (feature-major), then each lane updates four consecutive inputs of four
    // features with 16-byte shared loads and 16-byte global stores.
    const int g = warp & 3, hf = (warp - 2) >> 2;
    float* gS = reinterpret_cast<float*>(smem + Cfg::kGOff) + (warp - 2) * (16 * 32);
    const float eta = args.eta;
    uint32_t ch = 0;
    bool ok = true;
    int it = 0;
    const int k4 = (lane & 7) * 4, i0 = lane >> 3;   // phase-2 position of this lane
    for (int t = blockIdx.x; ok && t < T; t += gridDim.x, ++it) {
      const TileIdx ti = decode(B, t);
      const DwLayer& L = B.layer[ti.layer];
      const int M = L.M, N = L.N;
      const int worker = AGN_LD(args.slot_worker + ti.slot);
      const int b = it & 1;
      // waits are warp-uniform: a lane that gave up takes its whole warp out
      // before the next .sync.aligned TMEM load
      ok = __all_sync(0xffffffffu, tc::wait_or_abort(&tfull[b], (it >> 1) & 1, abort_flag,
                                                      kWaitNs));
      if (!ok) break;
      tc::tc_fence_after();
      const int k0 = ti.m_tile * 128 + 32 * g;            // first input of this quadrant
      const bool quad_ok = k0 + k4 < M;                   // M % 8 == 0: all four or none
      const int kb = M - k0;                              // bias row, if 0 <= kb < 32
      const uint32_t tbase = tmem + ((uint32_t)(32 * g) << 16) + (uint32_t)b * Cfg::kAccCols +
                             (uint32_t)(16 * hf);
      const int64_t rbase = (int64_t)worker * args.ld_param;
      float* theta = args.theta + rbase;
      float* acc = kAcc ? args.acc + rbase : nullptr;
      bf16* tb = args.theta_b ? args.theta_b + rbase : nullptr;   // bf16 mode only
      const int nch = min(Cfg::kChunks, (N - ti.n_tile * BN + kCF - 1) / kCF);
      for (int c = 0; c < nch; ++c) {
        const int r = ch % kRing;
        uint32_t v[16];
        tc::tmem_ld_32x32b_x16(tbase + (uint32_t)(c * kCF), v);
        if (kSplit == 3) {
          uint32_t v2[16];
          tc::tmem_ld_32x32b_x16(tbase + (uint32_t)(BN + c * kCF), v2);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i)
            v[i] = __float_as_uint(__fadd_rn(__uint_as_float(v[i]), __uint_as_float(v2[i])));
        } else {
          tc::tmem_ld_wait();
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) gS[i * 32 + lane] = __uint_as_float(v[i]);
        if (kGrad) {   // raw gradient out: grad[w][p] = g, coalesced 16-byte stores
          __syncwarp();
          const int fbase = ti.n_tile * BN + c * kCF + 16 * hf;
          float* gout = args.grad_out + rbase;
          if (quad_ok) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int i = i0 + 4 * u;
              if (fbase + i < N)
                AGN_ST(reinterpret_cast<float4*>(gout + L.woff + (int64_t)(fbase + i) * M + k0 + k4),
                       *reinterpret_cast<const float4*>(gS + i * 32 + k4));
            }
          }
          if (kb >= 0 && kb < 32 && lane < 16 && fbase + lane < N)
            AGN_ST(gout + L.boff + fbase + lane, gS[lane * 32 + kb]);
          __syncwarp();
          continue;
        }
        ok = __all_sync(0xffffffffu,
                        tc::wait_or_abort(&cfull[r], (ch / kRing) & 1, abort_flag, kWaitNs));
        if (!ok) break;
        __syncwarp();
        const uint8_t* slot = smem + Cfg::kRingOff + (size_t)r * kSlotBytes;
        const int fbase = ti.n_tile * BN + c * kCF + 16 * hf;   // first feature of this warp
        if (quad_ok) {
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int i = i0 + 4 * u;                           // feature fbase + i
            if (fbase + i < N) {
              const float4 gv = *reinterpret_cast<const float4*>(gS + i * 32 + k4);
              const int so = (16 * hf + i) * 128 + 32 * g + k4;   // in the fp32 chunks
              const float4 tv = *reinterpret_cast<const float4*>(
                  reinterpret_cast<const float*>(slot) + so);
              float tn[4];
              tn[0] = local_step(tv.x, eta, gv.x);
              tn[1] = local_step(tv.y, eta, gv.y);
              tn[2] = local_step(tv.z, eta, gv.z);
              tn[3] = local_step(tv.w, eta, gv.w);
              const int64_t p = L.woff + (int64_t)(fbase + i) * M + k0 + k4;
              AGN_ST(reinterpret_cast<float4*>(theta + p), make_float4(tn[0], tn[1], tn[2], tn[3]));
              if (kAccRing) {
                const float4 av = *reinterpret_cast<const float4*>(
                    reinterpret_cast<const float*>(slot + kChunkBytes) + so);
                AGN_ST(reinterpret_cast<float4*>(acc + p),
                       make_float4(av.x + gv.x, av.y + gv.y, av.z + gv.z, av.w + gv.w));
              } else if (kAcc) {   // a_k += g in the L2 (one add per element and launch)
                AGN_RED4(reinterpret_cast<float*>(acc + p), gv);
              }
              // the bf16 copy (bf16 mode); the fp32 mode's GEMMs split the
              // fp32 weights themselves
              if (kSplit == 1) AGN_ST(reinterpret_cast<uint2*>(tb + p), bf16x4(tn));
            }
          }
        }
        if (kb >= 0 && kb < 32 && lane < 16 && fbase + lane < N) {   // bias row: b_l[f]
          const float* sTb =
              reinterpret_cast<const float*>(slot + Cfg::kArrays * kChunkBytes);
          const float gb = gS[lane * 32 + kb];
          const int64_t pb = L.boff + fbase + lane;
          const float tn = local_step(sTb[16 * hf + lane], eta, gb);
          AGN_ST(theta + pb, tn);
          if (kAccRing) AGN_ST(acc + pb, sTb[kCF + 16 * hf + lane] + gb);
          else if (kAcc) AGN_RED(acc + pb, gb);
          if (kSplit == 1) AGN_ST(tb + pb, __float2bfloat16_rn(tn));
        }
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&cempty[r]);
        ++ch;
      }
      if (!ok) break;
      tc::tc_fence_before();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&tempty[b]);
    }
    if (!ok) *abort_flag = 1;
  }
  __syncwarp();
  pdl_fence_exit();
  tc::tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) atomicExch(args.err, 1);
  if (warp == 1) tc::tmem_dealloc(tmem, Cfg::kTmemCols);
}

template <int BN, int kSplit, int kStages, int kBKs, int kMode>
Status launch_dw(const DwBatch& batch, const TcArgs& args, int num_sms, cudaStream_t st) {
  using Cfg = DwCfg<BN, kSplit, kStages, kBKs, kMode>;
  static_assert(Cfg::kSmem <= 232448, "shared memory");
  static_assert(Cfg::kSmem > 232448 / 2, "one CTA per SM (all 512 TMEM columns)");
  static_assert(Cfg::kTmemCols == 512, "TMEM columns");
  auto kern = tc_dw_kernel<BN, kSplit, kStages, kBKs, kMode>;
  static std::mutex mu;
  static std::set<int> done;
  {
    int dev = 0;
    AGN_TRY_CUDA(cudaGetDevice(&dev));
    std::lock_guard<std::mutex> lock(mu);
    if (!done.count(dev)) {
      AGN_TRY_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)Cfg::kSmem));
      done.insert(dev);
    }
  }
  if (batch.total_tiles <= 0) return Status::Ok();
  const int grid = std::min(batch.total_tiles, num_sms);
  {
    auto kf = kern;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kThreads, Cfg::kSmem, st, batch, args));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

}  // namespace

Status tc_backward_dw(const DwLayerMaps* layers, int n_layers, const TcArgs& args, int slots,
                      cudaStream_t st, bool split, int num_sms) {
  const int bn = split ? kTcDwBNSplit : kTcDwBN;
  for (int l0 = 0; l0 < n_layers; l0 += kMaxDwLayers) {
    DwBatch batch;
    std::memset(&batch, 0, sizeof(batch));
    int64_t tiles = 0, acc_bytes = 0;
    batch.n_layers = std::min(kMaxDwLayers, n_layers - l0);
    for (int i = 0; i < batch.n_layers; ++i) {
      const DwLayerMaps& d = layers[l0 + i];
      if (d.M <= 0 || d.N <= 0) return Status::Err(AGN_E_INVALID, "empty dW layer");
      batch.a[i] = *d.h_mn;
      batch.b[i] = *d.dz_mn;
      batch.th[i] = *d.theta;
      batch.ac[i] = *d.acc;
      DwLayer& L = batch.layer[i];
      L.M = d.M;
      L.N = d.N;
      L.woff = d.woff;
      L.a_direct = d.a_direct;
      L.boff = d.boff;
      L.mt = d.M / 128 + 1;          // rows 0 .. M, row M the bias
      L.nt = (d.N + bn - 1) / bn;
      acc_bytes += ((int64_t)d.M + 1) * d.N * 4 * slots;
      L.tile_begin = (int)tiles;
      tiles += (int64_t)L.mt * L.nt * slots;
      if (tiles > INT32_MAX) return Status::Err(AGN_E_UNSUPPORTED, "dW tile count overflows");
    }
    batch.total_tiles = (int)tiles;
    // split mode: 32 samples per stage, so that two stages fit beside the
    // parameter ring (the next tile's operands land while this one multiplies)
    // grad_out: gradient only; else acc null: accumulator elided; else a_k
    // through L2 adds while the launch's accumulators fit well within the L2
    // (small waves, where the chunk ring's latency bounds the kernel and
    // half the ring's bytes per chunk buy twice the chunks in flight), or
    // through the ring (large waves, which stream theta_k and a_k from DRAM
    // at the copy bandwidth: there the L2's adds slowed the stream by 4 %;
    // and always with args.acc_ring)
    constexpr int64_t kRedAccBytes = 64ll << 20;
    const bool ring = args.acc_ring || acc_bytes > kRedAccBytes;
    const int mode = args.grad_out ? kDwGrad
                     : !args.acc   ? kDwUpd
                     : ring        ? kDwUpdAcc
                                   : kDwUpdRed;
    Status r = Status::Ok();
    if (split) {
      r = mode == kDwGrad     ? launch_dw<kTcDwBNSplit, 3, 2, 32, kDwGrad>(batch, args, num_sms, st)
          : mode == kDwUpd    ? launch_dw<kTcDwBNSplit, 3, 2, 32, kDwUpd>(batch, args, num_sms, st)
          : mode == kDwUpdAcc ? launch_dw<kTcDwBNSplit, 3, 2, 32, kDwUpdAcc>(batch, args, num_sms, st)
                              : launch_dw<kTcDwBNSplit, 3, 2, 32, kDwUpdRed>(batch, args, num_sms, st);
    } else {
      r = mode == kDwGrad     ? launch_dw<kTcDwBN, 1, 2, 64, kDwGrad>(batch, args, num_sms, st)
          : mode == kDwUpd    ? launch_dw<kTcDwBN, 1, 2, 64, kDwUpd>(batch, args, num_sms, st)
          : mode == kDwUpdAcc ? launch_dw<kTcDwBN, 1, 2, 64, kDwUpdAcc>(batch, args, num_sms, st)
                              : launch_dw<kTcDwBN, 1, 2, 64, kDwUpdRed>(batch, args, num_sms, st);
    }
    if (!r.ok()) return r;
  }
  return Status::Ok();
}

AGN_BOUNDS_UNIT(dw)

}  // namespace agn
