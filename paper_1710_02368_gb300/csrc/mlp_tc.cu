// Kernels (a) and (b) on the 5th-generation tensor cores (bf16 mode): the
// batched-over-workers forward, dX and dW GEMMs of the MLP as tcgen05.mma
// kind::f16 (bf16 operands, f32 accumulators in TMEM), operands staged in
// shared memory by TMA with 128-byte swizzle, fused epilogues read from TMEM.
//
// Every GEMM puts the wide feature dimension on M = 128 (one TMEM lane per
// feature), so each epilogue access is coalesced across a warp's lanes:
//   forward: D[f][j] = sum_k W[f][k] H[j][k]       A = W    (K-major)
//            B = H_{l-1} (K-major); out H_l[j][f] = relu(D + b[f])    (Eq. 1)
//   dX     : D[k][j] = sum_f W[f][k] dZ[j][f]     A = W^T  (MN-major)
//            B = dZ_l (K-major); out dZ_{l-1}[j][k] = D [H_{l-1} > 0]
//   dW     : D[k][f] = sum_j H[j][k] dZ[j][f]     A = H^T  (MN-major)
//            B = dZ^T (MN-major); theta_k[f][k] -= eta D, a_k[f][k] += D and
//            the bf16 copy (Algorithm 1's local step and accumulation)
// One CTA computes one 128 x BN tile of one slot: warp 0 issues TMA loads
// into a ring of stages, warp 1 issues the MMAs (one thread) and owns the
// TMEM allocation, then all eight warps run the epilogue (warp w reads TMEM
// lanes 32 (w % 4) .. +31, column half w / 4).  Every mbarrier wait is bounded
// (2 s of global time): on expiry the kernel sets *err, stops issuing, waits
// for its own copies in flight (bounded), frees TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>
#include <type_traits>

#include "mlp.cuh"
#include "mlp_tc.cuh"
#include "tc_ptx.cuh"

namespace agn {

namespace {

constexpr int kThreads = 256;
constexpr uint64_t kWaitNs = 2000000000ull;   // 2 s
constexpr int kEpiTBytes = 8 * 32 * 32 * 4;   // forward / dX epilogue transpose tiles
// fp32 mode: each k step's fp32 weights (128 x K per stage) are converted in
// place into their bf16 pieces by kConvWarps warps
constexpr int kConvWarps = 6;

// K per stage: 64 bf16, one 128-byte row (128-byte swizzle); 32 bf16, one
// 64-byte row (64-byte swizzle), for the fp32 mode's forward and dX GEMMs,
// whose stages hold three pieces of each operand: half the bytes per stage,
// so twice the stages in flight to hide the load and conversion latency.
constexpr int stage_k(int split, int epi) { return split == 3 && epi != kEpiDW ? kTcSplitBK : 64; }
// fp32 mode, forward and dX, column tiles up to 128: the converters write the
// weight pieces (the MMA's A operand) into tensor memory instead of shared
// memory.  The stages' shared-memory traffic (TMA writes, the converters'
// reads and writes, the MMAs' operand reads) had bound the mainloop; the MMAs
// then read only B from shared memory.
constexpr bool a_in_tmem(int split, int epi, int bn) {
  return split == 3 && epi != kEpiDW && bn <= 128;
}
// Fused output layer (kEpiFwdHead): at most kHC classes; shared scratch of
// W_L's 128 x kHC slice, the warps' partial logits [8][16][kHC] and the
// chunk's logits / dZ_L [32][kHC].
constexpr int kHC = kHeadMaxClasses;
constexpr int kHeadScratch = (kHC * 128 + 8 * 16 * kHC + 32 * kHC) * 4 + 8 * 256 * 2;

// A stage holds kSplit A pieces then kSplit B pieces (kSplit = 3 in the fp32
// mode, where every fp32 operand is the exact sum of three bf16 pieces), of
// kBK k each (rows of 2 kBK bytes).  With A in tensor memory (kATmem) the
// stage holds the fp32 weight tile the converters read, then the B pieces,
// and A's pieces take kACols TMEM columns per stage after the accumulators.
// kMT = 2 (bf16 forward and dX of full waves): two 128-row A tiles per stage
// share the B tile, each with its own accumulator.
template <int BN, int kSplit, int kBKs = 64, bool kATmemT = false, int kMTT = 1>
struct TileCfg {
  static constexpr int kBK = kBKs;
  static constexpr bool kATmem = kATmemT;
  static constexpr int kRowBytes = 2 * kBK;
  static constexpr int kABytes = 128 * kRowBytes;
  static constexpr int kBBytes = BN * kRowBytes;
  static constexpr uint32_t kA32Bytes = 128 * kBK * 4;   // an fp32 weight tile
  static constexpr int kAArea = kATmem ? (int)kA32Bytes : kSplit * kABytes * kMTT;
  static constexpr int kStageBytes = kAArea + kSplit * kBBytes;
  // split mode keeps two accumulators: columns [0, BN) take the leading
  // piece products a0 b0, columns [BN, 2 BN) the five smaller pairs, so the
  // rounding of the tensor core's running sums is relative to each part
  static constexpr uint32_t kAccCols = (kSplit == 1 ? 1 : 2) * BN * kMTT;
  static constexpr uint32_t kACols = kSplit * kBK / 2;   // A pieces of one stage in TMEM
  static constexpr uint32_t kTmemCols = kATmem ? 512 : kAccCols;   // power of two >= 32
};

// The forward / dX epilogue's transpose tiles sit after the barriers when the
// CTA's shared memory has room for them (then the whole stage ring can hold
// split-K partial sums), else at the end of the ring.
template <int BN, int kSplit, int kStages, int kBKs, bool kATmem, int kMT = 1>
struct EpiT {
  static constexpr size_t kRing =
      (size_t)kStages * TileCfg<BN, kSplit, kBKs, kATmem, kMT>::kStageBytes;
  static constexpr bool kSeparate = kRing + 1280 + kEpiTBytes <= 232448;
  static constexpr size_t kOff = kSeparate ? kRing + 256 : kRing - kEpiTBytes;
  static constexpr size_t kRingFree = kSeparate ? kRing : kRing - kEpiTBytes;
  // the fused output layer's scratch, at the end of the free ring (below the
  // split-K partial sums' reach, which the host bounds accordingly)
  static constexpr size_t kHeadOff = kRingFree - kHeadScratch;
};

// Piece pairs (i, j) with i + j <= 2 of the split product: the dropped pairs
// are below 2^-25 |a b|, under the rounding of one fp32 product.
__device__ __constant__ const int kPairA[6] = {0, 0, 1, 0, 1, 2};
__device__ __constant__ const int kPairB[6] = {0, 1, 0, 2, 1, 0};

__device__ __forceinline__ float from_act(bf16 v) { return __bfloat162float(v); }
__device__ __forceinline__ float from_act(float v) { return v; }

// Four consecutive activations (16-byte aligned fp32, or 8-byte aligned bf16).
__device__ __forceinline__ float4 load4(const float* p) {
  return AGN_LD(reinterpret_cast<const float4*>(p));
}
__device__ __forceinline__ float4 load4(const bf16* p) {
  const uint2 u = AGN_LD(reinterpret_cast<const uint2*>(p));
  const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
  const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
  return make_float4(__low2float(lo), __high2float(lo), __low2float(hi), __high2float(hi));
}
__device__ __forceinline__ uint2 bf16x4(const float (&x)[4]) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(x[0], x[1]);
  const __nv_bfloat162 hi = __floats2bfloat162_rn(x[2], x[3]);
  return make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
}
__device__ __forceinline__ void store4(float* p, const float (&v)[4]) {
  AGN_ST(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
}
__device__ __forceinline__ void store4(bf16* p, const float (&v)[4]) {
  AGN_ST(reinterpret_cast<uint2*>(p), bf16x4(v));
}
// The three exact bf16 pieces of four floats (split3 of each), packed.
__device__ __forceinline__ void split3_x4(const float (&x)[4], uint2& q0, uint2& q1, uint2& q2) {
  float r[4];
  q0 = bf16x4(x);
  const __nv_bfloat162* p0 = reinterpret_cast<const __nv_bfloat162*>(&q0);
  r[0] = __fsub_rn(x[0], __low2float(p0[0]));
  r[1] = __fsub_rn(x[1], __high2float(p0[0]));
  r[2] = __fsub_rn(x[2], __low2float(p0[1]));
  r[3] = __fsub_rn(x[3], __high2float(p0[1]));
  q1 = bf16x4(r);
  const __nv_bfloat162* p1 = reinterpret_cast<const __nv_bfloat162*>(&q1);
  r[0] = __fsub_rn(r[0], __low2float(p1[0]));
  r[1] = __fsub_rn(r[1], __high2float(p1[0]));
  r[2] = __fsub_rn(r[2], __low2float(p1[1]));
  r[3] = __fsub_rn(r[3], __high2float(p1[1]));
  q2 = bf16x4(r);
}

// Wait that also gives up when another role has aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity,
                                              volatile int* abort_flag) {
  return tc::wait_or_abort(bar, parity, abort_flag, kWaitNs);
}

// The dW kernel is bound by its epilogue's DRAM traffic: two CTAs per SM
// (registers capped at 128) keep more loads in flight.
// kSplit = 1: bf16 operands (bf16 mode), 3D tensor maps (inner, rows, batch);
// kSplit = 3: fp32 operands as three exact bf16 pieces, 4D tensor maps
// (inner, rows, batch, piece), fp32 activations in the epilogues and the
// three pieces of the updated weights written by dW.
// kMT = 2: a CTA computes two 128-row tiles (rows 256 x blockIdx.x ..) that
// share each B stage (bf16 forward and dX without split K): half the B bytes
// per output, half the CTAs of a full wave.
template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages, int kSplit, int kMT = 1>
__global__ void __launch_bounds__(kThreads, kEpi == kEpiDW ? 2 : 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const TcArgs args) {
  constexpr int kBK = stage_k(kSplit, kEpi);
  constexpr bool kATmem = a_in_tmem(kSplit, kEpi, BN);
  static_assert(kMT == 1 || (kSplit == 1 && (kEpi == kEpiFwd || kEpi == kEpiDX)),
                "two row tiles per CTA: bf16 forward and dX only");
  using Cfg = TileCfg<BN, kSplit, kBK, kATmem, kMT>;
  using Epi = EpiT<BN, kSplit, kStages, kBK, kATmem, kMT>;
  static_assert(!kATmem || Cfg::kAccCols + kStages * Cfg::kACols <= Cfg::kTmemCols, "TMEM");
  constexpr int kABytes = Cfg::kABytes;
  constexpr uint32_t kA32Bytes = Cfg::kA32Bytes;
  constexpr int kBox = kBK * 128;   // one 64-wide MN box of kBK rows (MN-major operands)
  using TAct = typename std::conditional<kSplit == 1, bf16, float>::type;
  // fp32 mode, forward and dX: A = W arrives as fp32 (TMA, 128 x kBK floats
  // into the first 16 KB of the stage's 24 KB of A pieces) and warps 2-7
  // replace it, in place, by its three bf16 pieces in the swizzled layout the
  // MMA reads; the replicas hold no weight pieces.
  constexpr bool kWConv = kSplit == 3 && kEpi != kEpiDW;
  static_assert(!kWConv || kA32Bytes <= 3 * kABytes, "fp32 tile within the A slots");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * Cfg::kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* done = empty + kStages;
  uint64_t* red = done + 1;              // split K: the other ranks' partial sums landed
  uint64_t* conv = red + 1;              // fp32 weights: stage s's A pieces written
  uint64_t* afull = conv + kStages;      // fp32 weights: stage s's fp32 tile landed
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(afull + kStages);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  // A CTA that gave up earlier in this launch (or run) makes the rest return
  // at once, before they allocate anything.
  __shared__ int s_skip;
  if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int*>(args.err);
  __syncthreads();
  if (s_skip != 0) return;   // uniform across the CTA
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ks = kEpi == kEpiDW || kMT > 1 ? 1 : args.ksplit;   // CTAs sharing one output tile
  const int m_tile = blockIdx.x, n_tile = blockIdx.y;
  const int slot = blockIdx.z / ks, sk = blockIdx.z % ks;
  const int worker = AGN_LD(args.slot_worker + slot);
  // k steps [kt0, kt0 + KT) of this CTA (the host picks ks so that none is empty)
  const int KT_all = (args.K + kBK - 1) / kBK;
  const int kt_per = (KT_all + ks - 1) / ks;
  const int kt0 = sk * kt_per;
  const int KT = min(KT_all, kt0 + kt_per) - kt0;
  const int a_z = args.a_by_worker ? worker : slot;
  // layer 1's B straight from the padded shards: the worker's shard at the
  // slot's minibatch row (tile rows past m belong to the next rows of the
  // shard; their accumulator columns are never stored)
  const bool b_direct = !kBMN && args.x_b_direct && args.x_shard > 0;
  const int b_z = b_direct ? worker : args.b_by_worker ? worker : slot;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    tc::mbar_init(done, 1);
    tc::mbar_init(red, 1);
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&conv[s], kConvWarps);
      tc::mbar_init(&afull[s], 1);
    }
    *abort_flag = 0;
    tc::fence_mbar_init();
    tc::tma_prefetch_desc(&tmA);
    tc::tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_holder, Cfg::kTmemCols);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const uint32_t tmem = tmem_base;

  // Programmatic dependent launch: the setup above ran while the preceding
  // kernel finished.  Everything that reads or writes global memory waits
  // for it (pdl_begin), except the producer's loads of the weights for the
  // first stages (forward and dX: A = W, last written two or more kernels
  // back, where the preceding kernel only started once its own predecessor
  // was complete, or by the preceding kernel itself when that is the dW, a
  // pull or the Adam step, which let this one launch only after all their
  // CTAs exited with their writes fenced) and the converter warps, which
  // touch only shared and tensor memory until the epilogue (they wait before
  // it): the prefetched weight stages are converted while the preceding
  // kernel still runs.
  constexpr bool kPrefetchA = kEpi != kEpiDW;
  const bool producer = warp == 0 && lane == 0;
  const bool converter = kWConv && warp >= 2;
  if (!producer && !converter) pdl_begin();
  if (warp == 0) {
    if (lane == 0) {
      // one box of 3D maps (kSplit = 1) or of 4D maps with the piece index
      auto load = [&](uint8_t* dst, const CUtensorMap* map, int x, int y, int z, int p,
                      uint64_t* bar) {
        if (kSplit == 1) tc::tma_load_3d(dst, map, bar, x, y, z);
        else tc::tma_load_4d(dst, map, bar, x, y, z, p);
      };
      auto load_a = [&](int kt, int s) {
        uint8_t* sa0 = smem + s * Cfg::kStageBytes;
        const int kc = (kt0 + kt) * kBK;
#pragma unroll
        for (int mh = 0; mh < kMT; ++mh) {
          const int r0 = (m_tile * kMT + mh) * 128;
#pragma unroll
          for (int p = 0; p < kSplit; ++p) {
            uint8_t* sa = sa0 + (mh * kSplit + p) * kABytes;
            if (!kAMN) {
              load(sa, &tmA, kc, r0, a_z, p, &full[s]);
            } else {
              load(sa, &tmA, r0, kc, a_z, p, &full[s]);
              load(sa + kBox, &tmA, r0 + 64, kc, a_z, p, &full[s]);
            }
          }
        }
      };
      // fp32 weights of k step kt into stage s's A slots, on their own barrier
      // (afull[s]) so that the converters can start before the activations
      // land, for prefetched stages before the preceding kernel completes
      auto load_a32 = [&](int kt, int s) {
        uint8_t* dst = smem + s * Cfg::kStageBytes;
        const int kc = (kt0 + kt) * kBK;
        tc::mbar_arrive_expect_tx(&afull[s], kA32Bytes);
        if (!kAMN) tc::tma_load_3d(dst, &tmA, &afull[s], kc, m_tile * 128, a_z);
        else tc::tma_load_3d(dst, &tmA, &afull[s], m_tile * 128, kc, a_z);
      };
      // prefetched stages count the A bytes now and arrive with the B bytes
      // below, so no phase can complete before its B boxes are requested
      constexpr uint32_t kABytesAll = kWConv ? 0u : kSplit * kABytes * kMT;   // A bytes on full[s]
      constexpr uint32_t kBBytesAll = kSplit * Cfg::kBBytes;
      const int npre = kPrefetchA && !args.no_a_prefetch ? min(KT, kStages) : 0;
      // (slot_t0 is written by the host before the launch)
      const int b_row0 =
          b_direct ? (int)batch_row0(args.slot_t0, slot, args.step, args.N, args.x_shard) : 0;
      auto load_b = [&](int kt, int s) {
        uint8_t* sb0 = smem + s * Cfg::kStageBytes + Cfg::kAArea;
        const int kc = (kt0 + kt) * kBK;
#pragma unroll
        for (int p = 0; p < kSplit; ++p) {
          uint8_t* sb = sb0 + p * Cfg::kBBytes;
          if (!kBMN) {
            load(sb, &tmB, kc, n_tile * BN + b_row0, b_z, p, &full[s]);
          } else {
#pragma unroll
            for (int c = 0; c < BN / 64; ++c)
              load(sb + c * kBox, &tmB, n_tile * BN + c * 64, kc, b_z, p, &full[s]);
          }
        }
      };
      for (int kt = 0; kt < npre; ++kt) {
        if (kWConv) load_a32(kt, kt);
        if (b_direct) {
          // B from the padded shards, which no kernel writes: the whole stage
          // is requested before the wait
          tc::mbar_arrive_expect_tx(&full[kt], kABytesAll + kBBytesAll);
          if (!kWConv) load_a(kt, kt);
          load_b(kt, kt);
        } else if (!kWConv) {
          tc::mbar_expect_tx(&full[kt], kABytesAll);
          load_a(kt, kt);
        }
      }
      pdl_begin();
      int kt = 0;
      for (; kt < KT; ++kt) {
        const int s = kt % kStages;
        if (kt >= kStages && !wait_or_abort(&empty[s], ((kt / kStages) - 1) & 1, abort_flag)) {
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        if (kt >= npre) {
          tc::mbar_arrive_expect_tx(&full[s], kABytesAll + kBBytesAll);
          if (kWConv) load_a32(kt, s);
          else load_a(kt, s);
        } else if (b_direct) {
          continue;   // requested whole before the wait
        } else {
          tc::mbar_arrive_expect_tx(&full[s], kBBytesAll);
        }
        load_b(kt, s);
      }
      if (*abort_flag) {
        // drain: wait (bounded) for the copies of the last stages we armed;
        // prefetched stages not reached yet get their arrival first (with B
        // from the padded shards they had it before the wait)
        if (!b_direct)
          for (int j = kt; j < npre; ++j) tc::mbar_arrive(&full[j]);
        for (int j = kt; j < npre; ++j) tc::mbar_wait_bounded(&full[j], 0, kWaitNs);
        for (int j = kt - 1; j >= 0 && j >= kt - kStages; --j)
          tc::mbar_wait_bounded(&full[j % kStages], (j / kStages) & 1, kWaitNs);
        if (kWConv)   // the fp32 weight tiles armed (prefetched or in the loop)
          for (int j = max(kt, npre) - 1; j >= 0 && j >= max(kt, npre) - kStages; --j)
            tc::mbar_wait_bounded(&afull[j % kStages], (j / kStages) & 1, kWaitNs);
      }
    }
  } else if (kWConv && kATmem && warp >= 2) {
    if constexpr (kATmem) {
      // Converters, A in tensor memory: warp w writes TMEM lanes 32 (w % 4) ..
      // + 31, the rows (features; dX: inputs) of that quadrant.  Quadrants 2
      // and 3 have two converter warps (2, 6 and 3, 7), each taking half of the
      // k step; quadrants 0 and 1 have one (4, 5), taking all of it.  A thread
      // loads its row's fp32 values (the forward's K-major tile lands with a
      // 128-byte swizzle, so the warp's 16-byte loads do not conflict; dX's
      // MN-major tile is read down a column), splits them into three pieces and
      // stores each piece's bf16 pairs (the lower k in the lower half) into its
      // lane's columns: piece p of the stage at columns p kBK / 2 .. + kBK / 2.
      constexpr int kHalfK = kBK / 2;
      const int qd = warp & 3;
      const int kb = qd >= 2 ? (warp >= 6 ? kHalfK : 0) : 0;   // first k of this warp
      const int ke = qd >= 2 ? kb + kHalfK : kBK;
      const int row = 32 * qd + lane;
      const uint32_t lane_addr = (uint32_t)(32 * qd) << 16;
      for (int kt = 0; kt < KT; ++kt) {
        const int s = kt % kStages;
        if (!__all_sync(0xffffffffu, wait_or_abort(&afull[s], (kt / kStages) & 1, abort_flag))) {
          if (lane == 0) *abort_flag = 1;
          break;
        }
        const float* a32 = reinterpret_cast<const float*>(smem + s * Cfg::kStageBytes);
        const uint32_t acol = tmem + lane_addr + Cfg::kAccCols + (uint32_t)s * Cfg::kACols;
  #pragma unroll 1
        for (int h0 = kb; h0 < ke; h0 += kHalfK) {
          float x[kHalfK];
          if (!kAMN) {
  #pragma unroll
            for (int c = 0; c < kHalfK / 4; ++c) {
              const int cc = (h0 / 4 + c) ^ (row & 7);
              const float4 v = *reinterpret_cast<const float4*>(a32 + row * kBK + 4 * cc);
              x[4 * c] = v.x;
              x[4 * c + 1] = v.y;
              x[4 * c + 2] = v.z;
              x[4 * c + 3] = v.w;
            }
          } else {
  #pragma unroll
            for (int k = 0; k < kHalfK; ++k) x[k] = a32[(h0 + k) * 128 + row];
          }
          uint32_t p0[kHalfK / 2], p1[kHalfK / 2], p2[kHalfK / 2];
  #pragma unroll
          for (int j = 0; j < kHalfK / 2; ++j) {
            bf16 a0, a1, a2, b0, b1, b2;
            split3(x[2 * j], a0, a1, a2);
            split3(x[2 * j + 1], b0, b1, b2);
            const __nv_bfloat162 v0 = __halves2bfloat162(a0, b0);
            const __nv_bfloat162 v1 = __halves2bfloat162(a1, b1);
            const __nv_bfloat162 v2 = __halves2bfloat162(a2, b2);
            p0[j] = *reinterpret_cast<const uint32_t*>(&v0);
            p1[j] = *reinterpret_cast<const uint32_t*>(&v1);
            p2[j] = *reinterpret_cast<const uint32_t*>(&v2);
          }
          const uint32_t col = acol + (uint32_t)(h0 / 2);
          tc::tmem_st_32x32b_x8(col, p0);
          tc::tmem_st_32x32b_x8(col + kBK / 2, p1);
          tc::tmem_st_32x32b_x8(col + kBK, p2);
        }
        tc::tmem_st_wait();
        tc::tc_fence_before();   // the stores, before the MMA thread's wait on conv[s]
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&conv[s]);
      }
    }
    pdl_begin();   // before the epilogue's global accesses
  } else if (kWConv && warp >= 2) {
    // Converters: the fp32 weight tile of each k step into its three bf16
    // pieces (x0 = bf16(x), x1 = bf16(x - x0), x2 = bf16(x - x0 - x1)), in
    // place: every converter thread first loads its elements (four
    // consecutive floats per item, 16-byte shared loads), the six warps meet
    // at a named barrier, then each writes its items' pieces (three 8-byte
    // stores at the 128-byte-swizzled positions the TMA would have used).
    // The barrier also ANDs the warps' waits, so that they give up together.
    const int ct = threadIdx.x - 64;
    constexpr int kItems = 128 * kBK / 4, kPer = (kItems + kConvWarps * 32 - 1) / (kConvWarps * 32);
    constexpr int kQ = kBK / 4;   // 4-float items per K-major row
    for (int kt = 0; kt < KT; ++kt) {
      const int s = kt % kStages;
      const bool got = __all_sync(0xffffffffu,
                                  wait_or_abort(&afull[s], (kt / kStages) & 1, abort_flag));
      int all_ok;
      asm volatile("{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
                   "bar.red.and.pred q, 1, %2, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
                   : "=r"(all_ok) : "r"((unsigned)got), "n"(kConvWarps * 32) : "memory");
      if (!all_ok) {
        if (lane == 0) *abort_flag = 1;
        break;
      }
      uint8_t* sa0 = smem + s * Cfg::kStageBytes;
      const float* a32 = reinterpret_cast<const float*>(sa0);
      float4 x[kPer];
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        const int it = ct + j * kConvWarps * 32;
        if (it < kItems) {
          if (!kAMN) x[j] = *reinterpret_cast<const float4*>(a32 + (it / kQ) * kBK + 4 * (it % kQ));
          else x[j] = *reinterpret_cast<const float4*>(a32 + (it >> 5) * 128 + 4 * (it & 31));
        }
      }
      asm volatile("bar.sync 1, %0;" ::"n"(kConvWarps * 32) : "memory");
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        const int it = ct + j * kConvWarps * 32;
        if (it < kItems) {
          int off;                        // byte offset in a piece tile
          if (!kAMN) {                    // K-major: 128 rows (features) x kBK k
            // 16-byte chunk c of row r sits at chunk c ^ (r mod 8) (128-byte
            // swizzle) or c ^ ((r / 2) mod 4) (64-byte swizzle)
            const int r = it / kQ, q = it % kQ;
            const int sw = kBK == 64 ? (r & 7) : ((r >> 1) & 3);
            off = r * (2 * kBK) + ((((q >> 1) ^ sw)) << 4) + (q & 1) * 8;
          } else {                        // MN-major: kBK k rows x 128 inputs, two 64-wide boxes
            const int f = it >> 5, q = it & 31, mh = q >> 4, qm = q & 15;
            off = mh * kBox + f * 128 + ((((qm >> 1) ^ (f & 7))) << 4) + (qm & 1) * 8;
          }
          const float xv[4] = {x[j].x, x[j].y, x[j].z, x[j].w};
          uint2 q0, q1, q2;
          split3_x4(xv, q0, q1, q2);
          *reinterpret_cast<uint2*>(sa0 + off) = q0;
          *reinterpret_cast<uint2*>(sa0 + kABytes + off) = q1;
          *reinterpret_cast<uint2*>(sa0 + 2 * kABytes + off) = q2;
        }
      }
      tc::fence_proxy_async_smem();       // before the MMAs (async proxy) read them
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&conv[s]);
    }
    pdl_begin();   // before the epilogue's global accesses
  } else if (warp == 1) {
    if (lane == 0) {
      // A in TMEM is read row by row (K-major) whatever the weights' layout
      constexpr uint32_t kIdesc = tc::idesc_bf16_f32(128, BN, kATmem ? false : kAMN, kBMN);
      for (int kt = 0; kt < KT; ++kt) {
        const int s = kt % kStages;
        if (!wait_or_abort(&full[s], (kt / kStages) & 1, abort_flag) ||
            (kWConv && !wait_or_abort(&conv[s], (kt / kStages) & 1, abort_flag))) {
          *abort_flag = 1;
          break;
        }
        tc::tc_fence_after();
        const uint32_t sa0 = tc::smem_u32(smem + s * Cfg::kStageBytes);
        const uint32_t sb0 = sa0 + Cfg::kAArea;
        const uint32_t ta0 = tmem + Cfg::kAccCols + (uint32_t)s * Cfg::kACols;   // A in TMEM
        constexpr int kPairs = kSplit == 1 ? 1 : 6;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
#pragma unroll
          for (int mq = 0; mq < kMT * kPairs; ++mq) {
            const int q = mq % kPairs, mh = mq / kPairs;   // (kMT > 1: kPairs = 1)
            const uint32_t sa = sa0 + (mh * kSplit + (kSplit == 1 ? 0 : kPairA[q])) * kABytes;
            const uint32_t sb = sb0 + (kSplit == 1 ? 0 : kPairB[q]) * Cfg::kBBytes;
            // MN-major: 16 k rows of 128 bytes per k16 step, the two 64-wide
            // boxes kBox apart; K-major: 32 bytes along the row per k16 step,
            // 8-row groups 8 rows apart
            const uint64_t ad = kAMN ? tc::smem_desc_sw128(sa + kk * 2048, kBox, 1024)
                                : kBK == 64 ? tc::smem_desc_sw128(sa + kk * 32, 16, 1024)
                                            : tc::smem_desc_sw64(sa + kk * 32, 16, 512);
            const uint64_t bd = kBMN ? tc::smem_desc_sw128(sb + kk * 2048, kBox, 1024)
                                : kBK == 64 ? tc::smem_desc_sw128(sb + kk * 32, 16, 1024)
                                            : tc::smem_desc_sw64(sb + kk * 32, 16, 512);
            const uint32_t dcol = (kSplit == 3 && q > 0) ? (uint32_t)BN : (uint32_t)(mh * BN);
            const bool acc_on = kSplit == 1 ? (kt | kk | q) != 0
                                            : (q == 0 ? (kt | kk) != 0 : ((kt | kk) != 0 || q > 1));
            if (kATmem)
              tc::mma_bf16_ts(tmem + dcol, ta0 + (uint32_t)(kPairA[q] * (kBK / 2) + kk * 8), bd,
                              kIdesc, acc_on ? 1u : 0u);
            else
              tc::mma_bf16(tmem + dcol, ad, bd, kIdesc, acc_on ? 1u : 0u);
          }
        }
        tc::mma_commit(&empty[s]);
      }
      tc::mma_commit(done);
    }
  }
  __syncwarp();

  // CTA 0 clears the counter arrays the previous launch used (every thread
  // has passed its dependency wait by now; this launch's own arrays were
  // cleared by the launch before it)
  if (blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0) {
    if (args.counter_clear)
      for (int i = threadIdx.x; i < args.counter_clear_n; i += kThreads)
        AGN_ST(args.counter_clear + i, 0);
    if (kEpi == kEpiFwdHead && args.head_counter_clear)
      for (int i = threadIdx.x; i < args.head_counter_clear_n; i += kThreads)
        AGN_ST(args.head_counter_clear + i, 0);
  }
  // block-uniform, so that the epilogue's barriers and warp-wide TMEM loads
  // are reached by every thread or by none
  const bool ok = __syncthreads_and(wait_or_abort(done, 0, abort_flag) && !*abort_flag) != 0;
  tc::tc_fence_after();
  if (!ok) {
    if (threadIdx.x == 0) atomicExch(args.err, 1);
  } else {
    // kMT = 2: the CTA's two row tiles in turn, accumulators BN columns apart
#pragma unroll 1
    for (int mh = 0; mh < kMT; ++mh) {
      const int m_tile = (int)blockIdx.x * kMT + mh;
      const uint32_t tmem = tmem_base + (uint32_t)(mh * BN);
      const int g = warp & 3, half = warp >> 2;
      const int row = 128 * m_tile + 32 * g + lane;   // M index of this thread
      const bool row_ok = row < args.M;
      const uint32_t lane_base = (uint32_t)(32 * g) << 16;
      float* theta = args.theta + (int64_t)worker * args.ld_param;
      // Accumulated values of this thread's row for columns c0 .. c0 + 15: from
      // TMEM (the sum of the two accumulators in the split mode), or, with
      // split K, the partial sums of all ks CTAs of the tile in rank order.
      const int64_t tile_id = ((int64_t)slot * gridDim.y + n_tile) * gridDim.x + m_tile;
      const int trow = 32 * g + lane;
      auto tmem_vals = [&](int c0, uint32_t (&r)[16]) {
        tc::tmem_ld_32x32b_x16(tmem + lane_base + (uint32_t)c0, r);
        if (kSplit == 3) {
          uint32_t r2[16];
          tc::tmem_ld_32x32b_x16(tmem + lane_base + (uint32_t)(BN + c0), r2);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i)
            r[i] = __float_as_uint(__fadd_rn(__uint_as_float(r[i]), __uint_as_float(r2[i])));
        }
        tc::tmem_ld_wait();
      };
      // Split K (forward / dX): chunk j of the tile (columns 32 j .. 32 j + 31)
      // is finished by rank j % ks.  Every rank stores its partial sums of the
      // chunks it does not finish ([column][row], rows contiguous) and counts
      // itself in on the tile's counter (an array the previous launch cleared).
      // A rank that finishes chunks waits until all ks ranks are in (the CTAs
      // of a launch with ks > 1 are resident together: at most one per SM, no
      // more than the SMs), copies the other ranks' partial sums of its chunks
      // into its stage ring and adds them in rank order, its own from TMEM.
      // Warps 0-3 take columns 0-15 of every chunk, warps 4-7 columns 16-31.
      constexpr int kNch = BN / 32;
      constexpr uint32_t kChunkBytes = 128u * 32u * 4u;
      const bool split_k = kEpi != kEpiDW && ks > 1;
      const int own_rank = split_k ? sk : 0, kstride = split_k ? ks : 1;
      const int n_own = (kNch - own_rank + kstride - 1) / kstride;   // chunks own_rank + o ks
      const int co = 16 * half;                                       // this warp's columns of a chunk
      const float* red_smem = reinterpret_cast<const float*>(smem);   // the free stage ring
      // Forward and dX epilogues: the warp's 32 rows x 16 columns go through a
      // warp-private shared-memory tile (column-major) so that each lane then
      // handles four consecutive rows (features, contiguous in memory) of four
      // columns: 16-byte bias / mask loads, 16-byte stores of the output and
      // 8-byte stores of each bf16 piece.
      float* tT = reinterpret_cast<float*>(smem + Epi::kOff) +
                  warp * (32 * 32);
      const int r4 = (lane & 7) * 4, jl = lane >> 3;          // rows r4 .. r4 + 3, columns jl + 4 u
      const int row4 = 128 * m_tile + 32 * g + r4;             // first row of this lane
      const bool row4_ok = row4 < args.M;                      // M % 4 == 0: all four or none
      const TAct* mask = kEpi == kEpiDX
                             ? static_cast<const TAct*>(args.mask) + (int64_t)slot * args.mask_bstride
                             : nullptr;
      // the mask of the warp's first columns (and the bias) are loaded before
      // the split-K exchange: they do not depend on it
      float4 hm[4];
      auto load_mask = [&](int c0) {
        if (kEpi == kEpiDX && row4_ok) {   // all mask loads in flight before any store
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = n_tile * BN + c0 + jl + 4 * u;
            hm[u] = j < args.N ? load4(mask + (int64_t)j * args.ldo + row4)
                               : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
      };
      constexpr bool kFwd = kEpi == kEpiFwd || kEpi == kEpiFwdHead;
      float4 bias4 = make_float4(0.f, 0.f, 0.f, 0.f);
      if (kFwd && row4_ok && n_own > 0)
        bias4 = AGN_LD(reinterpret_cast<const float4*>(theta + args.boff + row4));
      if (n_own > 0) load_mask(32 * own_rank + co);
      // fused output layer: this tile's 128 columns of W_L (kHC x 128, zero past
      // C and M), loads in flight across the split-K exchange
      constexpr int kW3Per = kHC * 128 / kThreads;
      float w3v_reg[kEpi == kEpiFwdHead ? kW3Per : 1];
      if (kEpi == kEpiFwdHead) {
        const float* w3g = theta + args.head_woff;
#pragma unroll
        for (int k = 0; k < kW3Per; ++k) {
          const int i = threadIdx.x + k * kThreads;
          const int c = i >> 7, rr = 128 * m_tile + (i & 127);
          w3v_reg[k] = (c < args.head_C && rr < args.M) ? AGN_LD(w3g + (int64_t)c * args.M + rr) : 0.f;
        }
      }
      bool have = true;   // the other ranks' partial sums of this CTA's chunks are in the ring
      if (split_k) {
        float* mine = args.part + (tile_id * ks + sk) * (int64_t)(128 * BN);
#pragma unroll 1
        for (int j = 0; j < kNch; ++j) {
          if (j % ks == sk) continue;
          uint32_t r[16];
          tmem_vals(32 * j + co, r);
#pragma unroll
          for (int i = 0; i < 16; ++i)
            AGN_STCG(mine + (int64_t)(32 * j + co + i) * 128 + trow, __uint_as_float(r[i]));
        }
        // the CTA's stores, ordered by the barrier, are released by one
        // acquire-release arrival; the wait acquires the other ranks'
        __shared__ int s_have;
        __syncthreads();
        if (threadIdx.x == 0) {
          int* ctr = args.counter + tile_id;
          bool got = AGN_BOUNDS_OK(ctr, 4);
          if (!got) AGN_BOUNDS_FAIL(ctr);   // bounds-checked build: no wait on a stray counter
          if (got && sk + 1 != args.withhold_rank) tc::atomic_add_acq_rel_gpu(ctr, 1);
          if (got && n_own > 0) {
            got = tc::wait_count_low(ctr, ks, abort_flag, args.wait_ns ? args.wait_ns : kWaitNs);
            if (got) {
              tc::fence_proxy_async_global();   // the ranks' stores, before the bulk reads
              tc::mbar_arrive_expect_tx(red, kChunkBytes * (uint32_t)(n_own * (ks - 1)));
              for (int o = 0, d = 0; o < n_own; ++o) {
                const int j = sk + o * ks;
                for (int q = 0; q < ks; ++q) {
                  if (q == sk) continue;
                  const float* src = args.part + (tile_id * ks + q) * (int64_t)(128 * BN) +
                                     (int64_t)j * (32 * 128);
                  if (AGN_BOUNDS_OK(src, kChunkBytes)) {
                    tc::bulk_load(smem + (size_t)d * kChunkBytes, src, kChunkBytes, red);
                  } else {   // bounds-checked build: account for the bytes, skip the copy
                    AGN_BOUNDS_FAIL(src);
                    tc::mbar_complete_tx(red, kChunkBytes);
                  }
                  ++d;
                }
              }
            }
          }
          s_have = got;
        }
        __syncthreads();
        have = s_have != 0;
        if (have && n_own > 0) have = __syncthreads_and(wait_or_abort(red, 0, abort_flag)) != 0;
        if (threadIdx.x == 0 && !have) atomicExch(args.err, 1);   // gave up: report, skip the epilogue
      }
      // the accumulated values of this thread's row for columns c0 .. c0 + 15
      // of chunk j = own_rank + o ks (c0 = 32 j + co)
      auto vals = [&](int o, int c0, uint32_t (&r)[16]) {
        tmem_vals(c0, r);
        if (!split_k) return;
        float v[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
        for (int q = 0, d = 0; q < ks; ++q) {
          if (q == sk) {
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += __uint_as_float(r[i]);
          } else {
            const float* pq = red_smem + (size_t)(o * (ks - 1) + d) * (32 * 128) + co * 128 + trow;
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] += pq[i * 128];
            ++d;
          }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) r[i] = __float_as_uint(v[i]);
      };
      // fused output layer: W_L's rows for this tile's 128 features, the number
      // of 32-sample chunks with samples, and the scratch
      float* sW3 = reinterpret_cast<float*>(smem + Epi::kHeadOff);
      float* sPart = sW3 + kHC * 128;
      float* sG = sPart + 8 * 16 * kHC;
      uint16_t* sMask = reinterpret_cast<uint16_t*>(sG + 32 * kHC);   // [owned chunk][thread]
      const int nchk = (args.N + 31) / 32;
      if (kEpi == kEpiFwdHead && have) {
#pragma unroll
        for (int k = 0; k < kW3Per; ++k) sW3[threadIdx.x + k * kThreads] = w3v_reg[k];
        __syncthreads();
      }
      if (!have) {
        // reported above
      } else if (kEpi == kEpiFwd || kEpi == kEpiDX || kEpi == kEpiFwdHead) {
        TAct* out = static_cast<TAct*>(args.out) + (int64_t)slot * args.out_bstride;
#pragma unroll 1
        for (int o = 0; o < n_own; ++o) {
          const int c0 = 32 * (own_rank + o * kstride) + co;
          if (o > 0) load_mask(c0);
          uint32_t r[16];
          vals(o, c0, r);
#pragma unroll
          for (int i = 0; i < 16; ++i) tT[i * 32 + lane] = __uint_as_float(r[i]);
          __syncwarp();
          if (kEpi == kEpiFwdHead && (c0 - co) / 32 < nchk) {
            // Pass 1 of the fused output layer, before this chunk's stores (so
            // that the release below orders only the partials): this CTA's
            // share of the chunk's logits, sum over its 128 features of
            // H_{L-1}[j][f] W_L[c][f].  A lane sums its four features; the eight
            // lanes of a column fold by a fixed shuffle tree; the four row
            // quadrants of a column half are added in order below.  The ReLU
            // mask of the lane's 4 x 4 values goes to shared memory for pass 2.
            // This code runs once per chunk and launch, from a cold instruction
            // cache: it loops over the lane's four columns (u) rather than
            // unrolling them, which keeps it a quarter of the size.
            const int C = args.head_C;
            uint32_t mbits = 0;
            // W_L rows past C are zero in shared memory: all kHC classes are
            // summed unguarded, as independent chains
            const float4* w3v = reinterpret_cast<const float4*>(sW3 + 32 * g + r4);
#pragma unroll 1
            for (int u = 0; u < 4; ++u) {
              const int j = n_tile * BN + c0 + jl + 4 * u;
              float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
              if (row4_ok && j < args.N) {
                a = *reinterpret_cast<const float4*>(tT + (jl + 4 * u) * 32 + r4);
                a.x = fmaxf(a.x + bias4.x, 0.f);
                a.y = fmaxf(a.y + bias4.y, 0.f);
                a.z = fmaxf(a.z + bias4.z, 0.f);
                a.w = fmaxf(a.w + bias4.w, 0.f);
              }
              const float hq[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
              for (int e = 0; e < 4; ++e)   // the mask of the value as stored
                mbits |= (static_cast<float>(static_cast<TAct>(hq[e])) > 0.f ? 1u : 0u)
                         << (4 * u + e);
              float zp[kHC];
#pragma unroll
              for (int c = 0; c < kHC; ++c) {
                const float4 w = w3v[c * 32];
                float t = hq[0] * w.x;
                t = fmaf(hq[1], w.y, t);
                t = fmaf(hq[2], w.z, t);
                zp[c] = fmaf(hq[3], w.w, t);
              }
              // fold the eight lanes of the column (lane bits 0-2) by a fixed
              // reduce-scatter: each round a lane keeps half of its classes and
              // adds its partner's share of them; afterwards the lane holds the
              // column's sums of classes kb and kb + 1, kb = 8 b2 + 4 b1 + 2 b0
              static_assert(kHC == 16, "the reduce-scatter folds 16 classes");
              const int b2 = (lane >> 2) & 1, b1 = (lane >> 1) & 1, b0 = lane & 1;
              float k8[8], k4[4], k2[2];
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const float keep = b2 ? zp[k + 8] : zp[k], send = b2 ? zp[k] : zp[k + 8];
                k8[k] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
              }
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const float keep = b1 ? k8[k + 4] : k8[k], send = b1 ? k8[k] : k8[k + 4];
                k4[k] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
              }
#pragma unroll
              for (int k = 0; k < 2; ++k) {
                const float keep = b0 ? k4[k + 2] : k4[k], send = b0 ? k4[k] : k4[k + 2];
                k2[k] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
              }
              *reinterpret_cast<float2*>(sPart + (warp * 16 + jl + 4 * u) * kHC + 8 * b2 + 4 * b1 +
                                         2 * b0) = make_float2(k2[0], k2[1]);
            }
            sMask[o * kThreads + threadIdx.x] = (uint16_t)mbits;
            __syncthreads();
            const int chunk = (c0 - co) / 32;
            float* gp = args.head_part +
                        (((int64_t)slot * nchk + chunk) * gridDim.x + m_tile) * (32 * kHC);
            for (int i = threadIdx.x; i < 32 * kHC; i += kThreads) {
              const int cc = i / kHC, c = i % kHC, hf = cc >> 4, jcl = cc & 15;
              float sum = 0.f;
              if (c < C)
                for (int gq = 0; gq < 4; ++gq) sum += sPart[((gq + 4 * hf) * 16 + jcl) * kHC + c];
              AGN_STCG(gp + i, sum);
            }
            __syncthreads();
            // count in: the CTA's partials, ordered before by the barrier, are
            // released by one acquire-release arrival
            if (threadIdx.x == 0) {
              int* hc = args.head_counter + slot * nchk + chunk;
              if (AGN_BOUNDS_OK(hc, 4)) tc::atomic_add_acq_rel_gpu(hc, 1);
              else AGN_BOUNDS_FAIL(hc);
            }
          }
          if (row4_ok) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const int jc = jl + 4 * u;
              const int j = n_tile * BN + c0 + jc;
              if (j < args.N) {
                const float4 a = *reinterpret_cast<const float4*>(tT + jc * 32 + r4);
                float v[4] = {a.x, a.y, a.z, a.w};
                if (kFwd) {
                  v[0] += bias4.x; v[1] += bias4.y; v[2] += bias4.z; v[3] += bias4.w;
                  if (args.relu) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) v[e] = fmaxf(v[e], 0.f);
                  }
                } else {
                  const float hv[4] = {hm[u].x, hm[u].y, hm[u].z, hm[u].w};
#pragma unroll
                  for (int e = 0; e < 4; ++e) v[e] = hv[e] > 0.f ? v[e] : 0.f;
                }
                const int64_t o4 = (int64_t)j * args.ldo + row4;
                store4(out + o4, v);
                if (kSplit == 3 && args.out_pieces) {
                  uint2 q0, q1, q2;
                  split3_x4(v, q0, q1, q2);
                  bf16* pp = args.out_pieces + (int64_t)slot * args.out_bstride + o4;
                  AGN_ST(reinterpret_cast<uint2*>(pp), q0);
                  AGN_ST(reinterpret_cast<uint2*>(pp + args.out_plane), q1);
                  AGN_ST(reinterpret_cast<uint2*>(pp + 2 * args.out_plane), q2);
                }
              }
            }
          }
          __syncwarp();
        }
        if (kEpi == kEpiFwdHead) {
          // Pass 2: once every feature tile's partials of a chunk are in (all
          // CTAs of this launch are resident), the chunk's logits are summed in
          // tile order plus b_L; every half-warp takes softmax cross-entropy and
          // dZ_L = (softmax - onehot(y)) / m of a sample (the first feature tile
          // writes dZ_L and the chunk's loss); every CTA then writes dZ_{L-1} =
          // (dZ_L W_L) [H_{L-1} > 0] for its own features (W_L before its
          // update).
          __shared__ int s_hok;
          const int C = args.head_C;
          const float* bl = theta + args.head_boff;
          TAct* dh = static_cast<TAct*>(args.dh) + (int64_t)slot * args.out_bstride;
          const int mtn = (int)gridDim.x;
#pragma unroll 1
          for (int o = 0; o < n_own; ++o) {
            const int chunk = own_rank + o * kstride;
            if (chunk >= nchk) continue;   // CTA-uniform
            int* ctr = args.head_counter + slot * nchk + chunk;
            if (threadIdx.x == 0)
              s_hok = AGN_BOUNDS_OK(ctr, 4) &&
                      tc::wait_count_low(ctr, mtn, abort_flag, args.wait_ns ? args.wait_ns : kWaitNs);
            __syncthreads();
            if (!s_hok) {
              if (threadIdx.x == 0) atomicExch(args.err, 1);
              break;
            }
            // the feature tiles' partials in tile order: each thread sums two of
            // the chunk's 32 x kHC logits, up to 2 x 16 loads in flight; thread
            // t holds class t % kHC of samples t / kHC and 16 + t / kHC, so the
            // 16 lanes of a half-warp hold one sample's logits
            static_assert(32 * kHC == 2 * kThreads, "two logits per thread");
            static_assert(kHC == 16, "one sample per half-warp");
            const float* gp0 = args.head_part + ((int64_t)slot * nchk + chunk) * mtn * (32 * kHC);
            float zz[2] = {0.f, 0.f};
            for (int m0 = 0; m0 < mtn; m0 += 16) {
              float p0[16], p1[16];
#pragma unroll
              for (int q = 0; q < 16; ++q) {
                const float* pq = gp0 + (int64_t)(m0 + q) * (32 * kHC) + threadIdx.x;
                p0[q] = m0 + q < mtn ? AGN_LDCG(pq) : 0.f;
                p1[q] = m0 + q < mtn ? AGN_LDCG(pq + kThreads) : 0.f;
              }
#pragma unroll
              for (int q = 0; q < 16; ++q) {
                zz[0] += p0[q];
                zz[1] += p1[q];
              }
            }
            // softmax cross-entropy and dZ_L = (softmax - onehot(y)) / m of the
            // thread's two (sample, class) entries: max and sum over the
            // sample's classes by a fixed shuffle tree within the half-warp;
            // the first feature tile writes dZ_L
            float* sCE = sPart;   // [32] per-sample cross-entropy (pass 1 is done with sPart)
            {
              const int cl = threadIdx.x % kHC;
              const bool cv = cl < C;
              const float inv_m = 1.0f / (float)args.N;
              const float bc = cv ? AGN_LD(bl + cl) : 0.f;
#pragma unroll 1
              for (int hh = 0; hh < 2; ++hh) {
                const int sl = 16 * hh + (threadIdx.x >> 4);   // sample within the chunk
                const int j = n_tile * BN + 32 * chunk + sl;
                const bool valid = j < args.N;
                const float z = cv ? (hh ? zz[1] : zz[0]) + bc : -INFINITY;
                float mx = z;
#pragma unroll
                for (int off = 8; off > 0; off >>= 1)
                  mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
                const float ex = cv ? expf(z - mx) : 0.f;
                float se = ex;
#pragma unroll
                for (int off = 8; off > 0; off >>= 1) se += __shfl_xor_sync(0xffffffffu, se, off);
                const int y = !valid ? -1
                              : args.x_shard > 0
                                  ? AGN_LD(args.yb + (int64_t)worker * (args.x_shard + args.N) +
                                           batch_row0(args.slot_t0, slot, args.step, args.N,
                                                      args.x_shard) + j)
                                  : AGN_LD(args.yb + (int64_t)slot * args.N + j);
                const float zy = __shfl_sync(0xffffffffu, z, (lane & 16) + (y > 0 ? y : 0));
                float pr = ex * (1.0f / se);
                if (cl == y) pr -= 1.0f;
                const float gz = valid ? pr * inv_m : 0.f;
                sG[sl * kHC + cl] = gz;
                if (m_tile == 0 && valid && cv) {
                  const TAct gv = static_cast<TAct>(gz);
                  const int64_t zi = ((int64_t)slot * args.N + j) * args.ldz + cl;
                  AGN_ST(static_cast<TAct*>(args.dzl) + zi, gv);
                  if (args.dzl_pieces) {
                    bf16 q0, q1, q2;
                    split3(static_cast<float>(gv), q0, q1, q2);
                    AGN_ST(args.dzl_pieces + zi, q0);
                    AGN_ST(args.dzl_pieces + args.dzl_plane + zi, q1);
                    AGN_ST(args.dzl_pieces + 2 * args.dzl_plane + zi, q2);
                  }
                }
                if (cl == 0) sCE[sl] = valid ? (logf(se) + mx) - zy : 0.f;
              }
            }
            __syncthreads();
            float ce = 0.f;
            if (warp == 0) {   // the chunk's cross-entropy sum, fixed tree over its samples
              ce = sCE[lane];
#pragma unroll
              for (int off = 16; off > 0; off >>= 1) ce += __shfl_xor_sync(0xffffffffu, ce, off);
            }
            if (row4_ok) {
              const uint32_t mbits = sMask[o * kThreads + threadIdx.x];
              const float4* w3v = reinterpret_cast<const float4*>(sW3 + 32 * g + r4);
              // dZ_{L-1} of the lane's 4 features x 4 columns: 16 independent
              // chains over the classes (dZ_L is zero past C)
              float d[4][4];
#pragma unroll
              for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int e = 0; e < 4; ++e) d[u][e] = 0.f;
#pragma unroll 2
              for (int c = 0; c < kHC; ++c) {
                const float4 w = w3v[c * 32];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                  const float gzc = sG[(co + jl + 4 * u) * kHC + c];
                  d[u][0] = fmaf(gzc, w.x, d[u][0]);
                  d[u][1] = fmaf(gzc, w.y, d[u][1]);
                  d[u][2] = fmaf(gzc, w.z, d[u][2]);
                  d[u][3] = fmaf(gzc, w.w, d[u][3]);
                }
              }
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const int j = n_tile * BN + 32 * chunk + co + jl + 4 * u;
                if (j < args.N) {
                  float dv[4];
#pragma unroll
                  for (int e = 0; e < 4; ++e) dv[e] = (mbits >> (4 * u + e)) & 1u ? d[u][e] : 0.f;
                  const int64_t o4 = (int64_t)j * args.ldo + row4;
                  store4(dh + o4, dv);
                  if (kSplit == 3 && args.dh_pieces) {
                    uint2 q0, q1, q2;
                    split3_x4(dv, q0, q1, q2);
                    bf16* pp = args.dh_pieces + (int64_t)slot * args.out_bstride + o4;
                    AGN_ST(reinterpret_cast<uint2*>(pp), q0);
                    AGN_ST(reinterpret_cast<uint2*>(pp + args.dh_plane), q1);
                    AGN_ST(reinterpret_cast<uint2*>(pp + 2 * args.dh_plane), q2);
                  }
                }
              }
            }
            if (threadIdx.x == 0) {
              // the chunk's loss contribution (sum of its samples' cross-entropy
              // over m) in the chunk's slot; the run's loss kernel adds the slots
              // in order
              if (m_tile == 0) {
                const float part = ce / (float)args.N;
                AGN_ST(args.loss_parts +
                           ((int64_t)AGN_LD(args.slot_commit + slot) * args.lam + args.step) * nchk +
                           chunk,
                       part);
                if (!isfinite(part)) atomicExch(args.nonfinite, 1);
              }
            }
          }
        }
      } else {   // kEpiDW
        float* acc = args.acc + (int64_t)worker * args.ld_param;
        bf16* tb = args.theta_b + (int64_t)worker * args.ld_param;
        const float eta = args.eta;
        // Chunks of 16 columns; the loads of chunk c + 1 are issued before the
        // stores of chunk c, so every thread keeps 32 loads in flight while it
        // writes (the epilogue is bound by DRAM latency x bandwidth).
        constexpr int kCh = 16;
        constexpr int kChunks = (BN / 2) / kCh;
        const float* __restrict__ th_in = theta;
        const float* __restrict__ ac_in = acc;
        const int cbase = n_tile * BN + half * (BN / 2);     // first column of this half
        const int64_t pbase = args.woff + (int64_t)cbase * args.M + row;
        float thn[kCh], acn[kCh];
        auto load_chunk = [&](int ch) {
          const int nvalid = row_ok ? min(kCh, args.N - (cbase + ch * kCh)) : 0;
#pragma unroll
          for (int i = 0; i < kCh; ++i) {
            if (i < nvalid) {
              const int64_t p = pbase + (int64_t)(ch * kCh + i) * args.M;
              thn[i] = AGN_LDCS(th_in + p);
              acn[i] = AGN_LDCS(ac_in + p);
            }
          }
        };
        load_chunk(0);
#pragma unroll
        for (int ch = 0; ch < kChunks; ++ch) {
          float th[kCh], ac[kCh];
#pragma unroll
          for (int i = 0; i < kCh; ++i) {
            th[i] = thn[i];
            ac[i] = acn[i];
          }
          uint32_t r[kCh];
          const uint32_t col = (uint32_t)(half * (BN / 2) + ch * kCh);
          tc::tmem_ld_32x32b_x16(tmem + lane_base + col, r);
          uint32_t r2[kCh];
          if (kSplit == 3) tc::tmem_ld_32x32b_x16(tmem + lane_base + (uint32_t)BN + col, r2);
          if (ch + 1 < kChunks) load_chunk(ch + 1);
          tc::tmem_ld_wait();
          if (kSplit == 3) {
#pragma unroll
            for (int i = 0; i < kCh; ++i)
              r[i] = __float_as_uint(__fadd_rn(__uint_as_float(r[i]), __uint_as_float(r2[i])));
          }
          const int nvalid = row_ok ? min(kCh, args.N - (cbase + ch * kCh)) : 0;
#pragma unroll
          for (int i = 0; i < kCh; ++i) {
            if (i < nvalid) {
              const int64_t p = pbase + (int64_t)(ch * kCh + i) * args.M;
              const float gr = __uint_as_float(r[i]);
              const float t = local_step(th[i], eta, gr);
              AGN_ST(theta + p, t);
              AGN_ST(acc + p, ac[i] + gr);
              if (kSplit == 1) AGN_ST(tb + p, __float2bfloat16_rn(t));   // fp32 mode: no pieces
            }
          }
        }
      }
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) tc::tmem_dealloc(tmem, Cfg::kTmemCols);
}

// Bias gradient and update for a hidden layer: g_b[f] = sum_j dZ[j][f];
// b -= eta g_b, a_b += g_b, and the bf16 copy (or its three pieces).  A block
// covers 32 features of one slot: its 8 warps sum interleaved sample groups
// (coalesced rows of dZ), then one warp adds the 8 partials in a fixed order.
constexpr int kBiasGroups = 8;
template <typename TD, int kSplit>
__global__ void __launch_bounds__(32 * kBiasGroups)
bias_update_kernel(const TD* __restrict__ dz, int m, int d, int64_t dz_bstride,
                   const int* __restrict__ slot_worker, float* theta, float* acc,
                   bf16* theta_b, int64_t ld_param, int64_t boff, float eta,
                   int64_t piece_plane) {
  pdl_begin();
  __shared__ float red[kBiasGroups][32];
  const int fx = threadIdx.x & 31, gy = threadIdx.x >> 5;
  const int f = blockIdx.x * 32 + fx;
  const int z = blockIdx.y;
  const TD* col = dz + (int64_t)z * dz_bstride + f;
  float part = 0.f;
  if (f < d)
    for (int j = gy; j < m; j += kBiasGroups) part += from_act(AGN_LD(col + (int64_t)j * d));
  red[gy][fx] = part;
  __syncthreads();
  if (gy != 0 || f >= d) return;
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < kBiasGroups; ++q) s += red[q][fx];
  const int64_t p = (int64_t)AGN_LD(slot_worker + z) * ld_param + boff + f;
  const float t = local_step(AGN_LD(theta + p), eta, s);
  AGN_ST(theta + p, t);
  AGN_ST(acc + p, AGN_LD(acc + p) + s);
  if (kSplit == 1 && theta_b) AGN_ST(theta_b + p, __float2bfloat16_rn(t));   // fp32 mode: no pieces
}

// out[p * plane + i] = piece p of x[i] (x = piece 0 + piece 1 + piece 2 exactly).
__global__ void split_pieces_kernel(const float* __restrict__ x, bf16* __restrict__ out,
                                    int64_t count, int64_t plane) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count; i += stride) {
    bf16 q0, q1, q2;
    split3(AGN_LD(x + i), q0, q1, q2);
    AGN_ST(out + i, q0);
    AGN_ST(out + plane + i, q1);
    AGN_ST(out + 2 * plane + i, q2);
  }
}

template <int BN, int kSplit, int kStages, int kBK, bool kATmem, int kMT = 1>
size_t smem_bytes() {
  // Shared memory requested per CTA also caps the CTAs per SM so that their
  // TMEM columns never exceed the 512 an SM has.
  using Cfg = TileCfg<BN, kSplit, kBK, kATmem, kMT>;
  const size_t ring = (size_t)kStages * Cfg::kStageBytes + 1024 + 256 +
                      (EpiT<BN, kSplit, kStages, kBK, kATmem, kMT>::kSeparate ? kEpiTBytes : 0);
  const size_t floor_for_tmem = (size_t)(233472 / (512 / Cfg::kTmemCols + 1)) + 1024;
  return std::max(ring, floor_for_tmem);
}

template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages, int kSplit, int kMT = 1>
Status launch_tc(const CUtensorMap& a, const CUtensorMap& b, const TcArgs& args, int slots,
                 cudaStream_t st, bool* launched = nullptr) {
  constexpr int kBK = stage_k(kSplit, kEpi);
  constexpr bool kATmem = a_in_tmem(kSplit, kEpi, BN);
  using Epi = EpiT<BN, kSplit, kStages, kBK, kATmem, kMT>;
  static_assert(kStages * TileCfg<BN, kSplit, kBK, kATmem, kMT>::kStageBytes + 1280 <= 232448,
                "smem");
  auto kern = tc_gemm_kernel<BN, kAMN, kBMN, kEpi, kStages, kSplit, kMT>;
  const size_t smem = smem_bytes<BN, kSplit, kStages, kBK, kATmem, kMT>();
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  });
  AGN_TRY_CUDA(attr_err);
  // split K: every rank with a non-empty range of k steps
  int ks = kEpi == kEpiDW || kMT > 1 ? 1 : std::max(1, args.ksplit);
  if (ks > 1) {
    // a rank that finishes chunks holds the other ranks' partial sums of
    // them (16 KB per chunk and rank) in its stage ring
    const int ring = (int)(kEpi == kEpiFwdHead ? Epi::kHeadOff : Epi::kRingFree);
    auto need = [](int k) { return ((BN / 32 + k - 1) / k) * (k - 1) * (128 * 32 * 4); };
    while (ks > 1 && need(ks) > ring) --ks;
    const int kt = (args.K + kBK - 1) / kBK;
    ks = std::min(ks, kt);
    if (ks > 1) ks = (kt + (kt + ks - 1) / ks - 1) / ((kt + ks - 1) / ks);
  }
  if (ks > 1 || kEpi == kEpiFwdHead) {
    // the split-K exchange and the fused output layer's wait need every CTA
    // of the launch resident at once (one CTA per SM: see smem_bytes)
    int dev = 0, sms = 0;
    AGN_TRY_CUDA(cudaGetDevice(&dev));
    AGN_TRY_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    const int64_t tiles = (int64_t)ceil_div(args.M, 128) * ceil_div(args.N, BN) * slots;
    if (tiles * ks > sms) ks = 1;
    if (kEpi == kEpiFwdHead && (tiles > sms || ceil_div(args.N, BN) != 1)) {
      if (launched) *launched = false;
      return Status::Ok();
    }
  }
  if (ks > 1 && (!args.part || !args.counter))
    return Status::Err(AGN_E_INVALID, "split-K GEMM without workspace");
  dim3 grid((unsigned)ceil_div(args.M, 128 * kMT), (unsigned)ceil_div(args.N, BN),
            (unsigned)(slots * ks));
  TcArgs a2 = args;
  a2.ksplit = ks;
  {
    auto kf = kern;
    AGN_TRY_CUDA(launch_pdl(kf, grid, kThreads, smem, st, a, b, a2));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  if (launched) *launched = true;
  return Status::Ok();
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

Status encode(CUtensorMap* map, int rank, const void* base, const cuuint64_t* dims,
              const cuuint64_t* strides_bytes, const cuuint32_t* box,
              CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, int esize = 2,
              CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  AGN_TRY(tc_init());
  if (reinterpret_cast<uintptr_t>(base) & 15)
    return Status::Err(AGN_E_UNSUPPORTED, "tensor map base not 16-byte aligned");
  if ((dims[0] * esize) % 16)
    return Status::Err(AGN_E_UNSUPPORTED, "tensor map rows not 16-byte aligned");
  if ((box[0] * esize) % 16)
    return Status::Err(AGN_E_UNSUPPORTED, "tensor map box rows not a multiple of 16 bytes");
  for (int i = 0; i < rank - 1; ++i)
    if (strides_bytes[i] % 16)
      return Status::Err(AGN_E_UNSUPPORTED, "tensor map stride not a multiple of 16 bytes");
#ifdef AGN_BOUNDS_CHECK
  {   // bounds-checked build: the whole span the map addresses lies in one known buffer
    size_t span = (size_t)dims[0] * esize;
    for (int i = 1; i < rank; ++i) span += (size_t)(dims[i] - 1) * strides_bytes[i - 1];
    if (!bounds_host_ok(base, span))
      return Status::Err(AGN_E_BOUNDS, "bounds-checked build: a tensor map spans " +
                                           std::to_string(span) + " bytes beyond a known buffer");
  }
#endif
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  CUresult r = g_encode(map, dtype, rank, const_cast<void*>(base), dims, strides_bytes, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return Status::Err(AGN_E_CUDA, "cuTensorMapEncodeTiled failed with code " + std::to_string(r));
  return Status::Ok();
}

}  // namespace

Status tc_init() {
  static std::once_flag once;
  static Status st = Status::Ok();
  std::call_once(once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e =
        cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
      st = Status::Err(AGN_E_UNSUPPORTED, "cuTensorMapEncodeTiled not available from the driver");
    else
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return st;
}

Status make_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                         uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                         uint32_t box_inner, uint32_t box_rows) {
  cuuint64_t dims[3] = {inner, rows, batch};
  cuuint64_t strides[2] = {row_stride_elems * 2, batch_stride_elems * 2};
  cuuint32_t box[3] = {box_inner, box_rows, 1};
  return encode(map, 3, base, dims, strides, box);
}

Status make_tmap_bf16_4d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                         uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                         uint64_t piece_stride_elems, uint32_t box_inner, uint32_t box_rows) {
  cuuint64_t dims[4] = {inner, rows, batch, 3};
  cuuint64_t strides[3] = {row_stride_elems * 2, batch_stride_elems * 2, piece_stride_elems * 2};
  cuuint32_t box[4] = {box_inner, box_rows, 1, 1};
  // rows of 64 bytes take the 64-byte swizzle, rows of 128 bytes the 128-byte one
  return encode(map, 4, base, dims, strides, box, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                box_inner * 2 == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B);
}

Status make_tmap_f32_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                        uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                        uint32_t box_inner, uint32_t box_rows, bool swizzle128) {
  cuuint64_t dims[3] = {inner, rows, batch};
  cuuint64_t strides[2] = {row_stride_elems * 4, batch_stride_elems * 4};
  cuuint32_t box[3] = {box_inner, box_rows, 1};
  return encode(map, 3, base, dims, strides, box, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4,
                swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE);
}

// Two 128-row tiles per CTA (kMT = 2) for the bf16 forward and dX when the
// one-tile launch would need more than one round of CTAs on the SMs (full
// waves): each B stage then feeds twice the MMAs, and the CTAs of a full
// wave halve.  Not with split K, nor with column tiles under 128 (there the
// weights, read once anyway, dominate the stages' bytes).
bool use_row_pairs(const TcArgs& args, int slots, bool split, int bn) {
  if (split || bn < 128 || args.ksplit > 1 || args.one_row_tile) return false;
  static int sms = 0;
  if (sms == 0) {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      (void)cudaGetLastError();
      return false;
    }
    sms = n;
  }
  return ceil_div(args.M, 128) * ceil_div(args.N, bn) * (int64_t)slots > sms;
}

Status tc_forward(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args, int slots,
                  cudaStream_t st, bool split, int bn) {
  if (split) {
    if (bn == 64) return launch_tc<64, false, false, kEpiFwd, 6, 3>(w_k, h_k, args, slots, st);
    if (bn == 128) return launch_tc<128, false, false, kEpiFwd, 4, 3>(w_k, h_k, args, slots, st);
    return launch_tc<256, false, false, kEpiFwd, 3, 3>(w_k, h_k, args, slots, st);
  }
  if (use_row_pairs(args, slots, split, bn)) {
    if (bn == 128) return launch_tc<128, false, false, kEpiFwd, 4, 1, 2>(w_k, h_k, args, slots, st);
    return launch_tc<256, false, false, kEpiFwd, 3, 1, 2>(w_k, h_k, args, slots, st);
  }
  if (bn == 64) return launch_tc<64, false, false, kEpiFwd, 6, 1>(w_k, h_k, args, slots, st);
  if (bn == 128) return launch_tc<128, false, false, kEpiFwd, 5, 1>(w_k, h_k, args, slots, st);
  return launch_tc<256, false, false, kEpiFwd, 4, 1>(w_k, h_k, args, slots, st);
}

Status tc_forward_head(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args,
                       int slots, cudaStream_t st, bool split, int bn, int num_sms,
                       bool* launched) {
  *launched = false;
  if (args.head_C < 1 || args.head_C > kHC || !args.head_part || !args.head_counter ||
      !args.dh || !args.dzl || !args.loss_parts)
    return Status::Err(AGN_E_INVALID, "fused output layer without its buffers");
  if ((int64_t)ceil_div(args.M, 128) * slots > num_sms) return Status::Ok();
  if (split) {
    if (bn == 64)
      return launch_tc<64, false, false, kEpiFwdHead, 6, 3>(w_k, h_k, args, slots, st, launched);
    if (bn == 128)
      return launch_tc<128, false, false, kEpiFwdHead, 4, 3>(w_k, h_k, args, slots, st, launched);
    return launch_tc<256, false, false, kEpiFwdHead, 3, 3>(w_k, h_k, args, slots, st, launched);
  }
  if (bn == 64)
    return launch_tc<64, false, false, kEpiFwdHead, 6, 1>(w_k, h_k, args, slots, st, launched);
  if (bn == 128)
    return launch_tc<128, false, false, kEpiFwdHead, 5, 1>(w_k, h_k, args, slots, st, launched);
  return launch_tc<256, false, false, kEpiFwdHead, 4, 1>(w_k, h_k, args, slots, st, launched);
}

Status tc_backward_dx(const CUtensorMap& w_mn, const CUtensorMap& dz_k, const TcArgs& args,
                      int slots, cudaStream_t st, bool split, int bn) {
  if (split) {
    if (bn == 64) return launch_tc<64, true, false, kEpiDX, 6, 3>(w_mn, dz_k, args, slots, st);
    if (bn == 128) return launch_tc<128, true, false, kEpiDX, 4, 3>(w_mn, dz_k, args, slots, st);
    return launch_tc<256, true, false, kEpiDX, 3, 3>(w_mn, dz_k, args, slots, st);
  }
  if (use_row_pairs(args, slots, split, bn)) {
    if (bn == 128) return launch_tc<128, true, false, kEpiDX, 4, 1, 2>(w_mn, dz_k, args, slots, st);
    return launch_tc<256, true, false, kEpiDX, 3, 1, 2>(w_mn, dz_k, args, slots, st);
  }
  if (bn == 64) return launch_tc<64, true, false, kEpiDX, 6, 1>(w_mn, dz_k, args, slots, st);
  if (bn == 128) return launch_tc<128, true, false, kEpiDX, 5, 1>(w_mn, dz_k, args, slots, st);
  return launch_tc<256, true, false, kEpiDX, 4, 1>(w_mn, dz_k, args, slots, st);
}

Status tc_backward_dw_tiled(const CUtensorMap& h_mn, const CUtensorMap& dz_mn, const TcArgs& args,
                            int slots, cudaStream_t st, bool split) {
  if (split) return launch_tc<kTcDwBNSplit, true, true, kEpiDW, 1, 3>(h_mn, dz_mn, args, slots, st);
  return launch_tc<kTcDwBN, true, true, kEpiDW, 2, 1>(h_mn, dz_mn, args, slots, st);
}

Status bias_update(const void* dz, int m, int d, int64_t dz_bstride, const int* slot_worker,
                   float* theta, float* acc, bf16* theta_b, int64_t ld_param, int64_t boff,
                   float eta, int slots, cudaStream_t st, bool split, int64_t piece_plane) {
  dim3 grid((unsigned)ceil_div(d, 32), (unsigned)slots);
  const int threads = 32 * kBiasGroups;
  if (split)
    {
      auto kf = bias_update_kernel<float, 3>;
      AGN_TRY_CUDA(launch_pdl(kf, grid, threads, 0, st, static_cast<const float*>(dz),
                              m, d, dz_bstride, slot_worker, theta, acc, theta_b, ld_param, boff,
                              eta, piece_plane));
    }
  else
    {
      auto kf = bias_update_kernel<bf16, 1>;
      AGN_TRY_CUDA(launch_pdl(kf, grid, threads, 0, st, static_cast<const bf16*>(dz),
                              m, d, dz_bstride, slot_worker, theta, acc, theta_b, ld_param, boff,
                              eta, piece_plane));
    }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

Status split_pieces(const float* x, bf16* out, int64_t count, int64_t plane, cudaStream_t st) {
  if (count <= 0) return Status::Ok();
  const int grid = (int)std::min<int64_t>(ceil_div(count, 256), 152 * 8);
  {
    auto kf = split_pieces_kernel;
    AGN_TRY_CUDA(launch_pdl(kf, grid, 256, 0, st, x, out, count, plane));
  }
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

AGN_BOUNDS_UNIT(tc)

}  // namespace agn
