// Kernel (b), weight-gradient half, on the tensor cores: D = H_{l-1}^T dZ_l
// for every slot of a wave, fused with Algorithm 1's local step and
// accumulation (theta_k -= eta g, a_k += g, and the bf16 copy of theta_k).
//
// The GEMM is tiny next to its epilogue (K = m samples against 18-22 bytes
// of fp32 master weight and accumulator traffic per parameter), so the kernel
// is laid out around the parameter stream, not the MMA:
//
//   warp 0     TMA producer.  Per tile, the GEMM operands (H^T and dZ^T
//              boxes, MN-major, 128-byte swizzle) into a ring of stages, then
//              the tile's theta_k and a_k rows, 32 output features x 128
//              inputs per chunk, into a second ring.  Each slot is refilled
//              as soon as it frees, so DRAM reads of the next chunks (and of
//              the next tile) are in flight while the current one is updated.
//   warp 1     MMA issuer (one thread) and TMEM owner.  Two accumulators
//              (double buffer): the GEMM of the next tile runs while the
//              epilogue drains this one.
//   warps 2-5  epilogue.  Warp w reads TMEM lanes 32 (w % 4) .. + 31, i.e.
//              32 consecutive inputs k of the tile, one chunk of 32 features
//              at a time, takes theta_k and a_k from shared memory and stores
//              the new values coalesced (32 consecutive k per feature row).
//
// The kernel is persistent (one CTA per SM: the rings take 192 KB of shared
// memory and the accumulators all 512 TMEM columns); tiles (slot, feature
// tile, input tile) are dealt out round-robin with input tiles fastest, so
// neighbouring CTAs stream neighbouring parts of the same weight rows.
// Every wait is bounded (2 s of global time): on expiry the CTA sets *err,
// stops issuing, drains its own copies and MMAs (bounded), frees TMEM and
// returns.
#include <cuda.h>

#include <algorithm>
#include <mutex>

#include "mlp.cuh"
#include "mlp_tc.cuh"
#include "tc_ptx.cuh"

namespace agn {

namespace {

constexpr int kWarps = 6;
constexpr int kThreads = 32 * kWarps;
constexpr int kBK = 64;                        // K (samples) per stage
constexpr int kABytes = 128 * 128;             // A box pair: 128 inputs x 64 samples, bf16
constexpr int kCF = 32;                        // output features per parameter chunk
constexpr int kChunkBytes = kCF * 128 * 4;     // one fp32 chunk: 32 rows x 128 inputs
constexpr int kRing = 3;                       // chunks (theta and a) in flight
constexpr uint64_t kWaitNs = 2000000000ull;    // 2 s

template <int BN, int kSplit, int kStages>
struct DwCfg {
  static constexpr int kBBytes = BN * 128;
  static constexpr int kStageBytes = kSplit * (kABytes + kBBytes);
  // one accumulator: BN columns, or two of BN in the split mode (the leading
  // piece products and the five smaller pairs, kept apart for accuracy)
  static constexpr uint32_t kAccCols = (kSplit == 1 ? 1 : 2) * BN;
  static constexpr uint32_t kTmemCols = 2 * kAccCols;
  static constexpr int kChunks = BN / kCF;
  static constexpr size_t kRingOff = (size_t)kStages * kStageBytes;
  static constexpr size_t kBarOff = kRingOff + (size_t)kRing * 2 * kChunkBytes;
  static constexpr size_t kSmem = kBarOff + 256 + 1024;   // barriers, alignment slack
};

// Piece pairs (i, j), i + j <= 2, of the split product (pair 0 = a0 b0).
__device__ __forceinline__ int pair_a(int q) { return q == 2 || q == 4 ? 1 : q == 5 ? 2 : 0; }
__device__ __forceinline__ int pair_b(int q) { return q == 1 || q == 4 ? 1 : q == 3 ? 2 : 0; }

struct TileIdx {
  int m_tile, n_tile, slot;
};
__device__ __forceinline__ TileIdx decode(int t, int mt, int nt) {
  TileIdx r;
  r.m_tile = t % mt;
  const int rest = t / mt;
  r.n_tile = rest % nt;
  r.slot = rest / nt;
  return r;
}

template <int BN, int kSplit, int kStages>
__global__ void __launch_bounds__(kThreads, 1)
tc_dw_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
             const __grid_constant__ CUtensorMap tmTheta,
             const __grid_constant__ CUtensorMap tmAcc, const TcArgs args, int slots) {
  using Cfg = DwCfg<BN, kSplit, kStages>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + Cfg::kBarOff);
  uint64_t* empty = full + kStages;
  uint64_t* cfull = empty + kStages;     // parameter chunk landed
  uint64_t* cempty = cfull + kRing;      // parameter chunk consumed (4 epilogue warps)
  uint64_t* tfull = cempty + kRing;      // accumulator b complete
  uint64_t* tempty = tfull + 2;          // accumulator b drained (4 epilogue warps)
  uint64_t* fin = tempty + 2;            // MMA drain on abort
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(fin + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  __shared__ int s_skip;
  if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int*>(args.err);
  __syncthreads();
  if (s_skip != 0) return;   // an earlier launch gave up: uniform across the CTA

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int M = args.M, N = args.N;
  const int mt = (M + 127) / 128, nt = (N + BN - 1) / BN;
  const int T = mt * nt * slots;
  const int KT = (args.K + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    for (int r = 0; r < kRing; ++r) {
      tc::mbar_init(&cfull[r], 1);
      tc::mbar_init(&cempty[r], 4);
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(&tfull[b], 1);
      tc::mbar_init(&tempty[b], 4);
    }
    tc::mbar_init(fin, 1);
    *abort_flag = 0;
    tc::fence_mbar_init();
    tc::tma_prefetch_desc(&tmA);
    tc::tma_prefetch_desc(&tmB);
    tc::tma_prefetch_desc(&tmTheta);
    tc::tma_prefetch_desc(&tmAcc);
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_holder, Cfg::kTmemCols);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t ml = 0, ch = 0;   // stage fills and chunk fills issued
      bool ok = true;
      for (int t = blockIdx.x; ok && t < T; t += gridDim.x) {
        const TileIdx ti = decode(t, mt, nt);
        const int worker = args.slot_worker[ti.slot];
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
              tc::tma_load_3d(sa, &tmA, &full[s], ti.m_tile * 128, kt * kBK, ti.slot);
              tc::tma_load_3d(sa + 8192, &tmA, &full[s], ti.m_tile * 128 + 64, kt * kBK, ti.slot);
#pragma unroll
              for (int c = 0; c < BN / 64; ++c)
                tc::tma_load_3d(sb + c * 8192, &tmB, &full[s], ti.n_tile * BN + c * 64, kt * kBK,
                                ti.slot);
            } else {
              tc::tma_load_4d(sa, &tmA, &full[s], ti.m_tile * 128, kt * kBK, ti.slot, p);
              tc::tma_load_4d(sa + 8192, &tmA, &full[s], ti.m_tile * 128 + 64, kt * kBK, ti.slot,
                              p);
#pragma unroll
              for (int c = 0; c < BN / 64; ++c)
                tc::tma_load_4d(sb + c * 8192, &tmB, &full[s], ti.n_tile * BN + c * 64, kt * kBK,
                                ti.slot, p);
            }
          }
          ++ml;
        }
        if (!ok) break;
        const int nch = min(Cfg::kChunks, (N - ti.n_tile * BN + kCF - 1) / kCF);
        for (int c = 0; c < nch; ++c) {
          const int r = ch % kRing;
          if (ch >= kRing &&
              !tc::wait_or_abort(&cempty[r], ((ch / kRing) - 1) & 1, abort_flag, kWaitNs)) {
            ok = false;
            break;
          }
          uint8_t* dst = smem + Cfg::kRingOff + (size_t)r * 2 * kChunkBytes;
          const int f0 = ti.n_tile * BN + c * kCF;
          tc::mbar_arrive_expect_tx(&cfull[r], 2 * kChunkBytes);
          tc::tma_load_3d(dst, &tmTheta, &cfull[r], ti.m_tile * 128, f0, worker);
          tc::tma_load_3d(dst + kChunkBytes, &tmAcc, &cfull[r], ti.m_tile * 128, f0, worker);
          ++ch;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        // drain (bounded) the copies armed but maybe not yet landed
        for (uint32_t j = ml > (uint32_t)kStages ? ml - kStages : 0; j < ml; ++j)
          tc::mbar_wait_bounded(&full[j % kStages], (j / kStages) & 1, kWaitNs);
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
        const int b = it & 1;
        if (it >= 2 && !tc::wait_or_abort(&tempty[b], ((it >> 1) - 1) & 1, abort_flag, kWaitNs)) {
          ok = false;
          break;
        }
        tc::tc_fence_after();
        const uint32_t dbase = tmem + (uint32_t)b * Cfg::kAccCols;
        for (int kt = 0; kt < KT; ++kt) {
          const int s = ml % kStages;
          if (!tc::wait_or_abort(&full[s], (ml / kStages) & 1, abort_flag, kWaitNs)) {
            ok = false;
            break;
          }
          tc::tc_fence_after();
          const uint32_t sa0 = tc::smem_u32(smem + s * Cfg::kStageBytes);
          const uint32_t sb0 = sa0 + kSplit * kABytes;
          constexpr int kPairs = kSplit == 1 ? 1 : 6;
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
#pragma unroll
            for (int q = 0; q < kPairs; ++q) {
              const uint32_t sa = sa0 + (kSplit == 1 ? 0 : pair_a(q)) * kABytes;
              const uint32_t sb = sb0 + (kSplit == 1 ? 0 : pair_b(q)) * Cfg::kBBytes;
              const uint64_t ad = tc::smem_desc_sw128(sa + kk * 2048, 8192, 1024);
              const uint64_t bd = tc::smem_desc_sw128(sb + kk * 2048, 8192, 1024);
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
    // epilogue warps 2..5 -> TMEM lane quadrants 2, 3, 0, 1
    const int g = warp & 3;
    const float eta = args.eta;
    uint32_t ch = 0;
    bool ok = true;
    int it = 0;
    for (int t = blockIdx.x; ok && t < T; t += gridDim.x, ++it) {
      const TileIdx ti = decode(t, mt, nt);
      const int worker = args.slot_worker[ti.slot];
      const int b = it & 1;
      // waits are warp-uniform: a lane that gave up takes its whole warp out
      // before the next .sync.aligned TMEM load
      ok = __all_sync(0xffffffffu, tc::wait_or_abort(&tfull[b], (it >> 1) & 1, abort_flag,
                                                      kWaitNs));
      if (!ok) break;
      tc::tc_fence_after();
      const int row = ti.m_tile * 128 + 32 * g + lane;   // input index k of this thread
      const bool row_ok = row < M;
      const uint32_t tbase = tmem + ((uint32_t)(32 * g) << 16) + (uint32_t)b * Cfg::kAccCols;
      const int64_t wbase = (int64_t)worker * args.ld_param + args.woff + row;
      float* theta = args.theta + wbase;
      float* acc = args.acc + wbase;
      bf16* tb = args.theta_b + wbase;
      const int nch = min(Cfg::kChunks, (N - ti.n_tile * BN + kCF - 1) / kCF);
      for (int c = 0; c < nch; ++c) {
        const int r = ch % kRing;
        uint32_t v[32];
        tc::tmem_ld_32x32b_x32(tbase + (uint32_t)(c * kCF), v);
        if (kSplit == 3) {
          uint32_t v2[32];
          tc::tmem_ld_32x32b_x32(tbase + (uint32_t)(BN + c * kCF), v2);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i)
            v[i] = __float_as_uint(__fadd_rn(__uint_as_float(v[i]), __uint_as_float(v2[i])));
        } else {
          tc::tmem_ld_wait();
        }
        ok = __all_sync(0xffffffffu,
                        tc::wait_or_abort(&cfull[r], (ch / kRing) & 1, abort_flag, kWaitNs));
        if (!ok) break;
        const float* sT = reinterpret_cast<const float*>(smem + Cfg::kRingOff +
                                                         (size_t)r * 2 * kChunkBytes) +
                          32 * g + lane;
        const float* sA = sT + kChunkBytes / 4;
        const int f0 = ti.n_tile * BN + c * kCF;
        const int nf = row_ok ? min(kCF, N - f0) : 0;
#pragma unroll
        for (int i = 0; i < kCF; ++i) {
          if (i < nf) {
            const float gr = __uint_as_float(v[i]);
            const float tn = fmaf(-eta, gr, sT[i * 128]);
            const float an = sA[i * 128] + gr;
            const int64_t p = (int64_t)(f0 + i) * M;
            theta[p] = tn;
            acc[p] = an;
            if (kSplit == 1) {
              tb[p] = __float2bfloat16_rn(tn);
            } else {
              bf16 q0, q1, q2;
              split3(tn, q0, q1, q2);
              tb[p] = q0;
              tb[args.piece_plane + p] = q1;
              tb[2 * args.piece_plane + p] = q2;
            }
          }
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
  tc::tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) atomicExch(args.err, 1);
  if (warp == 1) tc::tmem_dealloc(tmem, Cfg::kTmemCols);
}

template <int BN, int kSplit, int kStages>
Status launch_dw(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& th,
                 const CUtensorMap& ac, const TcArgs& args, int slots, int num_sms,
                 cudaStream_t st) {
  using Cfg = DwCfg<BN, kSplit, kStages>;
  static_assert(Cfg::kSmem <= 232448, "shared memory");
  static_assert(Cfg::kSmem > 232448 / 2, "one CTA per SM (all 512 TMEM columns)");
  static_assert(Cfg::kTmemCols == 512, "TMEM columns");
  auto kern = tc_dw_kernel<BN, kSplit, kStages>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)Cfg::kSmem);
  });
  AGN_TRY_CUDA(attr_err);
  const int64_t tiles = (int64_t)ceil_div(args.M, 128) * ceil_div(args.N, BN) * slots;
  if (tiles <= 0) return Status::Ok();
  if (tiles > INT32_MAX) return Status::Err(AGN_E_UNSUPPORTED, "dW tile count overflows");
  const int grid = (int)std::min<int64_t>(tiles, num_sms);
  kern<<<grid, kThreads, Cfg::kSmem, st>>>(a, b, th, ac, args, slots);
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

}  // namespace

Status tc_backward_dw(const CUtensorMap& h_mn, const CUtensorMap& dz_mn,
                      const CUtensorMap& theta_map, const CUtensorMap& acc_map,
                      const TcArgs& args, int slots, cudaStream_t st, bool split, int num_sms) {
  if (split)
    return launch_dw<kTcDwBNSplit, 3, 1>(h_mn, dz_mn, theta_map, acc_map, args, slots, num_sms,
                                         st);
  return launch_dw<kTcDwBN, 1, 2>(h_mn, dz_mn, theta_map, acc_map, args, slots, num_sms, st);
}

}  // namespace agn
