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
constexpr int kBK = 64;                       // K per stage: 64 bf16 = one 128-byte row
constexpr int kABytes = 128 * 128;            // 128 rows x 128 bytes
constexpr uint64_t kWaitNs = 2000000000ull;   // 2 s

// A stage holds kSplit A pieces then kSplit B pieces (kSplit = 3 in the fp32
// mode, where every fp32 operand is the exact sum of three bf16 pieces).
template <int BN, int kSplit>
struct TileCfg {
  static constexpr int kBBytes = BN * 128;
  static constexpr int kStageBytes = kSplit * (kABytes + kBBytes);
  // split mode keeps two accumulators: columns [0, BN) take the leading
  // piece products a0 b0, columns [BN, 2 BN) the five smaller pairs, so the
  // rounding of the tensor core's running sums is relative to each part
  static constexpr uint32_t kTmemCols = (kSplit == 1 ? 1 : 2) * BN;   // power of two >= 32
};

// Piece pairs (i, j) with i + j <= 2 of the split product: the dropped pairs
// are below 2^-25 |a b|, under the rounding of one fp32 product.
__device__ __constant__ const int kPairA[6] = {0, 0, 1, 0, 1, 2};
__device__ __constant__ const int kPairB[6] = {0, 1, 0, 2, 1, 0};

template <typename T>
__device__ __forceinline__ T to_act(float v);
template <>
__device__ __forceinline__ bf16 to_act<bf16>(float v) { return __float2bfloat16_rn(v); }
template <>
__device__ __forceinline__ float to_act<float>(float v) { return v; }
__device__ __forceinline__ float from_act(bf16 v) { return __bfloat162float(v); }
__device__ __forceinline__ float from_act(float v) { return v; }

// Three exact bf16 pieces of an fp32 output element (slot, offset o within
// the slot), written to the out_pieces planes for the next tensor-core GEMM.
__device__ __forceinline__ void write_pieces(const TcArgs& a, int slot, int64_t o, float v) {
  bf16 q0, q1, q2;
  split3(v, q0, q1, q2);
  bf16* p = a.out_pieces + (int64_t)slot * a.out_bstride + o;
  p[0] = q0;
  p[a.out_plane] = q1;
  p[2 * a.out_plane] = q2;
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
template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages, int kSplit>
__global__ void __launch_bounds__(kThreads, kEpi == kEpiDW ? 2 : 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const TcArgs args) {
  using Cfg = TileCfg<BN, kSplit>;
  using TAct = typename std::conditional<kSplit == 1, bf16, float>::type;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * Cfg::kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* done = empty + kStages;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  // A CTA that gave up earlier in this launch (or run) makes the rest return
  // at once, before they allocate anything.
  __shared__ int s_skip;
  if (threadIdx.x == 0) s_skip = *reinterpret_cast<volatile int*>(args.err);
  __syncthreads();
  if (s_skip != 0) return;   // uniform across the CTA
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tile = blockIdx.x, n_tile = blockIdx.y, slot = blockIdx.z;
  const int worker = args.slot_worker[slot];
  const int KT = (args.K + kBK - 1) / kBK;
  const int a_z = args.a_by_worker ? worker : slot;
  const int b_z = args.b_by_worker ? worker : slot;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], 1);
    }
    tc::mbar_init(done, 1);
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
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    if (lane == 0) {
      int kt = 0;
      for (; kt < KT; ++kt) {
        const int s = kt % kStages;
        if (kt >= kStages && !wait_or_abort(&empty[s], ((kt / kStages) - 1) & 1, abort_flag)) {
          *abort_flag = 1;
          break;
        }
        if (*abort_flag) break;
        uint8_t* sa0 = smem + s * Cfg::kStageBytes;
        uint8_t* sb0 = sa0 + kSplit * kABytes;
        tc::mbar_arrive_expect_tx(&full[s], Cfg::kStageBytes);
        // one box of 3D maps (kSplit = 1) or of 4D maps with the piece index
        auto load = [&](uint8_t* dst, const CUtensorMap* map, int x, int y, int z, int p) {
          if (kSplit == 1) tc::tma_load_3d(dst, map, &full[s], x, y, z);
          else tc::tma_load_4d(dst, map, &full[s], x, y, z, p);
        };
#pragma unroll
        for (int p = 0; p < kSplit; ++p) {
          uint8_t* sa = sa0 + p * kABytes;
          uint8_t* sb = sb0 + p * Cfg::kBBytes;
          if (!kAMN) {
            load(sa, &tmA, kt * kBK, m_tile * 128, a_z, p);
          } else {
            load(sa, &tmA, m_tile * 128, kt * kBK, a_z, p);
            load(sa + 8192, &tmA, m_tile * 128 + 64, kt * kBK, a_z, p);
          }
          if (!kBMN) {
            load(sb, &tmB, kt * kBK, n_tile * BN, b_z, p);
          } else {
#pragma unroll
            for (int c = 0; c < BN / 64; ++c)
              load(sb + c * 8192, &tmB, n_tile * BN + c * 64, kt * kBK, b_z, p);
          }
        }
      }
      if (*abort_flag) {
        // drain: wait (bounded) for the copies of the last stages we armed
        for (int j = kt - 1; j >= 0 && j >= kt - kStages; --j)
          tc::mbar_wait_bounded(&full[j % kStages], (j / kStages) & 1, kWaitNs);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t kIdesc = tc::idesc_bf16_f32(128, BN, kAMN, kBMN);
      for (int kt = 0; kt < KT; ++kt) {
        const int s = kt % kStages;
        if (!wait_or_abort(&full[s], (kt / kStages) & 1, abort_flag)) {
          *abort_flag = 1;
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
            const uint32_t sa = sa0 + (kSplit == 1 ? 0 : kPairA[q]) * kABytes;
            const uint32_t sb = sb0 + (kSplit == 1 ? 0 : kPairB[q]) * Cfg::kBBytes;
            const uint64_t ad = kAMN ? tc::smem_desc_sw128(sa + kk * 2048, 8192, 1024)
                                     : tc::smem_desc_sw128(sa + kk * 32, 16, 1024);
            const uint64_t bd = kBMN ? tc::smem_desc_sw128(sb + kk * 2048, 8192, 1024)
                                     : tc::smem_desc_sw128(sb + kk * 32, 16, 1024);
            const uint32_t dcol = (kSplit == 3 && q > 0) ? (uint32_t)BN : 0u;
            const bool acc_on = kSplit == 1 ? (kt | kk | q) != 0
                                            : (q == 0 ? (kt | kk) != 0 : ((kt | kk) != 0 || q > 1));
            tc::mma_bf16(tmem + dcol, ad, bd, kIdesc, acc_on ? 1u : 0u);
          }
        }
        tc::mma_commit(&empty[s]);
      }
      tc::mma_commit(done);
    }
  }
  __syncwarp();

  const bool ok = wait_or_abort(done, 0, abort_flag) && !*abort_flag;
  tc::tc_fence_after();
  if (!ok) {
    if (threadIdx.x == 0) atomicExch(args.err, 1);
  } else {
    const int g = warp & 3, half = warp >> 2;
    const int row = 128 * m_tile + 32 * g + lane;   // M index of this thread
    const bool row_ok = row < args.M;
    const uint32_t lane_base = (uint32_t)(32 * g) << 16;
    float* theta = args.theta + (int64_t)worker * args.ld_param;
    if (kEpi == kEpiFwd) {
      const float bias = row_ok ? theta[args.boff + row] : 0.f;
      TAct* out = static_cast<TAct*>(args.out) + (int64_t)slot * args.out_bstride;
#pragma unroll 1
      for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
        uint32_t r[32];
        tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)c0, r);
        if (kSplit == 3) {
          uint32_t r2[32];
          tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(BN + c0), r2);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i)
            r[i] = __float_as_uint(__fadd_rn(__uint_as_float(r[i]), __uint_as_float(r2[i])));
        }
        tc::tmem_ld_wait();
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int j = n_tile * BN + c0 + i;
            if (j < args.N) {
              float v = __uint_as_float(r[i]) + bias;
              if (args.relu) v = fmaxf(v, 0.f);
              const int64_t o = (int64_t)j * args.ldo + row;
              out[o] = to_act<TAct>(v);
              if (kSplit == 3 && args.out_pieces) write_pieces(args, slot, o, v);
            }
          }
        }
      }
    } else if (kEpi == kEpiDX) {
      TAct* out = static_cast<TAct*>(args.out) + (int64_t)slot * args.out_bstride;
      const TAct* mask = static_cast<const TAct*>(args.mask) + (int64_t)slot * args.mask_bstride;
#pragma unroll 1
      for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
        uint32_t r[32];
        tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)c0, r);
        if (kSplit == 3) {
          uint32_t r2[32];
          tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(BN + c0), r2);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i)
            r[i] = __float_as_uint(__fadd_rn(__uint_as_float(r[i]), __uint_as_float(r2[i])));
        }
        tc::tmem_ld_wait();
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int j = n_tile * BN + c0 + i;
            if (j < args.N) {
              const int64_t o = (int64_t)j * args.ldo + row;
              const float h = from_act(mask[o]);
              const float v = h > 0.f ? __uint_as_float(r[i]) : 0.f;
              out[o] = to_act<TAct>(v);
              if (kSplit == 3 && args.out_pieces) write_pieces(args, slot, o, v);
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
            thn[i] = __ldcs(th_in + p);
            acn[i] = __ldcs(ac_in + p);
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
            const float t = fmaf(-eta, gr, th[i]);
            theta[p] = t;
            acc[p] = ac[i] + gr;
            if (kSplit == 1) {
              tb[p] = __float2bfloat16_rn(t);
            } else {
              bf16 q0, q1, q2;
              split3(t, q0, q1, q2);
              tb[p] = q0;
              tb[args.piece_plane + p] = q1;
              tb[2 * args.piece_plane + p] = q2;
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
  __shared__ float red[kBiasGroups][32];
  const int fx = threadIdx.x & 31, gy = threadIdx.x >> 5;
  const int f = blockIdx.x * 32 + fx;
  const int z = blockIdx.y;
  const TD* col = dz + (int64_t)z * dz_bstride + f;
  float part = 0.f;
  if (f < d)
    for (int j = gy; j < m; j += kBiasGroups) part += from_act(col[(int64_t)j * d]);
  red[gy][fx] = part;
  __syncthreads();
  if (gy != 0 || f >= d) return;
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < kBiasGroups; ++q) s += red[q][fx];
  const int64_t p = (int64_t)slot_worker[z] * ld_param + boff + f;
  const float t = fmaf(-eta, s, theta[p]);
  theta[p] = t;
  acc[p] += s;
  if (kSplit == 1) {
    theta_b[p] = __float2bfloat16_rn(t);
  } else {
    bf16 q0, q1, q2;
    split3(t, q0, q1, q2);
    theta_b[p] = q0;
    theta_b[piece_plane + p] = q1;
    theta_b[2 * piece_plane + p] = q2;
  }
}

// out[p * plane + i] = piece p of x[i] (x = piece 0 + piece 1 + piece 2 exactly).
__global__ void split_pieces_kernel(const float* __restrict__ x, bf16* __restrict__ out,
                                    int64_t count, int64_t plane) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count; i += stride) {
    bf16 q0, q1, q2;
    split3(x[i], q0, q1, q2);
    out[i] = q0;
    out[plane + i] = q1;
    out[2 * plane + i] = q2;
  }
}

template <int BN, int kSplit, int kStages>
size_t smem_bytes() {
  // Shared memory requested per CTA also caps the CTAs per SM so that their
  // TMEM columns never exceed the 512 an SM has.
  const size_t ring = (size_t)kStages * TileCfg<BN, kSplit>::kStageBytes + 1024 + 256;
  const size_t floor_for_tmem =
      (size_t)(233472 / (512 / TileCfg<BN, kSplit>::kTmemCols + 1)) + 1024;
  return std::max(ring, floor_for_tmem);
}

template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages, int kSplit>
Status launch_tc(const CUtensorMap& a, const CUtensorMap& b, const TcArgs& args, int slots,
                 cudaStream_t st) {
  static_assert(kStages * TileCfg<BN, kSplit>::kStageBytes + 1280 <= 232448, "smem");
  auto kern = tc_gemm_kernel<BN, kAMN, kBMN, kEpi, kStages, kSplit>;
  const size_t smem = smem_bytes<BN, kSplit, kStages>();
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  });
  AGN_TRY_CUDA(attr_err);
  dim3 grid((unsigned)ceil_div(args.M, 128), (unsigned)ceil_div(args.N, BN), (unsigned)slots);
  kern<<<grid, kThreads, smem, st>>>(a, b, args);
  AGN_TRY_CUDA(cudaGetLastError());
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
  return encode(map, 4, base, dims, strides, box);
}

Status make_tmap_f32_3d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                        uint64_t batch, uint64_t row_stride_elems, uint64_t batch_stride_elems,
                        uint32_t box_inner, uint32_t box_rows) {
  cuuint64_t dims[3] = {inner, rows, batch};
  cuuint64_t strides[2] = {row_stride_elems * 4, batch_stride_elems * 4};
  cuuint32_t box[3] = {box_inner, box_rows, 1};
  return encode(map, 3, base, dims, strides, box, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4,
                CU_TENSOR_MAP_SWIZZLE_NONE);
}

Status tc_forward(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args, int slots,
                  cudaStream_t st, bool split, int bn) {
  if (split) {
    if (bn == 64) return launch_tc<64, false, false, kEpiFwd, 3, 3>(w_k, h_k, args, slots, st);
    if (bn == 128) return launch_tc<128, false, false, kEpiFwd, 2, 3>(w_k, h_k, args, slots, st);
    return launch_tc<256, false, false, kEpiFwd, 1, 3>(w_k, h_k, args, slots, st);
  }
  if (bn == 64) return launch_tc<64, false, false, kEpiFwd, 6, 1>(w_k, h_k, args, slots, st);
  if (bn == 128) return launch_tc<128, false, false, kEpiFwd, 5, 1>(w_k, h_k, args, slots, st);
  return launch_tc<256, false, false, kEpiFwd, 4, 1>(w_k, h_k, args, slots, st);
}

Status tc_backward_dx(const CUtensorMap& w_mn, const CUtensorMap& dz_k, const TcArgs& args,
                      int slots, cudaStream_t st, bool split, int bn) {
  if (split) {
    if (bn == 64) return launch_tc<64, true, false, kEpiDX, 3, 3>(w_mn, dz_k, args, slots, st);
    if (bn == 128) return launch_tc<128, true, false, kEpiDX, 2, 3>(w_mn, dz_k, args, slots, st);
    return launch_tc<256, true, false, kEpiDX, 1, 3>(w_mn, dz_k, args, slots, st);
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
    bias_update_kernel<float, 3><<<grid, threads, 0, st>>>(static_cast<const float*>(dz), m, d,
                                                           dz_bstride, slot_worker, theta, acc,
                                                           theta_b, ld_param, boff, eta,
                                                           piece_plane);
  else
    bias_update_kernel<bf16, 1><<<grid, threads, 0, st>>>(static_cast<const bf16*>(dz), m, d,
                                                          dz_bstride, slot_worker, theta, acc,
                                                          theta_b, ld_param, boff, eta,
                                                          piece_plane);
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

Status split_pieces(const float* x, bf16* out, int64_t count, int64_t plane, cudaStream_t st) {
  if (count <= 0) return Status::Ok();
  const int grid = (int)std::min<int64_t>(ceil_div(count, 256), 152 * 8);
  split_pieces_kernel<<<grid, 256, 0, st>>>(x, out, count, plane);
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

}  // namespace agn
