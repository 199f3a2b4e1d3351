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

#include "mlp.cuh"
#include "mlp_tc.cuh"
#include "tc_ptx.cuh"

namespace agn {

namespace {

constexpr int kThreads = 256;
constexpr int kBK = 64;                       // K per stage: 64 bf16 = one 128-byte row
constexpr int kABytes = 128 * 128;            // 128 rows x 128 bytes
constexpr uint64_t kWaitNs = 2000000000ull;   // 2 s

template <int BN>
struct TileCfg {
  static constexpr int kBBytes = BN * 128;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kTmemCols = BN;   // power of two >= 32
};

// Wait that also gives up when another role has aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity,
                                              volatile int* abort_flag) {
  if (tc::mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = tc::globaltimer_ns();
  for (uint32_t it = 0;; ++it) {
    if (tc::mbar_try_wait(bar, parity)) return true;
    if ((it & 63) == 63) {
      if (*abort_flag) return false;
      if (tc::globaltimer_ns() - t0 > kWaitNs) return false;
    }
  }
}

// The dW kernel is bound by its epilogue's DRAM traffic: two CTAs per SM
// (registers capped at 128) keep more loads in flight.
template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages>
__global__ void __launch_bounds__(kThreads, kEpi == kEpiDW ? 2 : 1)
tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const TcArgs args) {
  using Cfg = TileCfg<BN>;
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
        uint8_t* sa = smem + s * Cfg::kStageBytes;
        uint8_t* sb = sa + kABytes;
        tc::mbar_arrive_expect_tx(&full[s], Cfg::kStageBytes);
        if (!kAMN) {
          tc::tma_load_3d(sa, &tmA, &full[s], kt * kBK, m_tile * 128, a_z);
        } else {
          tc::tma_load_3d(sa, &tmA, &full[s], m_tile * 128, kt * kBK, a_z);
          tc::tma_load_3d(sa + 8192, &tmA, &full[s], m_tile * 128 + 64, kt * kBK, a_z);
        }
        if (!kBMN) {
          tc::tma_load_3d(sb, &tmB, &full[s], kt * kBK, n_tile * BN, b_z);
        } else {
#pragma unroll
          for (int c = 0; c < BN / 64; ++c)
            tc::tma_load_3d(sb + c * 8192, &tmB, &full[s], n_tile * BN + c * 64, kt * kBK, b_z);
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
        const uint32_t sa = tc::smem_u32(smem + s * Cfg::kStageBytes);
        const uint32_t sb = sa + kABytes;
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
          const uint64_t ad = kAMN ? tc::smem_desc_sw128(sa + kk * 2048, 8192, 1024)
                                   : tc::smem_desc_sw128(sa + kk * 32, 16, 1024);
          const uint64_t bd = kBMN ? tc::smem_desc_sw128(sb + kk * 2048, 8192, 1024)
                                   : tc::smem_desc_sw128(sb + kk * 32, 16, 1024);
          tc::mma_bf16(tmem, ad, bd, kIdesc, (kt | kk) != 0 ? 1u : 0u);
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
      bf16* out = static_cast<bf16*>(args.out) + (int64_t)slot * args.out_bstride;
#pragma unroll 1
      for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
        uint32_t r[32];
        tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)c0, r);
        tc::tmem_ld_wait();
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int j = n_tile * BN + c0 + i;
            if (j < args.N) {
              float v = __uint_as_float(r[i]) + bias;
              if (args.relu) v = fmaxf(v, 0.f);
              out[(int64_t)j * args.ldo + row] = __float2bfloat16_rn(v);
            }
          }
        }
      }
    } else if (kEpi == kEpiDX) {
      bf16* out = static_cast<bf16*>(args.out) + (int64_t)slot * args.out_bstride;
      const bf16* mask = args.mask + (int64_t)slot * args.mask_bstride;
#pragma unroll 1
      for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
        uint32_t r[32];
        tc::tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)c0, r);
        tc::tmem_ld_wait();
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int j = n_tile * BN + c0 + i;
            if (j < args.N) {
              const int64_t o = (int64_t)j * args.ldo + row;
              const float h = __bfloat162float(mask[o]);
              out[o] = __float2bfloat16_rn(h > 0.f ? __uint_as_float(r[i]) : 0.f);
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
        tc::tmem_ld_32x32b_x16(tmem + lane_base + (uint32_t)(half * (BN / 2) + ch * kCh), r);
        if (ch + 1 < kChunks) load_chunk(ch + 1);
        tc::tmem_ld_wait();
        const int nvalid = row_ok ? min(kCh, args.N - (cbase + ch * kCh)) : 0;
#pragma unroll
        for (int i = 0; i < kCh; ++i) {
          if (i < nvalid) {
            const int64_t p = pbase + (int64_t)(ch * kCh + i) * args.M;
            const float gr = __uint_as_float(r[i]);
            const float t = fmaf(-eta, gr, th[i]);
            theta[p] = t;
            acc[p] = ac[i] + gr;
            tb[p] = __float2bfloat16_rn(t);
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
// b -= eta g_b, a_b += g_b, bf16 copy.  One thread per (f, slot).
__global__ void bias_update_kernel(const bf16* __restrict__ dz, int m, int d, int64_t dz_bstride,
                                   const int* __restrict__ slot_worker, float* theta, float* acc,
                                   bf16* theta_b, int64_t ld_param, int64_t boff, float eta) {
  const int f = blockIdx.x * blockDim.x + threadIdx.x;
  const int z = blockIdx.y;
  if (f >= d) return;
  const bf16* col = dz + (int64_t)z * dz_bstride + f;
  float s = 0.f;
  for (int j = 0; j < m; ++j) s += __bfloat162float(col[(int64_t)j * d]);
  const int64_t p = (int64_t)slot_worker[z] * ld_param + boff + f;
  const float t = fmaf(-eta, s, theta[p]);
  theta[p] = t;
  acc[p] += s;
  theta_b[p] = __float2bfloat16_rn(t);
}

template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages>
size_t smem_bytes() {
  // Shared memory requested per CTA also caps the CTAs per SM so that their
  // TMEM columns never exceed the 512 an SM has.
  const size_t ring = (size_t)kStages * TileCfg<BN>::kStageBytes + 1024 + 256;
  const size_t floor_for_tmem = (size_t)(233472 / (512 / TileCfg<BN>::kTmemCols + 1)) + 1024;
  return std::max(ring, floor_for_tmem);
}

template <int BN, bool kAMN, bool kBMN, int kEpi, int kStages>
Status launch_tc(const CUtensorMap& a, const CUtensorMap& b, const TcArgs& args, int slots,
                 cudaStream_t st) {
  auto kern = tc_gemm_kernel<BN, kAMN, kBMN, kEpi, kStages>;
  const size_t smem = smem_bytes<BN, kAMN, kBMN, kEpi, kStages>();
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
  AGN_TRY(tc_init());
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (row_stride_elems * 2) % 16 ||
      (batch_stride_elems * 2) % 16 || (inner * 2) % 16)
    return Status::Err(AGN_E_UNSUPPORTED, "tensor map operand not 16-byte aligned");
  cuuint64_t dims[3] = {inner, rows, batch};
  cuuint64_t strides[2] = {row_stride_elems * 2, batch_stride_elems * 2};
  cuuint32_t box[3] = {box_inner, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return Status::Err(AGN_E_CUDA, "cuTensorMapEncodeTiled failed with code " + std::to_string(r));
  return Status::Ok();
}

Status tc_forward(const CUtensorMap& w_k, const CUtensorMap& h_k, const TcArgs& args, int slots,
                  cudaStream_t st) {
  switch (args.N <= 64 ? 64 : args.N <= 128 ? 128 : 256) {
    case 64: return launch_tc<64, false, false, kEpiFwd, 6>(w_k, h_k, args, slots, st);
    case 128: return launch_tc<128, false, false, kEpiFwd, 5>(w_k, h_k, args, slots, st);
    default: return launch_tc<256, false, false, kEpiFwd, 4>(w_k, h_k, args, slots, st);
  }
}

Status tc_backward_dx(const CUtensorMap& w_mn, const CUtensorMap& dz_k, const TcArgs& args,
                      int slots, cudaStream_t st) {
  switch (args.N <= 64 ? 64 : args.N <= 128 ? 128 : 256) {
    case 64: return launch_tc<64, true, false, kEpiDX, 6>(w_mn, dz_k, args, slots, st);
    case 128: return launch_tc<128, true, false, kEpiDX, 5>(w_mn, dz_k, args, slots, st);
    default: return launch_tc<256, true, false, kEpiDX, 4>(w_mn, dz_k, args, slots, st);
  }
}

Status tc_backward_dw(const CUtensorMap& h_mn, const CUtensorMap& dz_mn, const TcArgs& args,
                      int slots, cudaStream_t st) {
  return launch_tc<256, true, true, kEpiDW, 2>(h_mn, dz_mn, args, slots, st);
}

Status bias_update(const bf16* dz, int m, int d, int64_t dz_bstride, const int* slot_worker,
                   float* theta, float* acc, bf16* theta_b, int64_t ld_param, int64_t boff,
                   float eta, int slots, cudaStream_t st) {
  dim3 grid((unsigned)ceil_div(d, 128), (unsigned)slots);
  bias_update_kernel<<<grid, 128, 0, st>>>(dz, m, d, dz_bstride, slot_worker, theta, acc, theta_b,
                                           ld_param, boff, eta);
  AGN_TRY_CUDA(cudaGetLastError());
  return Status::Ok();
}

}  // namespace agn
