// The bounds-checked build (compiled with -DAGN_BOUNDS_CHECK; build.py's
// `check` variant, libagn_gb300_check.so).  compute-sanitizer cannot be used
// on the GPUs this library is tested on, so this build stands in for its
// memcheck on the hot path: every generic global load, store and L2 add of
// the kernels that AGN_ST / AGN_LD, their cache-hint forms and AGN_RED4 /
// AGN_RED wrap is first checked against the table of device buffers the
// library knows (the handles' allocations and the caller's buffers of a
// standalone commit call).  An access outside every buffer is not performed:
// the kernel records its address and counts it, a load returns zero, and the
// host turns the count into AGN_E_BOUNDS after the call.  Tensor-map (TMA)
// copies are checked on the host when the map is encoded (the whole span of
// the map must lie in one buffer; the copy engine itself stays within the
// map), and bulk copies on the device before they are issued.  In the normal
// build the macros are the plain accesses.
#pragma once

#include <cstdint>

namespace agn {

constexpr int kBoundsMax = 120;   // buffers the table can hold

// [lo, hi) byte ranges of the buffers kernels may touch.
struct BoundsTable {
  int n;
  unsigned long long lo[kBoundsMax], hi[kBoundsMax];
};

#ifdef AGN_BOUNDS_CHECK

// One copy per translation unit (internal linkage); AGN_BOUNDS_UNIT gives
// the host a setter and a reader for the unit's copy.
static __constant__ BoundsTable g_bounds;
static __device__ unsigned long long g_bounds_first;   // first bad address
static __device__ unsigned int g_bounds_count;         // accesses refused

__device__ __forceinline__ bool bounds_ok(const void* p, unsigned int bytes) {
  const unsigned long long a = reinterpret_cast<unsigned long long>(p);
  for (int i = 0; i < g_bounds.n; ++i)
    if (a >= g_bounds.lo[i] && a + bytes <= g_bounds.hi[i]) return true;
  return false;
}
__device__ __forceinline__ void bounds_fail(const void* p) {
  atomicCAS(&g_bounds_first, 0ull, reinterpret_cast<unsigned long long>(p));
  atomicAdd(&g_bounds_count, 1u);
}
template <typename T, typename V>
__device__ __forceinline__ void st_checked(T* p, const V& v) {
  if (bounds_ok(p, sizeof(T))) *p = static_cast<T>(v);
  else bounds_fail(p);
}
template <typename T>
__device__ __forceinline__ T ld_checked(const T* p) {
  if (bounds_ok(p, sizeof(T))) return *p;
  bounds_fail(p);
  return T{};
}
template <typename T>
__device__ __forceinline__ void stcg_checked(T* p, const T& v) {
  if (bounds_ok(p, sizeof(T))) __stcg(p, v);
  else bounds_fail(p);
}
template <typename T>
__device__ __forceinline__ T ldcg_checked(const T* p) {
  if (bounds_ok(p, sizeof(T))) return __ldcg(p);
  bounds_fail(p);
  return T{};
}
template <typename T>
__device__ __forceinline__ void stcs_checked(T* p, const T& v) {
  if (bounds_ok(p, sizeof(T))) __stcs(p, v);
  else bounds_fail(p);
}
template <typename T>
__device__ __forceinline__ T ldcs_checked(const T* p) {
  if (bounds_ok(p, sizeof(T))) return __ldcs(p);
  bounds_fail(p);
  return T{};
}

#define AGN_ST(p, v) ::agn::st_checked((p), (v))
#define AGN_LD(p) ::agn::ld_checked(p)
#define AGN_STCG(p, v) ::agn::stcg_checked((p), (v))
#define AGN_LDCG(p) ::agn::ldcg_checked(p)
#define AGN_LDCS(p) ::agn::ldcs_checked(p)
#define AGN_STCS(p, v) ::agn::stcs_checked((p), (v))
#define AGN_BOUNDS_OK(p, bytes) ::agn::bounds_ok((p), (bytes))
#define AGN_BOUNDS_FAIL(p) ::agn::bounds_fail(p)
// L2 adds (tc_ptx.cuh): four floats or one
#define AGN_RED4(p, v)                                                        \
  do {                                                                        \
    if (::agn::bounds_ok((p), 16)) ::agn::tc::red_add_f32x4((p), (v));        \
    else ::agn::bounds_fail(p);                                               \
  } while (0)
#define AGN_RED(p, v)                                                         \
  do {                                                                        \
    if (::agn::bounds_ok((p), 4)) ::agn::tc::red_add_f32((p), (v));           \
    else ::agn::bounds_fail(p);                                               \
  } while (0)

// Host side of one translation unit's table: bounds_set_<unit> uploads the
// table and clears the unit's record, bounds_get_<unit> reads the record
// (both on `st`, the reader synchronously).
#define AGN_BOUNDS_UNIT(unit)                                                                  \
  cudaError_t bounds_set_##unit(const ::agn::BoundsTable& t, cudaStream_t st) {                 \
    const unsigned long long z = 0;                                                            \
    const unsigned int zc = 0;                                                                 \
    cudaError_t e = cudaMemcpyToSymbolAsync(::agn::g_bounds, &t, sizeof(t), 0,                 \
                                            cudaMemcpyHostToDevice, st);                       \
    if (e == cudaSuccess)                                                                      \
      e = cudaMemcpyToSymbolAsync(::agn::g_bounds_first, &z, sizeof(z), 0,                     \
                                  cudaMemcpyHostToDevice, st);                                 \
    if (e == cudaSuccess)                                                                      \
      e = cudaMemcpyToSymbolAsync(::agn::g_bounds_count, &zc, sizeof(zc), 0,                    \
                                  cudaMemcpyHostToDevice, st);                                 \
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);                                       \
    return e;                                                                                  \
  }                                                                                            \
  cudaError_t bounds_get_##unit(unsigned long long* first, unsigned int* count,                 \
                                cudaStream_t st) {                                             \
    cudaError_t e = cudaStreamSynchronize(st);                                                 \
    if (e == cudaSuccess) e = cudaMemcpyFromSymbol(first, ::agn::g_bounds_first, sizeof(*first)); \
    if (e == cudaSuccess) e = cudaMemcpyFromSymbol(count, ::agn::g_bounds_count, sizeof(*count)); \
    return e;                                                                                  \
  }

#else

#define AGN_ST(p, v) (void)(*(p) = (v))
#define AGN_LD(p) (*(p))
#define AGN_STCG(p, v) __stcg((p), (v))
#define AGN_LDCG(p) __ldcg(p)
#define AGN_LDCS(p) __ldcs(p)
#define AGN_STCS(p, v) __stcs((p), (v))
#define AGN_BOUNDS_OK(p, bytes) true
#define AGN_BOUNDS_FAIL(p) ((void)0)
#define AGN_RED4(p, v) ::agn::tc::red_add_f32x4((p), (v))
#define AGN_RED(p, v) ::agn::tc::red_add_f32((p), (v))
#define AGN_BOUNDS_UNIT(unit)

#endif

}  // namespace agn
