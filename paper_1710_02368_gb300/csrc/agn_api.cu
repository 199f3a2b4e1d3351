// C ABI of the AGN library: handle life cycle, the host scheduler that turns
// a (worker, staleness) schedule into waves of batched local steps and runs of
// fused commits, and the standalone commit+pull entry point.
//
// Scheduling (Fig. 1's FIFO parameter server, Algorithm 1's workers): commit c
// of worker w_c is computed from theta~ after v_c = c - tau_c commits, and is
// a pure function of that version and the worker's data cursor.  So the host
// groups the commits whose version is already available into a wave, runs
// their lambda local steps as one batched launch sequence, then applies every
// computed commit in FIFO order (one fused commit+pull launch per run of at
// most kMaxCommitsPerLaunch commits); each pull happens right after the commit
// that creates the version it reads.  This gives the same theta~ as applying
// the commits one at a time in schedule order.
#include <chrono>
#include <cstdlib>
#include <mutex>
#include <cmath>
#include <cstdint>
#include <new>
#include <cstring>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "host_inputs.h"
#include "mlp.cuh"
#include "mlp_tc.cuh"

using agn::bf16;
using agn::CommitPlan;
using agn::Status;
using agn::ceil_div;
using agn::round_up;

namespace {

thread_local std::string g_error;   // message of the last handle-less failure

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

// NVTX range for the duration of a scope (a no-op without a tool attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};

struct Wave {
  int offset = 0;                 // first slot in the run's plan arrays
  int slots = 0;
  std::vector<CommitPlan> commits;
};

}  // namespace

#ifdef AGN_BOUNDS_CHECK
namespace agn {
// Each kernel translation unit's copy of the table (AGN_BOUNDS_UNIT).
#define AGN_BOUNDS_DECL(unit)                                                           \
  cudaError_t bounds_set_##unit(const BoundsTable& t, cudaStream_t st);                  \
  cudaError_t bounds_get_##unit(unsigned long long* first, unsigned int* count, cudaStream_t st);
AGN_BOUNDS_DECL(commit)
AGN_BOUNDS_DECL(eval)
AGN_BOUNDS_DECL(head)
AGN_BOUNDS_DECL(simt)
AGN_BOUNDS_DECL(tc)
AGN_BOUNDS_DECL(dw)
AGN_BOUNDS_DECL(optim)
#undef AGN_BOUNDS_DECL

namespace {
std::mutex g_bounds_mu;
std::vector<std::pair<unsigned long long, unsigned long long>> g_bounds_ranges;
}  // namespace

void bounds_add(const void* p, size_t bytes) {
  if (!p || bytes == 0) return;
  // self-test of the checker (tests/bounds_cases.py, case detect): every
  // buffer registered this many bytes short of its end, so that accesses near
  // the end, inside the real allocation, are refused
  static const long long shrink =
      std::getenv("AGN_BOUNDS_TEST_SHRINK") ? std::atoll(std::getenv("AGN_BOUNDS_TEST_SHRINK")) : 0;
  if (shrink > 0) bytes = bytes > (size_t)shrink ? bytes - (size_t)shrink : 0;
  std::lock_guard<std::mutex> lock(g_bounds_mu);
  const unsigned long long a = reinterpret_cast<unsigned long long>(p);
  g_bounds_ranges.push_back({a, a + bytes});
}

void bounds_remove(const void* p) {
  std::lock_guard<std::mutex> lock(g_bounds_mu);
  const unsigned long long a = reinterpret_cast<unsigned long long>(p);
  for (size_t i = 0; i < g_bounds_ranges.size(); ++i)
    if (g_bounds_ranges[i].first == a) {
      g_bounds_ranges.erase(g_bounds_ranges.begin() + (std::ptrdiff_t)i);
      return;
    }
}

bool bounds_host_ok(const void* p, size_t bytes) {
  std::lock_guard<std::mutex> lock(g_bounds_mu);
  const unsigned long long a = reinterpret_cast<unsigned long long>(p);
  for (const auto& r : g_bounds_ranges)
    if (a >= r.first && a + bytes <= r.second) return true;
  return false;
}

Status bounds_upload(cudaStream_t st) {
  BoundsTable t{};
  {
    std::lock_guard<std::mutex> lock(g_bounds_mu);
    if ((int)g_bounds_ranges.size() > kBoundsMax)
      return Status::Err(AGN_E_UNSUPPORTED, "bounds-checked build: more than " +
                                                std::to_string(kBoundsMax) + " live buffers");
    t.n = (int)g_bounds_ranges.size();
    for (int i = 0; i < t.n; ++i) {
      t.lo[i] = g_bounds_ranges[i].first;
      t.hi[i] = g_bounds_ranges[i].second;
    }
  }
  using SetFn = cudaError_t (*)(const BoundsTable&, cudaStream_t);
  for (SetFn f : {bounds_set_commit, bounds_set_eval, bounds_set_head, bounds_set_simt,
                  bounds_set_tc, bounds_set_dw, bounds_set_optim})
    AGN_TRY_CUDA(f(t, st));
  return Status::Ok();
}

Status bounds_collect(cudaStream_t st) {
  using GetFn = cudaError_t (*)(unsigned long long*, unsigned int*, cudaStream_t);
  unsigned long long first = 0;
  unsigned long long total = 0;
  for (GetFn f : {bounds_get_commit, bounds_get_eval, bounds_get_head, bounds_get_simt,
                  bounds_get_tc, bounds_get_dw, bounds_get_optim}) {
    unsigned long long a = 0;
    unsigned int c = 0;
    AGN_TRY_CUDA(f(&a, &c, st));
    total += c;
    if (!first) first = a;
  }
  if (total == 0) return Status::Ok();
  char buf[32];
  std::snprintf(buf, sizeof(buf), "%llx", first);
  return Status::Err(AGN_E_BOUNDS, "bounds-checked build: " + std::to_string(total) +
                                       " kernel accesses outside every known device buffer "
                                       "were refused, the first at 0x" + buf);
}
}  // namespace agn
#endif

struct agn_handle {
  // problem
  std::vector<int> dims;
  int L = 0, n = 0, lam = 0;
  double eta = 0.0;
  uint64_t seed = 0;
  int prec = AGN_PREC_FP32, m = 32, dist = AGN_DIST_UNIFORM, normalize = 1, gemm = 0;
  int commit_rule = AGN_COMMIT_AGN;
  // accumulator elided: `acc` holds each worker's theta at its last pull and
  // a commit adds (theta_k - theta_pull) scaled by 1/lambda (or 1/(tau+1), 1)
  bool elide = false;
  // Adam as the local optimizer: raw gradients go to grad, the moments m, v
  // persist per worker, the accumulator (if kept) sums the steps
  bool adam = false;
  float beta1 = 0.9f, beta2 = 0.999f, eps = 1e-8f;
  float* grad = nullptr;      // [n][P_pad]
  float* mom1 = nullptr;      // [n][P_pad]
  float* mom2 = nullptr;      // [n][P_pad]
  // held-out evaluation set (rows [N, N + n_eval) of the generator) and the
  // buffers of its forward pass, chunk rows at a time
  int64_t n_eval = 0, eval_chunk = 0;
  float* Xe = nullptr;        // [n_eval][d0] fp32
  int* ye = nullptr;          // [n_eval]
  float* He[2] = {nullptr, nullptr};   // [eval_chunk][max hidden d]
  float* Ze = nullptr;        // [eval_chunk][d_L]
  float* e_loss = nullptr;    // [n_eval]
  int* e_correct = nullptr;   // [n_eval]
  int* e_pred = nullptr;      // [n_eval]
  float* e_out = nullptr;     // [2]: mean loss, accuracy
  int* e_sw = nullptr;        // [1] = {0}
  int tau_lo = 0, tau_hi = 0;
  int64_t N = 0, S = 0;
  std::vector<int> tdims;
  int64_t P = 0, P_pad = 0;
  std::vector<int64_t> woff, boff, woff_flat, boff_flat;   // per layer (index l-1)
  int maxd = 0;
  // CUDA
  int device = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  cudaEvent_t ev0 = nullptr, ev1 = nullptr;
  std::vector<void*> allocs;
  // device state
  float* theta_c = nullptr;   // [P_pad]
  float* rep = nullptr;       // [n][P_pad] fp32 master replicas
  float* acc = nullptr;       // [n][P_pad] accumulators (sum of raw gradients)
  bf16* rep_b = nullptr;      // [n][P_pad] bf16 working copies (bf16 mode)
  void* X = nullptr;          // [N][d0] T
  int* y = nullptr;           // [N]
  void* Xb = nullptr;         // [n][m][d0] T
  int* yb = nullptr;          // [n][m]
  std::vector<void*> H;       // H[l] [n][m][d_l] T, l = 1..L-1 (H[0] = Xb)
  float* Z = nullptr;         // [n][m][d_L]
  std::vector<void*> dZ;      // dZ[l] [n][m][d_l] T, l = 1..L
  int* flag = nullptr;        // [0] non-finite loss or commit, [1] bounded wait gave up
  double* partials = nullptr;
  // tcgen05 path (bf16 mode): tensor maps per layer l = 1..L-1 (index l-1)
  bool use_tc = false;
  int tc_mask = 7;            // bit 0 forward, bit 1 dX, bit 2 dW, 3 tiled dW, 4 no split K,
                              // 5 output layer as its own kernel
  struct LayerMaps {
    CUtensorMap w_k, w_mn, h_k, h_mn, dz_k, dz_mn;
    CUtensorMap theta, acc;      // fp32 W_l of every replica / accumulator, box {128, 32}
    CUtensorMap h_mn32, dz_mn32; // split mode: 32-sample boxes for the dW kernel
  };
  int num_sms = 148;
  // maps of the output layer's dW when it runs in the tensor-core dW launch
  // (theta, acc, h_mn / h_mn32 over H_{L-1}, dz_mn / dz_mn32 over dZ_L)
  float* tc_part = nullptr;     // split-K partial sums: [SMs][BN <= 256][128]
  int* tc_counter = nullptr;    // split-K arrival counts per output tile: [2][SMs]
  int ctr_parity = 0;           // which half the next split-K launch counts in
  std::vector<LayerMaps> tmaps;
  LayerMaps out_maps;
  LayerMaps l1_alt;               // layer 1's maps over the alternate operand buffer
  // fp32 mode on the tensor cores: every operand is three exact bf16 pieces
  bool split = false;
  int64_t piece_plane = 0;        // 0: no replica keeps weight pieces (fp32 mode splits in the GEMMs)
  std::vector<bf16*> Hs;          // pieces of H_l, l = 0..L-2: [3][n][m][d_l]
  std::vector<bf16*> dZp;         // pieces of dZ_l, l = 1..L-1: [3][n][m][d_l]
  // output layer fused into one kernel (forward + softmax-CE + dX) when narrow
  bool use_head = false;
  // the output layer's dW runs as tiles of the persistent tensor-core dW
  // launch: dZ_L padded to ldz_out columns (zero beyond d_L) with its pieces,
  // and H_{L-1}'s pieces kept
  bool fuse_out_dw = false;
  int ldz_out = 0;
  float* ce_partial = nullptr;    // [n][ceil(m / kHeadSamples)]
  int* head_counter = nullptr;    // [n]
  // the output layer fused into the last hidden layer's tensor-core forward
  // (when the launch's CTAs fit the SMs at once): partial logits, counters
  bool fuse_head = false;
  float* fh_part = nullptr;       // [n][ceil(m / 32)][ceil(d_{L-1} / 128)][32][16]
  int* fh_counter = nullptr;      // [2][n][ceil(m / 32)]
  int fh_parity = 0;
  // loss_parts holds loss_q values per local step of a commit: the fused
  // output layer writes one per 32-sample chunk, the other paths the step's
  // loss in the first and zeros after it
  int loss_q = 1;
  // the gather copies a local step's minibatch before waiting for the
  // preceding kernel: the layer-1 operand the tensor-core kernels read
  // alternates between two buffers by local step (gparity)
  bool early_gather = false;
  int gparity = 0;
  // padded shards: layer 1's tensor-core operand and the labels read in
  // place, worker w's shard stored as S + m rows (row r = dataset row
  // w S + r mod S), so a local step's minibatch is m consecutive rows and
  // no gather runs; yb is then the padded labels [n][S + m]
  bool direct_x = false;
  void* Xpad = nullptr;           // bf16 mode: [n][S + m][d0]
  bf16* Hs0_pad = nullptr;        // fp32 mode: pieces [3][n][S + m][d0]
  long long* zero_t0 = nullptr;   // [n] zeros (the fill's step counters)
  void* Xb_alt = nullptr;         // bf16 mode: [n][m][d0]
  bf16* Hs0_alt = nullptr;        // fp32 mode: pieces [3][n][m][d0]
  // test hook of the bounded waits (agn_debug_waits)
  uint64_t dbg_wait_ns = 0;
  int dbg_withhold = 0;
  int grid = 0;
  float* loss = nullptr;      // [cap_commits]
  float* dnorm = nullptr;     // [cap_commits]
  int64_t cap_commits = 0;
  float* loss_parts = nullptr;
  int64_t cap_parts = 0;
  int* plan_worker = nullptr;
  int* plan_commit = nullptr;
  long long* plan_t0 = nullptr;
  int64_t cap_plan = 0;
  int* pull_list = nullptr;   // [n]
  // host state
  std::vector<float> hX, htheta0;
  std::vector<int32_t> hy;
  int64_t V = 0;                                  // commits applied
  std::vector<int64_t> prev, pulled_v, steps;     // per worker
  std::string err;
  double stats[5] = {0, 0, 0, 0, 0};
  // per-kernel profiling (agn_profile)
  bool prof = false;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  struct Pending {
    int cls;
    size_t e0;
    double flops, bytes;
  };
  std::vector<Pending> pend;
  double kstats[AGN_KERNEL_CLASSES][4] = {};
};

namespace {

int fail(agn_handle* h, const Status& s) {
  if (h) h->err = s.msg; else g_error = s.msg;
  return s.code;
}
int fail(agn_handle* h, int code, const std::string& msg) { return fail(h, Status::Err(code, msg)); }

Status dalloc(agn_handle* h, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) bytes = 16;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return Status::Err(AGN_E_OOM, "cudaMalloc of " + std::to_string(bytes) + " bytes failed: " +
                                      cudaGetErrorString(e));
  }
  h->allocs.push_back(*p);
  agn::bounds_add(*p, bytes);
  return Status::Ok();
}

void dfree(agn_handle* h, void* p) {
  if (!p) return;
  for (auto& a : h->allocs)
    if (a == p) a = nullptr;
  agn::bounds_remove(p);
  cudaFree(p);
}

template <typename Tp>
Status dalloc_t(agn_handle* h, Tp** p, size_t count) {
  void* v = nullptr;
  AGN_TRY(dalloc(h, &v, count * sizeof(Tp)));
  *p = static_cast<Tp*>(v);
  return Status::Ok();
}

// Grow a device array (keeps the first `keep` elements).
template <typename Tp>
Status grow(agn_handle* h, Tp** p, int64_t* cap, int64_t need, int64_t keep) {
  if (need <= *cap) return Status::Ok();
  int64_t nc = std::max<int64_t>(need, *cap * 2);
  Tp* np = nullptr;
  AGN_TRY(dalloc_t(h, &np, (size_t)nc));
  if (*p && keep > 0)
    AGN_TRY_CUDA(cudaMemcpyAsync(np, *p, (size_t)keep * sizeof(Tp), cudaMemcpyDeviceToDevice,
                                 h->stream));
  AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
  dfree(h, *p);
  *p = np;
  *cap = nc;
  return Status::Ok();
}

size_t elem_size(const agn_handle* h) { return h->prec == AGN_PREC_BF16 ? 2 : 4; }

// CUDA events around one launch when profiling is on; always counts it.
class Launch {
 public:
  Launch(agn_handle* h, int cls, double flops, double bytes, int64_t* counter)
      : h_(h), cls_(cls), flops_(flops), bytes_(bytes) {
    ++*counter;
    if (h_->prof) {
      e0_ = next();
      if (e0_ != kNone) cudaEventRecord(h_->ev_pool[e0_], h_->stream);
    }
  }
  ~Launch() {
    if (h_->prof && e0_ != kNone) {
      size_t e1 = next();
      if (e1 == kNone) return;
      cudaEventRecord(h_->ev_pool[e1], h_->stream);
      h_->pend.push_back({cls_, e0_, flops_, bytes_});
    }
  }

 private:
  static constexpr size_t kNone = ~size_t(0);
  size_t next() {
    if (h_->ev_used == h_->ev_pool.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return kNone;
      h_->ev_pool.push_back(e);
    }
    return h_->ev_used++;
  }
  agn_handle* h_;
  int cls_;
  double flops_, bytes_;
  size_t e0_ = kNone;
};

// After the stream has drained: fold the recorded event pairs into kstats.
void collect_profile(agn_handle* h) {
  for (const auto& p : h->pend) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, h->ev_pool[p.e0], h->ev_pool[p.e0 + 1]) == cudaSuccess) {
      h->kstats[p.cls][0] += 1;
      h->kstats[p.cls][1] += ms;
      h->kstats[p.cls][2] += p.flops;
      h->kstats[p.cls][3] += p.bytes;
    }
  }
  h->pend.clear();
  h->ev_used = 0;
}

// Layer l (1-based) runs on the tensor cores: bf16 mode, a hidden layer.
bool tc_layer(const agn_handle* h, int l) { return h->use_tc && l < h->L; }

agn::TcArgs tc_args(agn_handle* h, const int* sw, const long long* st0, int step) {
  agn::TcArgs t{};
  t.slot_worker = sw;
  t.slot_t0 = st0;
  t.step = step;
  t.x_shard = h->direct_x ? h->S : 0;
  t.ksplit = 1;
  t.part = h->tc_part;
  t.counter = nullptr;            // set per forward / dX launch (next_counters)
  t.err = h->flag + 1;
  t.theta = h->rep;
  t.acc = h->elide ? nullptr : h->acc;
  t.grad_out = h->adam ? h->grad : nullptr;
  t.theta_b = h->rep_b;
  t.ld_param = h->P_pad;
  t.piece_plane = h->piece_plane;
  t.wait_ns = h->dbg_wait_ns;
  t.withhold_rank = h->dbg_withhold;
  t.one_row_tile = (h->tc_mask & 128) ? 1 : 0;
  t.acc_ring = (h->tc_mask & 256) ? 1 : 0;
  return t;
}

// The split-K arrival counters of the next forward / dX launch: one half of
// tc_counter, the other half (the previous launch's) cleared by its CTA 0.
void next_counters(agn_handle* h, agn::TcArgs* t) {
  t->counter = h->tc_counter + h->ctr_parity * h->num_sms;
  t->counter_clear = h->tc_counter + (1 - h->ctr_parity) * h->num_sms;
  t->counter_clear_n = h->num_sms;
  h->ctr_parity ^= 1;
}

// Tensor maps of the tcgen05 path (addresses are fixed for the handle's life).
Status build_tc_maps(agn_handle* h) {
  const int n = h->n, m = h->m, L = h->L;
  const uint32_t bn = (uint32_t)agn::tc_bn(m);
  h->tmaps.assign(L - 1, {});
  for (int l = 1; l < L; ++l) {
    const uint64_t fi = h->dims[l - 1], fo = h->dims[l];
    auto& mp = h->tmaps[l - 1];
    AGN_TRY(agn::make_tmap_f32_3d(&mp.theta, h->rep + h->woff[l - 1], fi, fo, n, fi, h->P_pad,
                                  128, 32));
    AGN_TRY(agn::make_tmap_f32_3d(&mp.acc, h->acc + h->woff[l - 1], fi, fo, n, fi, h->P_pad,
                                  128, 32));
    if (h->split) {
      // the fp32 weights themselves (the GEMMs split them into pieces in
      // shared memory): a kTcSplitBK-deep k step of 128 features (forward,
      // K-major) or 128 inputs of kTcSplitBK features (dX); activations as 4D
      // piece maps, kTcSplitBK-deep k steps for the forward and dX
      constexpr uint32_t bk = agn::kTcSplitBK;
      const float* W = h->rep + h->woff[l - 1];
      // (with column tiles up to 128 the forward's converters read the tile
      // row by row into tensor memory: 128-byte swizzle, conflict-free)
      AGN_TRY(agn::make_tmap_f32_3d(&mp.w_k, W, fi, fo, n, fi, h->P_pad, bk, 128, bn <= 128));
      AGN_TRY(agn::make_tmap_f32_3d(&mp.w_mn, W, fi, fo, n, fi, h->P_pad, 128, bk));
      const bf16* Hp = h->Hs[l - 1];
      const uint64_t hp = (uint64_t)n * m * fi;
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_k, Hp, fi, m, n, fi, (uint64_t)m * fi, hp, bk, bn));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn, Hp, fi, m, n, fi, (uint64_t)m * fi, hp, 64, 64));
      const uint64_t dp = (uint64_t)n * m * fo;
      const bf16* dZp = h->dZp[l];
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.dz_k, dZp, fo, m, n, fo, (uint64_t)m * fo, dp, bk, bn));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.dz_mn, dZp, fo, m, n, fo, (uint64_t)m * fo, dp, 64, 64));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn32, Hp, fi, m, n, fi, (uint64_t)m * fi, hp, 64, 32));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.dz_mn32, dZp, fo, m, n, fo, (uint64_t)m * fo, dp, 64, 32));
      continue;
    }
    const bf16* W = h->rep_b + h->woff[l - 1];
    AGN_TRY(agn::make_tmap_bf16_3d(&mp.w_k, W, fi, fo, n, fi, h->P_pad, 64, 128));
    AGN_TRY(agn::make_tmap_bf16_3d(&mp.w_mn, W, fi, fo, n, fi, h->P_pad, 64, 64));
    const void* Hin = l == 1 ? h->Xb : h->H[l - 1];
    AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_k, Hin, fi, m, n, fi, (uint64_t)m * fi, 64, bn));
    AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_mn, Hin, fi, m, n, fi, (uint64_t)m * fi, 64, 64));
    const void* dZ = h->dZ[l];
    AGN_TRY(agn::make_tmap_bf16_3d(&mp.dz_k, dZ, fo, m, n, fo, (uint64_t)m * fo, 64, bn));
    AGN_TRY(agn::make_tmap_bf16_3d(&mp.dz_mn, dZ, fo, m, n, fo, (uint64_t)m * fo, 64, 64));
  }
  if (h->direct_x) {   // layer 1's operand maps over the padded shards
    const uint64_t fi = h->dims[0], rows = (uint64_t)(h->S + m);
    auto& mp = h->tmaps[0];
    if (h->split) {
      const uint64_t hp = (uint64_t)n * rows * fi;
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_k, h->Hs0_pad, fi, rows, n, fi, rows * fi, hp,
                                     agn::kTcSplitBK, bn));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn, h->Hs0_pad, fi, rows, n, fi, rows * fi, hp, 64,
                                     64));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn32, h->Hs0_pad, fi, rows, n, fi, rows * fi, hp, 64,
                                     32));
    } else {
      AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_k, h->Xpad, fi, rows, n, fi, rows * fi, 64, bn));
      AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_mn, h->Xpad, fi, rows, n, fi, rows * fi, 64, 64));
    }
  }
  if (h->early_gather) {   // layer 1's operand maps over the alternate buffer
    const uint64_t fi = h->dims[0];
    h->l1_alt = h->tmaps[0];
    auto& mp = h->l1_alt;
    if (h->split) {
      const uint64_t hp = (uint64_t)n * m * fi;
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_k, h->Hs0_alt, fi, m, n, fi, (uint64_t)m * fi, hp,
                                     agn::kTcSplitBK, bn));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn, h->Hs0_alt, fi, m, n, fi, (uint64_t)m * fi, hp, 64,
                                     64));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn32, h->Hs0_alt, fi, m, n, fi, (uint64_t)m * fi, hp,
                                     64, 32));
    } else {
      AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_k, h->Xb_alt, fi, m, n, fi, (uint64_t)m * fi, 64, bn));
      AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_mn, h->Xb_alt, fi, m, n, fi, (uint64_t)m * fi, 64, 64));
    }
  }
  if (h->fuse_out_dw) {   // the output layer's dW tiles: M = d_{L-1} inputs, N = d_L
    const uint64_t fi = h->dims[L - 1], fo = h->dims[L], lz = (uint64_t)h->ldz_out;
    auto& mp = h->out_maps;
    AGN_TRY(agn::make_tmap_f32_3d(&mp.theta, h->rep + h->woff[L - 1], fi, fo, n, fi, h->P_pad,
                                  128, 32));
    AGN_TRY(agn::make_tmap_f32_3d(&mp.acc, h->acc + h->woff[L - 1], fi, fo, n, fi, h->P_pad,
                                  128, 32));
    if (h->split) {
      const bf16* Hp = h->Hs[L - 1];
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.h_mn32, Hp, fi, m, n, fi, (uint64_t)m * fi,
                                     (uint64_t)n * m * fi, 64, 32));
      AGN_TRY(agn::make_tmap_bf16_4d(&mp.dz_mn32, h->dZp[L], lz, m, n, lz, (uint64_t)m * lz,
                                     (uint64_t)n * m * lz, 64, 32));
    } else {
      AGN_TRY(agn::make_tmap_bf16_3d(&mp.h_mn, h->H[L - 1], fi, m, n, fi, (uint64_t)m * fi, 64, 64));
      AGN_TRY(agn::make_tmap_bf16_3d(&mp.dz_mn, h->dZ[L], lz, m, n, lz, (uint64_t)m * lz, 64, 64));
    }
  }
  return Status::Ok();
}

// Split K of a forward or dX GEMM with M rows, N = m columns and K inner
// over s slots: one CTA per output tile, unless the tiles leave SMs idle
// (small waves); then ks CTAs share each tile, with ks <= SMs / tiles and
// every CTA's range of 64-deep k steps non-empty.
int pick_ksplit(const agn_handle* h, int M, int K, int s) {
  if (h->tc_mask & 16) return 1;
  const int64_t tiles = ceil_div(M, 128) * ceil_div(h->m, agn::tc_bn(h->m)) * (int64_t)s;
  if (tiles >= h->num_sms) return 1;
  const int kt = (int)ceil_div(K, 64);
  int ks = (int)std::min<int64_t>(kt, h->num_sms / tiles);
  if (ks <= 1) return 1;
  const int per = (int)ceil_div(kt, ks);
  return (int)ceil_div(kt, per);
}

// Pieces of an fp32 activation buffer [slots][m][d] (planes `plane` apart,
// default n m d) for the tensor-core GEMMs of the fp32 mode.
Status split_act(agn_handle* h, const void* src, bf16* dst, int d, int slots, int64_t* launches,
                 int64_t plane = -1) {
  const int64_t count = (int64_t)slots * h->m * d;
  const int64_t pl = plane >= 0 ? plane : (int64_t)h->n * h->m * d;
  Launch k(h, AGN_K_OTHER, 0.0, (double)count * 10.0, launches);
  return agn::split_pieces(static_cast<const float*>(src), dst, count, pl, h->stream);
}

// ---------------------------------------------------------------------------
// One wave: lambda local steps of every slot (Algorithm 1's inner loop)
// ---------------------------------------------------------------------------

template <typename T>
Status run_wave_steps(agn_handle* h, const Wave& wv, int64_t* launches) {
  const int s = wv.slots;
  const int* sw = h->plan_worker + wv.offset;
  const int* sc = h->plan_commit + wv.offset;
  const long long* st0 = h->plan_t0 + wv.offset;
  const int m = h->m, L = h->L, n = h->n;
  const T* W = h->prec == AGN_PREC_BF16 ? reinterpret_cast<const T*>(h->rep_b)
                                         : reinterpret_cast<const T*>(h->rep);
  const float eta = (float)h->eta;
  const double es = (double)sizeof(T);
  // bytes per parameter of the local step + accumulation: theta RMW, a RMW, and
  // the low-precision copy (one bf16, or three pieces in the split mode)
  // (with Adam the dW kernels only store the gradient, 4 bytes; the Adam
  // kernel's own traffic is counted at its launch)
  const double upd = h->adam ? 4.0
                             : (h->elide ? 8.0 : 16.0) + (h->prec == AGN_PREC_BF16 ? 2.0 : 0.0);
  // pieces of dZ_l (split mode, hidden tensor-core layers), planes n m d_l apart
  auto dz_pieces = [&](int l) -> bf16* {
    return (h->split && l >= 1 && tc_layer(h, l)) ? h->dZp[l] : nullptr;
  };
  auto dz_plane = [&](int l) -> int64_t { return (int64_t)n * m * h->dims[l]; };
  for (int i = 0; i < h->lam; ++i) {
    // this local step's buffer of layer 1's tensor-core operand
    const bool alt = h->early_gather && h->gparity;
    const agn_handle::LayerMaps& l1 = alt ? h->l1_alt : h->tmaps.empty() ? h->l1_alt : h->tmaps[0];
    auto maps_of = [&](int l) -> const agn_handle::LayerMaps& { return l == 1 ? l1 : h->tmaps[l - 1]; };
    if (!h->direct_x) {
      // fp32 mode with the early gather: the fp32 rows are not read by the
      // tensor-core kernels, only their pieces
      T* xb = h->early_gather ? (h->split ? nullptr : static_cast<T*>(alt ? h->Xb_alt : h->Xb))
                              : static_cast<T*>(h->Xb);
      Launch k(h, AGN_K_GATHER, 0.0,
               (double)s * m * ((xb ? 2.0 : 1.0) * h->dims[0] * es + 8.0 +
                                (h->split ? 6.0 * h->dims[0] : 0.0)),
               launches);
      AGN_TRY(agn::gather_batch<T>(static_cast<const T*>(h->X), h->y, xb, h->yb, h->dims[0], m,
                                   h->S, sw, st0, i, s, h->stream,
                                   h->split ? (alt ? h->Hs0_alt : h->Hs[0]) : nullptr,
                                   (int64_t)n * m * h->dims[0], h->early_gather ? 1 : 0));
    }
    if (h->early_gather) h->gparity ^= 1;
    bool dz_ready = false;   // pieces of the next layer's dZ already written by its producer
    // the output layer rides in the last hidden layer's forward when that
    // launch's CTAs fit the SMs at once
    const bool fuse_head_now =
        h->fuse_head && tc_layer(h, L - 1) &&
        ceil_div(h->dims[L - 1], 128) * (int64_t)s <= (int64_t)h->num_sms;
    bool head_done = false;
    // forward, l = 1..L
    for (int l = 1; l <= L; ++l) {
      if (l == L && head_done) continue;
      if (l == L && h->use_head) {   // output layer: forward + softmax-CE + dX, one kernel
        agn::HeadArgs a{};
        const int fi = h->dims[L - 1], C = h->dims[L];
        a.H = L == 1 ? h->Xb : h->H[L - 1];
        a.W = W; a.theta = h->rep; a.ld_param = h->P_pad;
        a.woff = h->woff[L - 1]; a.boff = h->boff[L - 1];
        a.K = fi; a.C = C; a.m = m;
        a.slot_worker = sw; a.yb = h->yb;
        a.slot_t0 = st0; a.x_shard = h->direct_x ? h->S : 0;
        a.dZL = h->dZ[L]; a.ldz = h->ldz_out;
        a.dZL_pieces = (h->fuse_out_dw && h->split) ? h->dZp[L] : nullptr;
        a.dZL_plane = (int64_t)n * m * h->ldz_out;
        a.dH = L > 1 ? h->dZ[L - 1] : nullptr;
        a.dH_pieces = L > 1 ? dz_pieces(L - 1) : nullptr;
        a.dH_plane = L > 1 ? dz_plane(L - 1) : 0;
        a.ce_partial = h->ce_partial; a.counter = h->head_counter;
        a.loss_parts = h->loss_parts; a.loss_q = h->loss_q; a.slot_commit = sc; a.lam = h->lam; a.step = i;
        a.flag = h->flag;
        Launch k(h, AGN_K_SOFTMAX, 4.0 * s * m * fi * C,
                 (double)s * ((double)C * fi * es + 2.0 * m * fi * es + (double)m * C * es), launches);
        AGN_TRY(agn::head_forward_backward<T>(a, s, h->stream));
        dz_ready = a.dH_pieces != nullptr;
        continue;
      }
      agn::GemmArgs g{};
      const int fi = h->dims[l - 1], fo = h->dims[l];
      g.M = m; g.N = fo; g.K = fi;
      g.a = l == 1 ? h->Xb : h->H[l - 1]; g.lda = fi; g.a_bstride = (int64_t)m * fi;
      g.b = W + h->woff[l - 1]; g.ldb = fi; g.b_bstride = h->P_pad; g.b_by_worker = 1;
      g.slot_worker = sw;
      g.out = l == L ? static_cast<void*>(h->Z) : h->H[l];
      g.ldo = fo; g.out_bstride = (int64_t)m * fo;
      g.relu = l < L;
      g.theta = h->rep; g.ld_param = h->P_pad; g.boff = h->boff[l - 1];
      const double oes = l == L ? 4.0 : es;
      // pieces of a hidden activation that the next tensor-core GEMMs read
      // (the forward of layer l + 1 and the dW of layer l + 1)
      bf16* h_pieces =
          (h->split && (l + 1 < L || (h->fuse_out_dw && l + 1 == L))) ? h->Hs[l] : nullptr;
      bool pieces_done = false;
      const bool fuse = fuse_head_now && l == L - 1;
      {
        // with the output layer fused: its forward and dX flops, W_L, dZ_L
        // and dZ_{L-1} (with pieces) bytes too
        const int C = h->dims[L];
        Launch k(h, fuse ? AGN_K_FORWARD_HEAD : AGN_K_FORWARD,
                 2.0 * s * m * fo * fi + (fuse ? 4.0 * s * m * fo * C : 0.0),
                 (double)s * ((double)fo * fi * es + 4.0 * fo + (double)m * fi * es +
                              (double)m * fo * (oes + (h_pieces ? 6.0 : 0.0))) +
                     (fuse ? (double)s * (4.0 * C * (fo + 1) +
                                          (double)m * C * (es + (h->split ? 6.0 : 0.0)) +
                                          (double)m * fo * (2.0 * es + (h->split ? 6.0 : 0.0)))
                           : 0.0),
                 launches);
        if (fuse) {
          agn::TcArgs t = tc_args(h, sw, st0, i);
          t.M = fo; t.N = m; t.K = fi;
          t.a_by_worker = 1;
          t.out = h->H[l]; t.ldo = fo; t.out_bstride = (int64_t)m * fo;
          t.relu = 1; t.boff = h->boff[l - 1];
          t.out_pieces = h_pieces; t.out_plane = (int64_t)n * m * fo;
          t.head_woff = h->woff[L - 1]; t.head_boff = h->boff[L - 1]; t.head_C = C;
          t.yb = h->yb;
          t.dzl = h->dZ[L]; t.ldz = h->ldz_out;
          t.dzl_pieces = (h->fuse_out_dw && h->split) ? h->dZp[L] : nullptr;
          t.dzl_plane = (int64_t)n * m * h->ldz_out;
          t.dh = h->dZ[L - 1]; t.dh_pieces = dz_pieces(L - 1); t.dh_plane = dz_plane(L - 1);
          t.head_part = h->fh_part;
          {   // the fused output layer's counters alternate like the split-K ones
            const int hn = n * (int)ceil_div(m, 32);
            t.head_counter = h->fh_counter + h->fh_parity * hn;
            t.head_counter_clear = h->fh_counter + (1 - h->fh_parity) * hn;
            t.head_counter_clear_n = hn;
            h->fh_parity ^= 1;
          }
          t.loss_parts = h->loss_parts; t.slot_commit = sc; t.lam = h->lam; t.step = i;
          t.nonfinite = h->flag;
          const auto& mp = maps_of(l);
          t.x_b_direct = l == 1;
          t.no_a_prefetch = l == 1 && (h->tc_mask & 512) ? 1 : 0;
          t.ksplit = pick_ksplit(h, fo, fi, s);
          next_counters(h, &t);
          bool launched = false;
          AGN_TRY(agn::tc_forward_head(mp.w_k, mp.h_k, t, s, h->stream, h->split,
                                       agn::tc_bn(m), h->num_sms, &launched));
          if (!launched) return Status::Err(AGN_E_CUDA, "internal: fused output layer not resident");
          pieces_done = true;
          head_done = true;
          dz_ready = t.dh_pieces != nullptr;
        } else if (tc_layer(h, l) && (h->tc_mask & 1)) {
          agn::TcArgs t = tc_args(h, sw, st0, i);
          t.M = fo; t.N = m; t.K = fi;
          t.a_by_worker = 1;
          t.out = h->H[l]; t.ldo = fo; t.out_bstride = (int64_t)m * fo;
          t.relu = 1; t.boff = h->boff[l - 1];
          t.out_pieces = h_pieces; t.out_plane = (int64_t)n * m * fo;
          const auto& mp = maps_of(l);
          t.x_b_direct = l == 1;
          t.no_a_prefetch = l == 1 && (h->tc_mask & 512) ? 1 : 0;
          t.ksplit = pick_ksplit(h, fo, fi, s);
          next_counters(h, &t);
          AGN_TRY(agn::tc_forward(mp.w_k, mp.h_k, t, s, h->stream, h->split, agn::tc_bn(m)));
          pieces_done = true;
        } else {
          AGN_TRY(agn::simt_forward<T>(g, l == L, s, h->stream));
        }
      }
      if (h_pieces && !pieces_done) AGN_TRY(split_act(h, h->H[l], h_pieces, fo, s, launches));
    }
    if (!h->use_head) {
      Launch k(h, AGN_K_SOFTMAX, 0.0, (double)s * m * (h->dims[L] * (4.0 + es) + 4.0), launches);
      AGN_TRY(agn::softmax_xent<T>(h->Z, h->yb, static_cast<T*>(h->dZ[L]), m, h->dims[L],
                                   h->loss_parts, sc, h->lam, i, h->flag, s, h->stream));
    }
    // backward: dX for l = L..2 (each reads W_l before its update), then the
    // weight and bias gradients with the local step of every layer
    std::vector<char> have_pieces(L + 1, 0);   // pieces of dZ_l written by its producer
    if (L > 1) have_pieces[L - 1] = dz_ready;
    auto ensure_pieces = [&](int l) -> Status {
      if (dz_pieces(l) && !have_pieces[l]) {
        AGN_TRY(split_act(h, h->dZ[l], dz_pieces(l), h->dims[l], s, launches, dz_plane(l)));
        have_pieces[l] = 1;
      }
      return Status::Ok();
    };
    for (int l = L; l >= 2; --l) {
      if (l == L && h->use_head) continue;   // the head already wrote dZ_{L-1}
      const int fi = h->dims[l - 1], fo = h->dims[l];
      const void* Hprev = h->H[l - 1];
      bf16* next_pieces = dz_pieces(l - 1);
      Launch k(h, AGN_K_BACKWARD_DX, 2.0 * s * m * fo * fi,
               (double)s * ((double)fo * fi * es + (double)m * fo * es +
                            (double)m * fi * (2.0 * es + (next_pieces ? 6.0 : 0.0))),
               launches);
      if (tc_layer(h, l) && (h->tc_mask & 2)) {
        AGN_TRY(ensure_pieces(l));
        agn::TcArgs t = tc_args(h, sw, st0, i);
        t.M = fi; t.N = m; t.K = fo;
        t.a_by_worker = 1;
        t.out = h->dZ[l - 1]; t.ldo = fi; t.out_bstride = (int64_t)m * fi;
        t.mask = Hprev; t.mask_bstride = (int64_t)m * fi;
        t.out_pieces = next_pieces; t.out_plane = dz_plane(l - 1);
        const auto& mp = h->tmaps[l - 1];
        t.ksplit = pick_ksplit(h, fi, fo, s);
        next_counters(h, &t);
        AGN_TRY(agn::tc_backward_dx(mp.w_mn, mp.dz_k, t, s, h->stream, h->split,
                                    agn::tc_bn(m)));
        have_pieces[l - 1] = next_pieces != nullptr;
      } else {
        agn::GemmArgs g{};
        g.M = m; g.N = fi; g.K = fo;
        g.a = h->dZ[l]; g.lda = fo; g.a_bstride = (int64_t)m * fo;
        g.b = W + h->woff[l - 1]; g.ldb = fi; g.b_bstride = h->P_pad; g.b_by_worker = 1;
        g.slot_worker = sw;
        g.out = h->dZ[l - 1]; g.ldo = fi; g.out_bstride = (int64_t)m * fi;
        g.mask = Hprev; g.mask_bstride = (int64_t)m * fi;
        g.theta = h->rep; g.ld_param = h->P_pad;
        AGN_TRY(agn::simt_backward_dx<T>(g, s, h->stream));
      }
    }
    // dW: the output layer, then the hidden layers (on the tensor cores, all
    // in one persistent launch)
    std::vector<agn::DwLayerMaps> tc_dw;
    double tc_flops = 0.0, tc_bytes = 0.0;
    for (int l = L; l >= 1; --l) {
      const int fi = h->dims[l - 1], fo = h->dims[l];
      const void* Hprev = l == 1 ? h->Xb : h->H[l - 1];
      const double flops = 2.0 * s * m * fo * fi;
      const double bytes =
          (double)s * (((double)fo * fi + fo) * upd + (double)m * fo * es + (double)m * fi * es);
      if (tc_layer(h, l) && (h->tc_mask & 4)) {
        AGN_TRY(ensure_pieces(l));
        if (h->tc_mask & 8) {   // the earlier one-tile-per-CTA kernel, layer by layer
          Launch k(h, AGN_K_BACKWARD_DW, flops, bytes, launches);
          agn::TcArgs t = tc_args(h, sw, st0, i);
          t.M = fi; t.N = fo; t.K = m;
          t.woff = h->woff[l - 1]; t.eta = eta;
          const auto& mp = h->tmaps[l - 1];
          AGN_TRY(agn::tc_backward_dw_tiled(mp.h_mn, mp.dz_mn, t, s, h->stream, h->split));
          AGN_TRY(agn::bias_update(h->dZ[l], m, fo, (int64_t)m * fo, sw, h->rep, h->acc,
                                   h->rep_b, h->P_pad, h->boff[l - 1], eta, s, h->stream,
                                   h->split, h->piece_plane));
        } else {
          const auto& mp = maps_of(l);
          tc_dw.push_back({h->split ? &mp.h_mn32 : &mp.h_mn, h->split ? &mp.dz_mn32 : &mp.dz_mn,
                           &mp.theta, &mp.acc, fi, fo, h->woff[l - 1], h->boff[l - 1],
                           l == 1 ? 1 : 0});
          tc_flops += flops;
          tc_bytes += bytes;
        }
        continue;
      }
      if (l == L && h->fuse_out_dw) {   // as tiles of the tensor-core dW launch
        const auto& mp = h->out_maps;
        tc_dw.insert(tc_dw.begin(), {h->split ? &mp.h_mn32 : &mp.h_mn,
                                     h->split ? &mp.dz_mn32 : &mp.dz_mn, &mp.theta, &mp.acc, fi,
                                     fo, h->woff[l - 1], h->boff[l - 1]});
        tc_flops += flops;
        tc_bytes += bytes;
        continue;
      }
      Launch k(h, AGN_K_BACKWARD_DW, flops, bytes, launches);
      if (l == L && h->use_head) {   // narrow output layer
        agn::HeadDwArgs d{};
        d.H = Hprev; d.dZL = h->dZ[l]; d.slot_worker = sw;
        d.theta = h->rep; d.acc = h->elide ? nullptr : h->acc; d.theta_b = h->rep_b;
        d.piece_plane = h->piece_plane;
        d.ld_param = h->P_pad; d.woff = h->woff[l - 1]; d.boff = h->boff[l - 1];
        d.K = fi; d.C = fo; d.m = m; d.eta = eta;
        d.grad_out = h->adam ? h->grad : nullptr;
        d.dz_early = L > 2 ? 1 : 0;   // a dX launch ran between the head and this one
        AGN_TRY(agn::head_backward_dw<T>(d, s, h->stream));
      } else {
        agn::GemmArgs g{};
        g.M = fo; g.N = fi; g.K = m;
        g.a = h->dZ[l]; g.lda = fo; g.a_bstride = (int64_t)m * fo;
        g.b = Hprev; g.ldb = fi; g.b_bstride = (int64_t)m * fi;
        g.slot_worker = sw;
        g.theta = h->rep; g.acc = h->elide ? nullptr : h->acc; g.theta_bf16 = h->rep_b;
        g.ld_param = h->P_pad;
        g.piece_plane = h->piece_plane;
        g.woff = h->woff[l - 1]; g.boff = h->boff[l - 1]; g.eta = eta;
        g.grad_out = h->adam ? h->grad : nullptr;
        AGN_TRY(agn::simt_backward_dw<T>(g, s, h->stream));
      }
    }
    if (!tc_dw.empty()) {
      Launch k(h, AGN_K_BACKWARD_DW, tc_flops, tc_bytes, launches);
      agn::TcArgs t = tc_args(h, sw, st0, i);
      t.K = m; t.eta = eta;
      AGN_TRY(agn::tc_backward_dw(tc_dw.data(), (int)tc_dw.size(), t, s, h->stream, h->split,
                                  h->num_sms));
    }
    if (h->adam) {   // the local step: Adam on the gradients the dW kernels stored
      agn::AdamArgs ad{};
      ad.grad = h->grad; ad.theta = h->rep; ad.acc = h->elide ? nullptr : h->acc;
      ad.m = h->mom1; ad.v = h->mom2; ad.theta_b = h->rep_b; ad.piece_plane = h->piece_plane;
      ad.P = h->P_pad; ad.ld = h->P_pad;
      ad.slot_worker = sw; ad.slot_t0 = st0; ad.step = i;
      ad.eta = eta; ad.beta1 = h->beta1; ad.beta2 = h->beta2; ad.eps = h->eps;
      const double copy_b = h->rep_b ? 2.0 : 0.0;
      Launch k(h, AGN_K_BACKWARD_DW, 0.0,
               (double)s * h->P * (4.0 + 16.0 + 8.0 + (h->elide ? 0.0 : 8.0) + copy_b), launches);
      AGN_TRY(agn::adam_step(ad, s, h->num_sms, h->stream));
    }
  }
  return Status::Ok();
}

// ---------------------------------------------------------------------------
// Planning
// ---------------------------------------------------------------------------

struct RunPlan {
  std::vector<int> start_pulls;
  std::vector<Wave> waves;
  std::vector<int> slot_worker, slot_commit;
  std::vector<long long> slot_t0;
  std::vector<int64_t> prev, pulled_v, steps;
};

Status build_plan(const agn_handle* h, int k, const int32_t* worker, const int32_t* tau, int ns,
                  RunPlan* out) {
  const int n = h->n;
  const int64_t V0 = h->V;
  std::vector<int64_t> prev = h->prev;
  std::vector<int64_t> v(ns);
  for (int i = 0; i < ns; ++i) {
    const int64_t c = V0 + i;
    const int w = worker[i];
    if (w < 0 || w >= n)
      return Status::Err(AGN_E_SCHEDULE, "commit " + std::to_string(c) + ": worker " +
                                             std::to_string(w) + " out of range");
    if (tau[i] < 0)
      return Status::Err(AGN_E_SCHEDULE, "commit " + std::to_string(c) + ": negative staleness");
    v[i] = c - tau[i];
    if (v[i] <= prev[w])
      return Status::Err(AGN_E_SCHEDULE,
                         "commit " + std::to_string(c) + ": worker " + std::to_string(w) +
                             " cannot read version " + std::to_string(v[i]) +
                             " (its previous commit is " + std::to_string(prev[w]) + ")");
    prev[w] = c;
  }
  // per-worker commits of this run and first look-ahead commit
  std::vector<std::vector<int>> q(n);
  std::vector<int> look(n, -1);
  for (int i = 0; i < ns; ++i) {
    const int w = worker[i];
    if (i < k) q[w].push_back(i);
    else if (look[w] < 0) look[w] = i;
  }
  std::vector<std::vector<int>> pulls_at(k + 1);   // pulls at version V0 + j
  std::vector<int64_t> pulled = h->pulled_v;
  for (int w = 0; w < n; ++w) {
    std::vector<int> lst = q[w];
    if (look[w] >= 0) lst.push_back(look[w]);
    for (size_t e = 0; e < lst.size(); ++e) {
      const int i = lst[e];
      const int64_t vc = v[i];
      if (e == 0) {
        if (vc < V0) {
          if (pulled[w] != vc)
            return Status::Err(AGN_E_SCHEDULE,
                               "commit " + std::to_string(V0 + i) + ": worker " +
                                   std::to_string(w) + " reads version " + std::to_string(vc) +
                                   ", which has passed without a pull (give the earlier call a "
                                   "longer look-ahead)");
          continue;
        }
        if (vc == V0) {
          if (pulled[w] != V0) pulls_at[0].push_back(w);
          pulled[w] = V0;
          continue;
        }
      }
      if (vc <= V0 + k) {
        pulls_at[vc - V0].push_back(w);
        pulled[w] = vc;
      }
    }
    if (!q[w].empty()) {
      // after its last commit of the run, the replica holds the pulled
      // look-ahead version if there is one, else nothing usable
      const int i_look = look[w];
      pulled[w] = (i_look >= 0 && v[i_look] <= V0 + k) ? v[i_look] : -1;
    }
  }
  out->start_pulls = pulls_at[0];
  // waves
  std::vector<int64_t> steps = h->steps;
  std::vector<char> computed(k, 0);
  std::vector<size_t> ptr(n, 0);
  int64_t Vc = V0;
  while (Vc < V0 + k) {
    Wave wv;
    wv.offset = (int)out->slot_worker.size();
    for (int w = 0; w < n; ++w) {
      if (ptr[w] < q[w].size()) {
        const int i = q[w][ptr[w]];
        if (v[i] <= Vc) {
          out->slot_worker.push_back(w);
          out->slot_commit.push_back(i);
          out->slot_t0.push_back(steps[w]);
          steps[w] += h->lam;
          ++ptr[w];
          computed[i] = 1;
        }
      }
    }
    wv.slots = (int)out->slot_worker.size() - wv.offset;
    if (wv.slots == 0) return Status::Err(AGN_E_SCHEDULE, "internal: empty wave");
    int j = (int)(Vc - V0);
    const int j0 = j;
    while (j < k && computed[j]) ++j;
    CommitPlan cp{};
    for (int i = j0; i < j; ++i) {
      const int np = (int)pulls_at[i + 1].size();
      if (cp.n_commits == agn::kMaxCommitsPerLaunch ||
          cp.pull_begin[cp.n_commits] + np > agn::kMaxPullsPerLaunch) {
        wv.commits.push_back(cp);
        cp = CommitPlan{};
      }
      const int c = cp.n_commits;
      cp.worker[c] = worker[i];
      cp.norm_slot[c] = (int)(V0 + i);
      if (h->commit_rule == AGN_COMMIT_DYNSGD) {   // Delta = -eta a / (tau_c + 1)
        cp.per_commit_scale = 1;
        cp.scale[c] = (h->elide || h->adam) ? (float)(1.0 / (double)(tau[i] + 1))
                                            : (float)(-(h->eta / (double)(tau[i] + 1)));
      }
      int pb = cp.pull_begin[c];
      // a run of pulls longer than one launch carries cannot arise while
      // n <= kMaxPullsPerLaunch (each worker pulls a version at most once)
      if (pb + np > agn::kMaxPullsPerLaunch)
        return Status::Err(AGN_E_INVALID, "internal: more pulls at one version than workers");
      for (int p : pulls_at[i + 1]) cp.pull_worker[pb++] = p;
      cp.pull_begin[c + 1] = pb;
      cp.n_commits = c + 1;
    }
    if (cp.n_commits > 0) wv.commits.push_back(cp);
    out->waves.push_back(std::move(wv));
    Vc = V0 + j;
  }
  out->prev = std::move(prev);
  // prev must only advance over the commits actually run
  for (int w = 0; w < n; ++w) out->prev[w] = h->prev[w];
  for (int i = 0; i < k; ++i) out->prev[worker[i]] = V0 + i;
  out->pulled_v = std::move(pulled);
  out->steps = std::move(steps);
  return Status::Ok();
}

Status do_run(agn_handle* h, int k, const int32_t* worker, const int32_t* tau, int ns) {
  const auto t_host0 = std::chrono::steady_clock::now();
  NvtxRange run_range("agn_run");
  RunPlan plan;
  {
    NvtxRange r("plan waves");
    AGN_TRY(build_plan(h, k, worker, tau, ns, &plan));
  }
  const int64_t V0 = h->V;
  const int64_t total_slots = (int64_t)plan.slot_worker.size();
  if (V0 + k > h->cap_commits) {   // loss and dnorm share one capacity
    int64_t c1 = h->cap_commits, c2 = h->cap_commits;
    AGN_TRY(grow(h, &h->loss, &c1, V0 + k, V0));
    AGN_TRY(grow(h, &h->dnorm, &c2, V0 + k, V0));
    h->cap_commits = c1;
  }
  AGN_TRY(grow(h, &h->loss_parts, &h->cap_parts, (int64_t)k * h->lam * h->loss_q, 0));
  if (total_slots > h->cap_plan) {  // the three plan arrays share one capacity
    int64_t c1 = h->cap_plan, c2 = h->cap_plan, c3 = h->cap_plan;
    AGN_TRY(grow(h, &h->plan_worker, &c1, total_slots, 0));
    AGN_TRY(grow(h, &h->plan_commit, &c2, total_slots, 0));
    AGN_TRY(grow(h, &h->plan_t0, &c3, total_slots, 0));
    h->cap_plan = c1;
  }
  AGN_TRY(agn::bounds_upload(h->stream));   // bounds-checked build: buffers as grown
  if (total_slots > 0) {
    AGN_TRY_CUDA(cudaMemcpyAsync(h->plan_worker, plan.slot_worker.data(), total_slots * sizeof(int),
                                 cudaMemcpyHostToDevice, h->stream));
    AGN_TRY_CUDA(cudaMemcpyAsync(h->plan_commit, plan.slot_commit.data(), total_slots * sizeof(int),
                                 cudaMemcpyHostToDevice, h->stream));
    AGN_TRY_CUDA(cudaMemcpyAsync(h->plan_t0, plan.slot_t0.data(), total_slots * sizeof(long long),
                                 cudaMemcpyHostToDevice, h->stream));
  }
  int64_t launches = 0;
  AGN_TRY_CUDA(cudaEventRecord(h->ev0, h->stream));
  if (!plan.start_pulls.empty()) {
    AGN_TRY_CUDA(cudaMemcpyAsync(h->pull_list, plan.start_pulls.data(),
                                 plan.start_pulls.size() * sizeof(int), cudaMemcpyHostToDevice,
                                 h->stream));
    Launch k(h, AGN_K_OTHER, 0.0,
             (double)h->P * (4.0 + plan.start_pulls.size() * (h->rep_b ? 6.0 : 4.0)), &launches);
    AGN_TRY(agn::pull_replicas(h->theta_c, h->rep, h->rep_b, h->P_pad, h->P_pad, h->pull_list,
                               (int)plan.start_pulls.size(), h->stream, h->piece_plane,
                               h->elide ? h->acc : nullptr));
  }
  // commit scale: of the raw gradient sum a (-eta / lambda, or -eta without
  // normalisation), or, with the accumulator elided, of theta_k - theta_pull
  // (which already carries -eta): 1 / lambda, or 1
  const bool steps = h->elide || h->adam;   // the committed quantity already carries -eta
  const float scale = steps ? (float)(h->normalize ? 1.0 / (double)h->lam : 1.0)
                            : (float)(h->normalize ? -(h->eta / (double)h->lam) : -h->eta);
  for (const Wave& wv : plan.waves) {
    NvtxRange wave_range("wave");
    {
      NvtxRange r("local steps");
      if (h->prec == AGN_PREC_BF16) AGN_TRY(run_wave_steps<bf16>(h, wv, &launches));
      else AGN_TRY(run_wave_steps<float>(h, wv, &launches));
    }
    NvtxRange commit_range("commit + pull");
    for (const CommitPlan& cp : wv.commits) {
      const double pulls = cp.pull_begin[cp.n_commits];
      {
        const double copy_b = h->rep_b ? 2.0 : 0.0;
        Launch kc(h, AGN_K_COMMIT, 2.0 * cp.n_commits * h->P,
                  (double)h->P * (8.0 + 8.0 * cp.n_commits +
                                  pulls * (4.0 + copy_b + (h->elide ? 4.0 : 0.0))),
                  &launches);
        AGN_TRY(agn::launch_commit_pull(cp, h->theta_c, h->acc, h->rep, h->rep_b, h->P_pad,
                                        h->P_pad, scale, true, h->partials, h->grid, nullptr,
                                        nullptr, h->stream, /*norms=*/false, h->piece_plane,
                                        h->elide));
      }
      Launch kn(h, AGN_K_NORMS, 0.0, 8.0 * cp.n_commits * h->grid, &launches);
      AGN_TRY(agn::launch_commit_norms(cp, h->partials, h->grid, h->dnorm, h->flag, h->stream));
    }
  }
  {
    Launch kl(h, AGN_K_OTHER, 0.0, 4.0 * k * (h->lam + 1), &launches);
    AGN_TRY(agn::reduce_losses(h->loss_parts, h->lam, h->loss_q, k, h->loss + V0, h->stream));
  }
  AGN_TRY_CUDA(cudaEventRecord(h->ev1, h->stream));
  int flags[2] = {0, 0};
  AGN_TRY_CUDA(cudaMemcpyAsync(flags, h->flag, 2 * sizeof(int), cudaMemcpyDeviceToHost, h->stream));
  const double host_ms =
      std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t_host0).count();
  AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
  const Status bounds = agn::bounds_collect(h->stream);   // bounds-checked build only
  float ms = 0.f;
  cudaEventElapsedTime(&ms, h->ev0, h->ev1);
  if (h->prof) collect_profile(h);
  h->stats[0] = (double)plan.waves.size();
  h->stats[1] = (double)launches;
  h->stats[2] = ms;
  h->stats[3] = (double)k * h->lam;
  h->stats[4] = host_ms;
  h->V = V0 + k;
  h->prev = plan.prev;
  h->pulled_v = plan.pulled_v;
  h->steps = plan.steps;
  if (flags[0] || flags[1]) {
    AGN_TRY_CUDA(cudaMemsetAsync(h->flag, 0, 2 * sizeof(int), h->stream));
    if (flags[1] && h->tc_counter)   // CTAs that gave up may have left tiles unfinished
      AGN_TRY_CUDA(cudaMemsetAsync(h->tc_counter, 0, (size_t)(2 * h->num_sms) * sizeof(int),
                                   h->stream));
    if (flags[1] && h->fuse_head) {
      AGN_TRY_CUDA(cudaMemsetAsync(h->fh_counter, 0,
                                   (size_t)(2 * h->n * ceil_div(h->m, 32)) * sizeof(int),
                                   h->stream));
    }
    AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
    if (!bounds.ok()) return bounds;
    if (flags[1])
      return Status::Err(AGN_E_TIMEOUT, "a tensor-core GEMM gave up on a bounded wait");
    return Status::Err(AGN_E_NONFINITE, "a loss or a commit was not finite");
  }
  return bounds;
}

Status create(agn_handle* h, const int32_t* dims, int32_t n_dims, int32_t n_workers, int32_t lambda,
              double eta, uint64_t seed, const agn_options& o) {
  if (!dims || n_dims < 2) return Status::Err(AGN_E_INVALID, "need at least two layer dims");
  for (int i = 0; i < n_dims; ++i)
    if (dims[i] <= 0) return Status::Err(AGN_E_INVALID, "layer dims must be positive");
  if (n_workers < 1 || n_workers > agn::kMaxPullsPerLaunch)
    return Status::Err(AGN_E_INVALID, "n_workers must be in [1, 256]");
  if (lambda < 1) return Status::Err(AGN_E_INVALID, "lambda must be >= 1");
  if (!(eta > 0.0) || !std::isfinite(eta)) return Status::Err(AGN_E_INVALID, "eta must be > 0");
  if (o.precision != AGN_PREC_FP32 && o.precision != AGN_PREC_BF16)
    return Status::Err(AGN_E_INVALID, "unknown precision");
  if (o.batch < 1) return Status::Err(AGN_E_INVALID, "batch must be >= 1");
  if (o.n_samples < n_workers) return Status::Err(AGN_E_INVALID, "need n_samples >= n_workers");
  if (o.input_dist != AGN_DIST_UNIFORM && o.input_dist != AGN_DIST_NORMAL)
    return Status::Err(AGN_E_INVALID, "unknown input distribution");
  if (o.tau_lo < 0 || o.tau_hi < o.tau_lo) return Status::Err(AGN_E_INVALID, "bad tau range");
  if (o.gemm != AGN_GEMM_AUTO && o.gemm != AGN_GEMM_SIMT && o.gemm != AGN_GEMM_TCGEN05)
    return Status::Err(AGN_E_INVALID, "unknown gemm backend");
  if (o.tc_mask < 0 || o.tc_mask > 1023) return Status::Err(AGN_E_INVALID, "tc_mask must be in [0, 1023]");
  if (o.commit_rule != AGN_COMMIT_AGN && o.commit_rule != AGN_COMMIT_DYNSGD)
    return Status::Err(AGN_E_INVALID, "unknown commit_rule");
  if (o.n_eval < 0 || o.n_eval > (int64_t)1 << 31)
    return Status::Err(AGN_E_INVALID, "n_eval must be in [0, 2^31]");
  if (o.n_eval > 0 && (o.x_init || o.y_init))
    return Status::Err(AGN_E_INVALID,
                       "the evaluation set is generated: not with caller-supplied inputs");
  if (o.local_optimizer != AGN_OPT_SGD && o.local_optimizer != AGN_OPT_ADAM)
    return Status::Err(AGN_E_INVALID, "unknown local_optimizer");
  if (o.adam_beta1 < 0.f || o.adam_beta1 >= 1.f || o.adam_beta2 < 0.f || o.adam_beta2 >= 1.f ||
      o.adam_eps < 0.f)
    return Status::Err(AGN_E_INVALID, "Adam betas must be in [0, 1) and eps >= 0 (0 = default)");
  if (o.local_optimizer == AGN_OPT_ADAM && (o.tc_mask & 8))
    return Status::Err(AGN_E_UNSUPPORTED,
                       "the one-tile-per-CTA dW kernel (tc_mask bit 3) has no gradient output");
  if (o.elide_accumulator && (o.tc_mask & 8))
    return Status::Err(AGN_E_UNSUPPORTED,
                       "the one-tile-per-CTA dW kernel (tc_mask bit 3) keeps the accumulator");
  h->dims.assign(dims, dims + n_dims);
  h->L = n_dims - 1;
  h->n = n_workers;
  h->lam = lambda;
  h->eta = eta;
  h->seed = seed;
  h->prec = o.precision;
  h->m = o.batch;
  h->N = o.n_samples;
  h->S = o.n_samples / n_workers;
  h->dist = o.input_dist;
  h->normalize = o.normalize ? 1 : 0;
  h->commit_rule = o.commit_rule;
  h->elide = o.elide_accumulator != 0;
  h->adam = o.local_optimizer == AGN_OPT_ADAM;
  if (o.adam_beta1 > 0.f) h->beta1 = o.adam_beta1;
  if (o.adam_beta2 > 0.f) h->beta2 = o.adam_beta2;
  if (o.adam_eps > 0.f) h->eps = o.adam_eps;
  h->gemm = o.gemm;
  h->tau_lo = o.tau_lo;
  h->tau_hi = o.tau_hi;
  if (o.teacher_dims && o.n_teacher_dims >= 2) {
    h->tdims.assign(o.teacher_dims, o.teacher_dims + o.n_teacher_dims);
    if (h->tdims.front() != dims[0] || h->tdims.back() != dims[n_dims - 1])
      return Status::Err(AGN_E_INVALID, "teacher dims must start at d_0 and end at d_L");
    for (int d : h->tdims)
      if (d <= 0) return Status::Err(AGN_E_INVALID, "teacher dims must be positive");
  } else {
    h->tdims = {dims[0], 64, dims[n_dims - 1]};
  }
  // parameter layouts: flat (the ABI's order) and padded (device, 64-element aligned tensors)
  int64_t off = 0, offp = 0;
  h->maxd = 0;
  for (int l = 1; l <= h->L; ++l) {
    const int64_t fi = dims[l - 1], fo = dims[l];
    h->woff_flat.push_back(off);
    h->boff_flat.push_back(off + fo * fi);
    off += fo * fi + fo;
    offp = round_up(offp, 64);
    h->woff.push_back(offp);
    offp = round_up(offp + fo * fi, 64);
    h->boff.push_back(offp);
    offp += fo;
    h->maxd = std::max<int>(h->maxd, (int)fo);
  }
  h->P = off;
  h->P_pad = round_up(offp, 64);
  // tcgen05 path: m <= 256, a hidden layer, every TMA row 16-byte aligned.
  // bf16 mode feeds bf16 operands; fp32 mode feeds each fp32 operand as three
  // exact bf16 pieces (split mode).
  bool tc_ok = h->m <= 256 && h->L >= 2;
  for (int l = 0; l < h->L; ++l) tc_ok = tc_ok && dims[l] % 8 == 0;
  if (o.gemm == AGN_GEMM_TCGEN05 && !tc_ok)
    return Status::Err(AGN_E_UNSUPPORTED,
                       "tcgen05 GEMMs need batch <= 256, at least one hidden layer "
                       "and d_0 .. d_{L-1} multiples of 8");
  h->use_tc = tc_ok && o.gemm != AGN_GEMM_SIMT;
  h->split = h->use_tc && h->prec == AGN_PREC_FP32;
  h->tc_mask = (o.tc_mask & 7) == 0 ? (o.tc_mask | 7) : o.tc_mask;
  h->prev.assign(h->n, -1);
  h->pulled_v.assign(h->n, 0);
  h->steps.assign(h->n, 0);

  AGN_TRY_CUDA(cudaGetDevice(&h->device));
  AGN_TRY_CUDA(cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device));
  if (o.stream) {
    h->stream = static_cast<cudaStream_t>(o.stream);
  } else {
    AGN_TRY_CUDA(cudaStreamCreateWithFlags(&h->stream, cudaStreamNonBlocking));
    h->own_stream = true;
  }
  AGN_TRY_CUDA(cudaEventCreate(&h->ev0));
  AGN_TRY_CUDA(cudaEventCreate(&h->ev1));

  // host inputs
  const int d0 = dims[0];
  h->hX.resize((size_t)h->N * d0);
  h->hy.resize((size_t)h->N);
  h->htheta0.resize((size_t)h->P);
  if (o.x_init) std::memcpy(h->hX.data(), o.x_init, h->hX.size() * sizeof(float));
  else agn::gen_dataset(seed, d0, h->N, h->dist, h->hX.data());
  if (o.y_init) {
    std::memcpy(h->hy.data(), o.y_init, h->hy.size() * sizeof(int32_t));
    for (int32_t v : h->hy)
      if (v < 0 || v >= dims[n_dims - 1]) return Status::Err(AGN_E_INVALID, "label out of range");
  } else {
    auto Ws = agn::gen_teacher(seed, h->tdims);
    agn::gen_teacher_labels(h->hX.data(), h->N, d0, h->dist, h->tdims, Ws, h->hy.data());
  }
  if (o.theta_init) std::memcpy(h->htheta0.data(), o.theta_init, h->htheta0.size() * sizeof(float));
  else agn::gen_init(seed, h->dims, h->htheta0.data());
  std::vector<float> hXe;
  std::vector<int32_t> hye;
  if (o.n_eval > 0) {   // held-out rows of the same generator, labelled by the same teacher
    h->n_eval = o.n_eval;
    hXe.resize((size_t)(o.n_eval * d0));
    hye.resize((size_t)o.n_eval);
    agn::gen_dataset_rows(seed, d0, h->N, o.n_eval, h->dist, hXe.data());
    auto Ws = agn::gen_teacher(seed, h->tdims);
    agn::gen_teacher_labels(hXe.data(), o.n_eval, d0, h->dist, h->tdims, Ws, hye.data());
  }

  // device buffers
  const size_t es = elem_size(h);
  const int64_t n = h->n, m = h->m;
  AGN_TRY(dalloc_t(h, &h->theta_c, (size_t)h->P_pad));
  AGN_TRY(dalloc_t(h, &h->rep, (size_t)(n * h->P_pad)));
  AGN_TRY(dalloc_t(h, &h->acc, (size_t)(n * h->P_pad)));
  if (h->prec == AGN_PREC_BF16) AGN_TRY(dalloc_t(h, &h->rep_b, (size_t)(n * h->P_pad)));
  if (h->adam) {   // gradients and the two moments of every worker, zero to start
    AGN_TRY(dalloc_t(h, &h->grad, (size_t)(n * h->P_pad)));
    AGN_TRY(dalloc_t(h, &h->mom1, (size_t)(n * h->P_pad)));
    AGN_TRY(dalloc_t(h, &h->mom2, (size_t)(n * h->P_pad)));
    for (float* p : {h->grad, h->mom1, h->mom2})
      AGN_TRY_CUDA(cudaMemset(p, 0, (size_t)(n * h->P_pad) * sizeof(float)));
  }
  h->use_head = h->prec == AGN_PREC_BF16 ? agn::head_fits<bf16>(dims[h->L - 1], dims[h->L])
                                         : agn::head_fits<float>(dims[h->L - 1], dims[h->L]);
  h->fuse_out_dw = h->use_tc && h->use_head && h->L >= 2 && (h->tc_mask & 4) && !(h->tc_mask & 8);
  h->ldz_out = h->fuse_out_dw ? (int)round_up(dims[h->L], 8) : dims[h->L];
  h->fuse_head = h->use_tc && h->use_head && h->L >= 2 && (h->tc_mask & 1) &&
                 !(h->tc_mask & 32) && dims[h->L] <= agn::kHeadMaxClasses;
  if (h->split) {   // three piece planes of the activations (the weights stay fp32)
    h->Hs.assign(h->L, nullptr);
    for (int l = 0; l + 1 < h->L + (h->fuse_out_dw ? 1 : 0); ++l)
      AGN_TRY(dalloc_t(h, &h->Hs[l], (size_t)(3 * n * m * dims[l])));
    h->dZp.assign(h->L + 1, nullptr);
    for (int l = 1; l < h->L; ++l) AGN_TRY(dalloc_t(h, &h->dZp[l], (size_t)(3 * n * m * dims[l])));
    if (h->fuse_out_dw) {
      AGN_TRY(dalloc_t(h, &h->dZp[h->L], (size_t)(3 * n * m * h->ldz_out)));
      AGN_TRY_CUDA(cudaMemset(h->dZp[h->L], 0, (size_t)(3 * n * m * h->ldz_out) * sizeof(bf16)));
    }
  }
  AGN_TRY(dalloc(h, &h->X, (size_t)h->N * d0 * es));
  AGN_TRY(dalloc_t(h, &h->y, (size_t)h->N));
  AGN_TRY(dalloc(h, &h->Xb, (size_t)(n * m * d0) * es));
  // the gather may run ahead of the preceding kernel when every reader of
  // layer 1's operand is a tensor-core kernel (forward and dW)
  h->early_gather = h->use_tc && (h->tc_mask & 1) && (h->tc_mask & 4) && !(h->tc_mask & 8) &&
                    h->L >= 2 && d0 % 4 == 0;
  // no gather at all when, besides, every reader of the labels is one of the
  // output-layer kernels (the padded shards replace the alternate buffers)
  h->direct_x = h->early_gather && h->use_head && !(h->tc_mask & 64);
  if (h->direct_x) {
    h->early_gather = false;
    const size_t rows = (size_t)(n * (h->S + m));
    if (h->split) AGN_TRY(dalloc_t(h, &h->Hs0_pad, 3 * rows * (size_t)d0));
    else AGN_TRY(dalloc(h, &h->Xpad, rows * (size_t)d0 * es));
    AGN_TRY(dalloc_t(h, &h->zero_t0, (size_t)n));
    AGN_TRY_CUDA(cudaMemset(h->zero_t0, 0, (size_t)n * sizeof(long long)));
  }
  if (h->early_gather) {
    if (h->split) AGN_TRY(dalloc_t(h, &h->Hs0_alt, (size_t)(3 * n * m * d0)));
    else AGN_TRY(dalloc(h, &h->Xb_alt, (size_t)(n * m * d0) * es));
  }
  AGN_TRY(dalloc_t(h, &h->yb, (size_t)(n * (h->direct_x ? h->S + m : m))));
  h->H.assign(h->L, nullptr);
  for (int l = 1; l < h->L; ++l) AGN_TRY(dalloc(h, &h->H[l], (size_t)(n * m * dims[l]) * es));
  AGN_TRY(dalloc_t(h, &h->Z, (size_t)(n * m * dims[h->L])));
  h->dZ.assign(h->L + 1, nullptr);
  for (int l = 1; l < h->L; ++l) AGN_TRY(dalloc(h, &h->dZ[l], (size_t)(n * m * dims[l]) * es));
  AGN_TRY(dalloc(h, &h->dZ[h->L], (size_t)(n * m * h->ldz_out) * es));
  AGN_TRY_CUDA(cudaMemset(h->dZ[h->L], 0, (size_t)(n * m * h->ldz_out) * es));
  AGN_TRY(dalloc_t(h, &h->flag, 2));
  AGN_TRY(dalloc_t(h, &h->ce_partial, (size_t)(n * ceil_div(m, agn::kHeadSamples))));
  AGN_TRY(dalloc_t(h, &h->head_counter, (size_t)n));
  if (h->n_eval > 0) {
    const int64_t E = h->n_eval;
    h->eval_chunk = std::min<int64_t>(E, 4096);
    int maxh = 1;
    for (int l = 1; l < h->L; ++l) maxh = std::max(maxh, dims[l]);
    AGN_TRY(dalloc_t(h, &h->Xe, (size_t)(E * d0)));
    AGN_TRY(dalloc_t(h, &h->ye, (size_t)E));
    AGN_TRY(dalloc_t(h, &h->He[0], (size_t)(h->eval_chunk * maxh)));
    AGN_TRY(dalloc_t(h, &h->He[1], (size_t)(h->eval_chunk * maxh)));
    AGN_TRY(dalloc_t(h, &h->Ze, (size_t)(h->eval_chunk * dims[h->L])));
    AGN_TRY(dalloc_t(h, &h->e_loss, (size_t)E));
    AGN_TRY(dalloc_t(h, &h->e_correct, (size_t)E));
    AGN_TRY(dalloc_t(h, &h->e_pred, (size_t)E));
    AGN_TRY(dalloc_t(h, &h->e_out, 2));
    AGN_TRY(dalloc_t(h, &h->e_sw, 1));
    AGN_TRY_CUDA(cudaMemcpy(h->Xe, hXe.data(), hXe.size() * sizeof(float), cudaMemcpyHostToDevice));
    AGN_TRY_CUDA(cudaMemcpy(h->ye, hye.data(), hye.size() * sizeof(int32_t), cudaMemcpyHostToDevice));
    AGN_TRY_CUDA(cudaMemset(h->e_sw, 0, sizeof(int)));
  }
  AGN_TRY_CUDA(cudaMemsetAsync(h->head_counter, 0, (size_t)n * sizeof(int), h->stream));
  if (h->fuse_head) {
    const int64_t nchk = ceil_div(m, 32), mt = ceil_div(dims[h->L - 1], 128);
    AGN_TRY(dalloc_t(h, &h->fh_part, (size_t)(n * nchk * mt * 32 * agn::kHeadMaxClasses)));
    AGN_TRY(dalloc_t(h, &h->fh_counter, (size_t)(2 * n * nchk)));
    AGN_TRY_CUDA(cudaMemsetAsync(h->fh_counter, 0, (size_t)(2 * n * nchk) * sizeof(int),
                                 h->stream));
    h->loss_q = (int)nchk;
  }
  h->grid = agn::commit_grid(h->P_pad);
  AGN_TRY(dalloc_t(h, &h->partials, (size_t)agn::kMaxCommitsPerLaunch * h->grid));
  AGN_TRY(dalloc_t(h, &h->pull_list, (size_t)n));
  AGN_TRY(dalloc_t(h, &h->dnorm, 1024));
  AGN_TRY(dalloc_t(h, &h->loss, 1024));
  h->cap_commits = 1024;

  // uploads
  std::vector<float> tpad((size_t)h->P_pad, 0.f);
  for (int l = 0; l < h->L; ++l) {
    const int64_t fi = dims[l], fo = dims[l + 1];
    std::memcpy(&tpad[h->woff[l]], &h->htheta0[h->woff_flat[l]], (size_t)(fo * fi) * sizeof(float));
    std::memcpy(&tpad[h->boff[l]], &h->htheta0[h->boff_flat[l]], (size_t)fo * sizeof(float));
  }
  AGN_TRY_CUDA(cudaMemcpy(h->theta_c, tpad.data(), tpad.size() * sizeof(float),
                          cudaMemcpyHostToDevice));
  if (h->prec == AGN_PREC_BF16) {
    std::vector<bf16> xb(h->hX.size());
    for (size_t i = 0; i < xb.size(); ++i) xb[i] = __float2bfloat16_rn(h->hX[i]);
    AGN_TRY_CUDA(cudaMemcpy(h->X, xb.data(), xb.size() * sizeof(bf16), cudaMemcpyHostToDevice));
  } else {
    AGN_TRY_CUDA(cudaMemcpy(h->X, h->hX.data(), h->hX.size() * sizeof(float),
                            cudaMemcpyHostToDevice));
  }
  AGN_TRY_CUDA(cudaMemcpy(h->y, h->hy.data(), h->hy.size() * sizeof(int32_t),
                          cudaMemcpyHostToDevice));
  AGN_TRY_CUDA(cudaMemsetAsync(h->acc, 0, (size_t)(n * h->P_pad) * sizeof(float), h->stream));
  AGN_TRY_CUDA(cudaMemsetAsync(h->flag, 0, 2 * sizeof(int), h->stream));
  if (h->use_tc) {
    AGN_TRY(build_tc_maps(h));
    AGN_TRY(dalloc_t(h, &h->tc_part, (size_t)h->num_sms * 256 * 128));
    AGN_TRY(dalloc_t(h, &h->tc_counter, (size_t)(2 * h->num_sms)));
    AGN_TRY_CUDA(cudaMemsetAsync(h->tc_counter, 0, (size_t)(2 * h->num_sms) * sizeof(int),
                                 h->stream));
  }
  std::vector<int> all(n);
  for (int w = 0; w < n; ++w) all[w] = w;
  AGN_TRY_CUDA(cudaMemcpyAsync(h->pull_list, all.data(), n * sizeof(int), cudaMemcpyHostToDevice,
                               h->stream));
  AGN_TRY(agn::bounds_upload(h->stream));   // bounds-checked build: the handle's buffers
  if (h->direct_x) {
    // the padded shards: worker w's rows r = 0 .. S + m - 1 are the gather of
    // one "step" of S + m rows from step counter 0 (row (0 + r) mod S)
    const int rows = (int)(h->S + m);
    const int64_t plane = n * (int64_t)rows * d0;
    if (h->split)
      AGN_TRY(agn::gather_batch<float>(static_cast<const float*>(h->X), h->y, nullptr, h->yb,
                                       d0, rows, h->S, h->pull_list, h->zero_t0, 0, (int)n,
                                       h->stream, h->Hs0_pad, plane, 0));
    else   // (the tensor cores' fp32 mode is the split one: this is bf16)
      AGN_TRY(agn::gather_batch<bf16>(static_cast<const bf16*>(h->X), h->y,
                                      static_cast<bf16*>(h->Xpad), h->yb, d0, rows, h->S,
                                      h->pull_list, h->zero_t0, 0, (int)n, h->stream, nullptr, 0,
                                      0));
  }
  AGN_TRY(agn::pull_replicas(h->theta_c, h->rep, h->rep_b, h->P_pad, h->P_pad, h->pull_list,
                             (int)n, h->stream, h->piece_plane,
                             h->elide ? h->acc : nullptr));   // every worker pulls version 0
  AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
  AGN_TRY(agn::bounds_collect(h->stream));
  return Status::Ok();
}

// Loss and accuracy of theta~ on the held-out set: the forward pass on the
// CUDA-core fp32 GEMMs (theta~ as every row block's weights), then per-sample
// log-sum-exp / argmax and fixed-order means.
Status evaluate(agn_handle* h, float* loss, float* accuracy, int32_t* pred, int64_t cap) {
  if (h->n_eval <= 0)
    return Status::Err(AGN_E_INVALID, "the handle has no evaluation set (agn_options.n_eval)");
  if (pred && cap < h->n_eval) return Status::Err(AGN_E_INVALID, "pred shorter than n_eval");
  const int L = h->L, C = h->dims[L];
  AGN_TRY(agn::bounds_upload(h->stream));   // bounds-checked build only
  for (int64_t r0 = 0; r0 < h->n_eval; r0 += h->eval_chunk) {
    const int rows = (int)std::min<int64_t>(h->eval_chunk, h->n_eval - r0);
    const float* in = h->Xe + r0 * h->dims[0];
    for (int l = 1; l <= L; ++l) {
      const int fi = h->dims[l - 1], fo = h->dims[l];
      agn::GemmArgs g{};
      g.M = rows; g.N = fo; g.K = fi;
      g.a = in; g.lda = fi;
      g.b = h->theta_c + h->woff[l - 1]; g.ldb = fi;   // b_bstride 0: one weight set
      g.slot_worker = h->e_sw;
      float* out = l == L ? h->Ze : h->He[l % 2];
      g.out = out; g.ldo = fo;
      g.relu = l < L;
      g.theta = h->theta_c; g.ld_param = 0; g.boff = h->boff[l - 1];
      AGN_TRY(agn::simt_forward<float>(g, l == L, 1, h->stream));
      in = out;
    }
    AGN_TRY(agn::eval_logits(h->Ze, h->ye + r0, rows, C, h->e_loss + r0, h->e_correct + r0,
                             h->e_pred + r0, h->stream));
  }
  AGN_TRY(agn::eval_reduce(h->e_loss, h->e_correct, h->n_eval, h->e_out, h->stream));
  float o2[2];
  AGN_TRY_CUDA(cudaMemcpyAsync(o2, h->e_out, sizeof(o2), cudaMemcpyDeviceToHost, h->stream));
  if (pred)
    AGN_TRY_CUDA(cudaMemcpyAsync(pred, h->e_pred, (size_t)h->n_eval * sizeof(int32_t),
                                 cudaMemcpyDeviceToHost, h->stream));
  AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
  AGN_TRY(agn::bounds_collect(h->stream));
  if (loss) *loss = o2[0];
  if (accuracy) *accuracy = o2[1];
  return Status::Ok();
}

Status read_params(agn_handle* h, const float* dev, float* out, int64_t cap) {
  if (!out || cap < h->P) return Status::Err(AGN_E_INVALID, "output buffer shorter than P");
  std::vector<float> tpad((size_t)h->P_pad);
  AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
  AGN_TRY_CUDA(cudaMemcpy(tpad.data(), dev, tpad.size() * sizeof(float), cudaMemcpyDeviceToHost));
  for (int l = 0; l < h->L; ++l) {
    const int64_t fi = h->dims[l], fo = h->dims[l + 1];
    std::memcpy(out + h->woff_flat[l], &tpad[h->woff[l]], (size_t)(fo * fi) * sizeof(float));
    std::memcpy(out + h->boff_flat[l], &tpad[h->boff[l]], (size_t)fo * sizeof(float));
  }
  return Status::Ok();
}

Status read_commit_array(agn_handle* h, const float* dev, float* out, int64_t cap) {
  if (h->V > 0 && (!out || cap < h->V))
    return Status::Err(AGN_E_INVALID, "output buffer shorter than the number of commits");
  AGN_TRY_CUDA(cudaStreamSynchronize(h->stream));
  if (h->V > 0)
    AGN_TRY_CUDA(cudaMemcpy(out, dev, (size_t)h->V * sizeof(float), cudaMemcpyDeviceToHost));
  return Status::Ok();
}

// ---------------------------------------------------------------------------
// Standalone commit + pull
// ---------------------------------------------------------------------------

Status commit_pull(float* theta_c, float* acc, float* reps, void* reps_b, int64_t P, int64_t ld,
                   int n, int C, const int32_t* cw, const int32_t* po, const int32_t* pw,
                   double eta, int lambda, int normalize, float* dnorm, cudaStream_t st) {
  if (P < 1 || ld < P || ld % 4 != 0 || n < 1 || C < 0 || lambda < 1 || !(eta > 0.0))
    return Status::Err(AGN_E_INVALID, "bad sizes (need P >= 1, ld >= P, ld % 4 == 0, n >= 1)");
  if (!theta_c || !acc || (C > 0 && (!cw || !po)))
    return Status::Err(AGN_E_INVALID, "null pointer");
  auto misaligned = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) != 0; };
  if (misaligned(theta_c) || misaligned(acc) || (reps && misaligned(reps)) ||
      (reps_b && (reinterpret_cast<uintptr_t>(reps_b) & 7) != 0))
    return Status::Err(AGN_E_INVALID, "device buffers must be 16-byte aligned");
  if (C == 0) return Status::Ok();
  if (po[0] != 0) return Status::Err(AGN_E_INVALID, "pull_offsets[0] must be 0");
  // offsets first (they bound every later read), then the pointers the pulls need
  for (int c = 0; c < C; ++c)
    if (po[c + 1] < po[c]) return Status::Err(AGN_E_INVALID, "pull_offsets must not decrease");
  if (po[C] > 0 && (!reps || !pw)) return Status::Err(AGN_E_INVALID, "pulls need replicas");
  for (int c = 0; c < C; ++c) {
    if (cw[c] < 0 || cw[c] >= n) return Status::Err(AGN_E_INVALID, "commit worker out of range");
    for (int p = po[c]; p < po[c + 1]; ++p)
      if (pw[p] < 0 || pw[p] >= n) return Status::Err(AGN_E_INVALID, "pull worker out of range");
  }
  const float scale = (float)(normalize ? -(eta / (double)lambda) : -eta);
  const int grid = agn::commit_grid(P);
  double* partials = nullptr;
  if (dnorm) AGN_TRY_CUDA(cudaMallocAsync((void**)&partials,
                                          sizeof(double) * agn::kMaxCommitsPerLaunch * grid, st));
  int* extra_dev = nullptr;
  // bounds-checked build: the caller's buffers are known for this call
  // (the extents this entry point's arguments give them)
  struct CallBuffers {
    std::vector<const void*> added;
    void add(const void* p, size_t b) {
      if (p) {
        agn::bounds_add(p, b);
        added.push_back(p);
      }
    }
    ~CallBuffers() {
      for (const void* p : added) agn::bounds_remove(p);
    }
  } call;
  call.add(theta_c, (size_t)P * sizeof(float));
  call.add(acc, (size_t)n * ld * sizeof(float));
  call.add(reps, (size_t)n * ld * sizeof(float));
  call.add(reps_b, (size_t)n * ld * sizeof(bf16));
  call.add(dnorm, (size_t)C * sizeof(float));
  call.add(partials, sizeof(double) * agn::kMaxCommitsPerLaunch * grid);
#ifdef AGN_BOUNDS_CHECK
  if (po[C] > 0) {   // the list of pulls beyond one launch's capacity, known up front
    AGN_TRY_CUDA(cudaMallocAsync((void**)&extra_dev, sizeof(int) * n, st));
    call.add(extra_dev, sizeof(int) * n);
  }
#endif
  AGN_TRY(agn::bounds_upload(st));
  Status result = Status::Ok();
  CommitPlan cp{};
  std::vector<int> extra;            // pulls that did not fit into the launch
  auto flush = [&]() -> Status {
    if (cp.n_commits > 0)
      AGN_TRY(agn::launch_commit_pull(cp, theta_c, acc, reps, static_cast<bf16*>(reps_b), P, ld,
                                      scale, true, partials, grid, dnorm, nullptr, st));
    if (!extra.empty()) {
      if (!extra_dev) AGN_TRY_CUDA(cudaMallocAsync((void**)&extra_dev, sizeof(int) * n, st));
      for (size_t b = 0; b < extra.size(); b += (size_t)n) {
        const int cnt = (int)std::min<size_t>((size_t)n, extra.size() - b);
        AGN_TRY_CUDA(cudaMemcpyAsync(extra_dev, extra.data() + b, sizeof(int) * cnt,
                                     cudaMemcpyHostToDevice, st));
        AGN_TRY(agn::pull_replicas(theta_c, reps, static_cast<bf16*>(reps_b), P, ld, extra_dev,
                                   cnt, st));
        // the host vector must outlive the copy
        AGN_TRY_CUDA(cudaStreamSynchronize(st));
      }
      extra.clear();
    }
    cp = CommitPlan{};
    return Status::Ok();
  };
  for (int c = 0; c < C && result.ok(); ++c) {
    bool dup = false;
    for (int i = 0; i < cp.n_commits; ++i) dup |= cp.worker[i] == cw[c];
    const int np = po[c + 1] - po[c];
    if (cp.n_commits == agn::kMaxCommitsPerLaunch || dup ||
        (cp.n_commits > 0 && cp.pull_begin[cp.n_commits] + np > agn::kMaxPullsPerLaunch)) {
      result = flush();
      if (!result.ok()) break;
    }
    const int i = cp.n_commits;
    cp.worker[i] = cw[c];
    cp.norm_slot[i] = c;
    int pb = cp.pull_begin[i];
    int p = po[c];
    for (; p < po[c + 1] && pb < agn::kMaxPullsPerLaunch; ++p) cp.pull_worker[pb++] = pw[p];
    cp.pull_begin[i + 1] = pb;
    cp.n_commits = i + 1;
    if (p < po[c + 1]) {   // more pulls than one launch holds: finish them after it
      for (; p < po[c + 1]; ++p) extra.push_back(pw[p]);
      result = flush();
    }
  }
  if (result.ok()) result = flush();
  if (result.ok()) result = agn::bounds_collect(st);   // bounds-checked build only
  if (partials) cudaFreeAsync(partials, st);
  if (extra_dev) cudaFreeAsync(extra_dev, st);
  return result;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

extern "C" {

void agn_default_options(agn_options* o) {
  if (!o) return;
  std::memset(o, 0, sizeof(*o));
  o->precision = AGN_PREC_FP32;
  o->batch = 32;
  o->n_samples = 2048;
  o->input_dist = AGN_DIST_UNIFORM;
  o->normalize = 1;
  o->gemm = AGN_GEMM_AUTO;
  o->tau_lo = 0;
  o->tau_hi = 0;
  o->commit_rule = AGN_COMMIT_AGN;
}

int agn_create(const int32_t* dims, int32_t n_dims, int32_t n_workers, int32_t lambda, double eta,
               uint64_t seed, const agn_options* opt, agn_handle** out) {
  if (!out) return fail(nullptr, AGN_E_INVALID, "out is null");
  *out = nullptr;
  agn_options o;
  if (opt) o = *opt; else agn_default_options(&o);
  agn_handle* h = new (std::nothrow) agn_handle();
  if (!h) return fail(nullptr, AGN_E_OOM, "host allocation failed");
  Status s;
  try {
    s = create(h, dims, n_dims, n_workers, lambda, eta, seed, o);
  } catch (const std::bad_alloc&) {
    s = Status::Err(AGN_E_OOM, "host allocation failed");
  }
  if (!s.ok()) {
    g_error = s.msg;
    agn_destroy(h);
    return s.code;
  }
  *out = h;
  return AGN_OK;
}

int agn_run(agn_handle* h, int32_t n_commits, const int32_t* worker, const int32_t* staleness,
            int32_t n_schedule) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  DeviceGuard g(h->device);
  if (n_commits < 0) return fail(h, AGN_E_INVALID, "n_commits < 0");
  if (n_commits == 0) return AGN_OK;
  std::vector<int32_t> w, t;
  if (!worker && !staleness) {
    const int64_t total = h->V + n_commits + h->n;
    w.resize(total);
    t.resize(total);
    agn::gen_schedule(h->n, total, h->tau_lo, h->tau_hi, h->seed, w.data(), t.data());
    worker = w.data() + h->V;
    staleness = t.data() + h->V;
    n_schedule = n_commits + h->n;
  } else if (!worker || !staleness) {
    return fail(h, AGN_E_INVALID, "give both schedule arrays or neither");
  }
  if (n_schedule < n_commits) return fail(h, AGN_E_INVALID, "n_schedule < n_commits");
  try {
    Status s = do_run(h, n_commits, worker, staleness, n_schedule);
    if (!s.ok()) return fail(h, s);
  } catch (const std::bad_alloc&) {
    return fail(h, AGN_E_OOM, "host allocation failed");
  }
  return AGN_OK;
}

int agn_central(agn_handle* h, float* out, int64_t cap) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  DeviceGuard g(h->device);
  Status s = read_params(h, h->theta_c, out, cap);
  return s.ok() ? AGN_OK : fail(h, s);
}

int agn_replica(agn_handle* h, int32_t k, float* out, int64_t cap) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  if (k < 0 || k >= h->n) return fail(h, AGN_E_INVALID, "replica index out of range");
  DeviceGuard g(h->device);
  Status s = read_params(h, h->rep + (int64_t)k * h->P_pad, out, cap);
  return s.ok() ? AGN_OK : fail(h, s);
}

int agn_loss(agn_handle* h, float* out, int64_t cap) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  DeviceGuard g(h->device);
  Status s = read_commit_array(h, h->loss, out, cap);
  return s.ok() ? AGN_OK : fail(h, s);
}

int agn_evaluate(agn_handle* h, float* loss, float* accuracy, int32_t* pred, int64_t cap) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  DeviceGuard g(h->device);
  Status s = evaluate(h, loss, accuracy, pred, cap);
  return s.ok() ? AGN_OK : fail(h, s);
}

int agn_temporal_efficiency(const double* ta, const double* fa, int64_t na, const double* tb,
                            const double* fb, int64_t nb, double* out) {
  Status s = agn::temporal_efficiency(ta, fa, na, tb, fb, nb, out);
  return s.ok() ? AGN_OK : fail(nullptr, s);
}

int agn_delta_norm(agn_handle* h, float* out, int64_t cap) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  DeviceGuard g(h->device);
  Status s = read_commit_array(h, h->dnorm, out, cap);
  return s.ok() ? AGN_OK : fail(h, s);
}

int64_t agn_num_params(const agn_handle* h) { return h ? h->P : -1; }
int64_t agn_num_commits(const agn_handle* h) { return h ? h->V : -1; }

int agn_last_run_stats(const agn_handle* h, double* out, int64_t cap) {
  if (!h || !out || cap < 4) return fail(const_cast<agn_handle*>(h), AGN_E_INVALID, "need 4 slots");
  for (int i = 0; i < (int)std::min<int64_t>(cap, 5); ++i) out[i] = h->stats[i];
  return AGN_OK;
}

int agn_generate_inputs(const int32_t* dims, int32_t n_dims, int32_t input_dist,
                        const int32_t* teacher_dims, int32_t n_teacher_dims, uint64_t seed,
                        int64_t row0, int64_t n_rows, float* x, int32_t* y, float* theta0) {
  if (!dims || n_dims < 2 || row0 < 0 || n_rows < 0 ||
      (input_dist != AGN_DIST_UNIFORM && input_dist != AGN_DIST_NORMAL))
    return fail(nullptr, AGN_E_INVALID, "bad arguments");
  for (int i = 0; i < n_dims; ++i)
    if (dims[i] <= 0) return fail(nullptr, AGN_E_INVALID, "layer dims must be positive");
  std::vector<int> td;
  if (teacher_dims && n_teacher_dims >= 2) td.assign(teacher_dims, teacher_dims + n_teacher_dims);
  else td = {dims[0], 64, dims[n_dims - 1]};
  if (td.front() != dims[0] || td.back() != dims[n_dims - 1])
    return fail(nullptr, AGN_E_INVALID, "teacher dims must start at d_0 and end at d_L");
  try {
    std::vector<float> xs;
    float* xp = x;
    if (!xp && y) {
      xs.resize((size_t)n_rows * dims[0]);
      xp = xs.data();
    }
    if (xp) agn::gen_dataset_rows(seed, dims[0], row0, n_rows, input_dist, xp);
    if (y) {
      auto Ws = agn::gen_teacher(seed, td);
      agn::gen_teacher_labels(xp, n_rows, dims[0], input_dist, td, Ws, y);
    }
    if (theta0) agn::gen_init(seed, std::vector<int>(dims, dims + n_dims), theta0);
  } catch (const std::bad_alloc&) {
    return fail(nullptr, AGN_E_OOM, "host allocation failed");
  }
  return AGN_OK;
}

int agn_export_inputs(agn_handle* h, float* x, int32_t* y, float* theta0) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  if (x) std::memcpy(x, h->hX.data(), h->hX.size() * sizeof(float));
  if (y) std::memcpy(y, h->hy.data(), h->hy.size() * sizeof(int32_t));
  if (theta0) std::memcpy(theta0, h->htheta0.data(), h->htheta0.size() * sizeof(float));
  return AGN_OK;
}

int agn_profile(agn_handle* h, int32_t mode) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  if (mode == 0) {
    if (h->prof) --agn::g_pdl_off;
    h->prof = false;
  } else if (mode == 1) {
    if (!h->prof) ++agn::g_pdl_off;   // no launch overlap while events time each kernel
    h->prof = true;
  } else if (mode == 2) {
    std::memset(h->kstats, 0, sizeof(h->kstats));
  }
  else return fail(h, AGN_E_INVALID, "mode must be 0, 1 or 2");
  return AGN_OK;
}

int agn_kernel_stats(const agn_handle* h, double* out, int64_t cap) {
  if (!h || !out || cap < 4 * AGN_KERNEL_CLASSES)
    return fail(const_cast<agn_handle*>(h), AGN_E_INVALID, "need 4 * AGN_KERNEL_CLASSES slots");
  std::memcpy(out, h->kstats, sizeof(h->kstats));
  return AGN_OK;
}

const char* agn_last_error(const agn_handle* h) { return h ? h->err.c_str() : g_error.c_str(); }

void agn_destroy(agn_handle* h) {
  if (!h) return;
  if (h->prof) --agn::g_pdl_off;
  DeviceGuard g(h->device);
  if (h->stream) cudaStreamSynchronize(h->stream);
  for (void* p : h->allocs)
    if (p) {
      agn::bounds_remove(p);
      cudaFree(p);
    }
  for (cudaEvent_t e : h->ev_pool) cudaEventDestroy(e);
  if (h->ev0) cudaEventDestroy(h->ev0);
  if (h->ev1) cudaEventDestroy(h->ev1);
  if (h->own_stream && h->stream) cudaStreamDestroy(h->stream);
  delete h;
}

int agn_make_schedule(int32_t n, int32_t n_commits, int32_t tau_lo, int32_t tau_hi, uint64_t seed,
                      int32_t* worker_out, int32_t* tau_out) {
  if (n < 1 || n_commits < 0 || tau_lo < 0 || tau_hi < tau_lo || (n_commits > 0 && (!worker_out || !tau_out)))
    return fail(nullptr, AGN_E_INVALID, "bad schedule arguments");
  agn::gen_schedule(n, n_commits, tau_lo, tau_hi, seed, worker_out, tau_out);
  return AGN_OK;
}

int agn_plan_waves(int32_t n_workers, int32_t lambda, int32_t n_commits, const int32_t* worker,
                   const int32_t* staleness, int32_t n_schedule, int32_t* n_waves_out,
                   int32_t* wave_slots, int32_t* wave_end, int32_t* slot_commit,
                   int64_t* slot_t0, int64_t pull_cap, int32_t* pull_version,
                   int32_t* pull_worker, int64_t* n_pulls_out) {
  if (n_workers < 1 || n_workers > agn::kMaxPullsPerLaunch || lambda < 1 || n_commits < 0 ||
      n_schedule < n_commits || pull_cap < 0 ||
      !n_waves_out || !n_pulls_out ||
      (n_schedule > 0 && (!worker || !staleness)) ||
      (n_commits > 0 && (!wave_slots || !wave_end || !slot_commit || !slot_t0)) ||
      (pull_cap > 0 && (!pull_version || !pull_worker)))
    return fail(nullptr, AGN_E_INVALID, "bad plan arguments");
  // the planning state of a fresh handle: no commits, every replica at version 0
  agn_handle h;
  h.n = n_workers;
  h.lam = lambda;
  h.V = 0;
  h.prev.assign(n_workers, -1);
  h.pulled_v.assign(n_workers, 0);
  h.steps.assign(n_workers, 0);
  RunPlan plan;
  Status s = build_plan(&h, n_commits, worker, staleness, n_schedule, &plan);
  if (!s.ok()) return fail(nullptr, s);
  int64_t np = 0;
  auto add_pull = [&](int v, int w) {
    if (np < pull_cap) {
      pull_version[np] = v;
      pull_worker[np] = w;
    }
    ++np;
  };
  for (int w : plan.start_pulls) add_pull(0, w);
  int applied = 0;
  for (size_t i = 0; i < plan.waves.size(); ++i) {
    const Wave& wv = plan.waves[i];
    wave_slots[i] = wv.slots;
    for (const CommitPlan& cp : wv.commits) {
      for (int c = 0; c < cp.n_commits; ++c) {
        for (int p = cp.pull_begin[c]; p < cp.pull_begin[c + 1]; ++p)
          add_pull(cp.norm_slot[c] + 1, cp.pull_worker[p]);
        ++applied;
      }
    }
    wave_end[i] = applied;
  }
  for (size_t s2 = 0; s2 < plan.slot_commit.size(); ++s2) {
    slot_commit[s2] = plan.slot_commit[s2];
    slot_t0[s2] = plan.slot_t0[s2];
  }
  *n_waves_out = (int32_t)plan.waves.size();
  *n_pulls_out = np;
  if (np > pull_cap) return fail(nullptr, AGN_E_INVALID, "pull buffer too short");
  return AGN_OK;
}

int agn_commit_pull(float* theta_c, float* acc, float* replicas, void* replicas_bf16, int64_t P,
                    int64_t ld, int32_t n, int32_t C, const int32_t* commit_worker,
                    const int32_t* pull_offsets, const int32_t* pull_workers, double eta,
                    int32_t lambda, int32_t normalize, float* delta_norm, void* stream) {
  Status s = commit_pull(theta_c, acc, replicas, replicas_bf16, P, ld, n, C, commit_worker,
                         pull_offsets, pull_workers, eta, lambda, normalize, delta_norm,
                         static_cast<cudaStream_t>(stream));
  return s.ok() ? AGN_OK : fail(nullptr, s);
}

int agn_debug_waits(agn_handle* h, int64_t wait_ns, int32_t withhold_rank) {
  if (!h) return fail(nullptr, AGN_E_INVALID, "null handle");
  if (wait_ns < 0 || wait_ns > 2000000000ll || withhold_rank < -1 || withhold_rank > 65534)
    return fail(h, AGN_E_INVALID, "wait_ns must be in [0, 2e9], withhold_rank >= -1");
  h->dbg_wait_ns = (uint64_t)wait_ns;
  h->dbg_withhold = withhold_rank + 1;
  return AGN_OK;
}

int agn_fill_commit_inputs(float* theta_c, float* acc, float* replicas, int64_t P, int64_t ld,
                           int32_t n, uint64_t seed, void* stream) {
  if (!theta_c || !acc || P < 1 || ld < P || n < 1)
    return fail(nullptr, AGN_E_INVALID, "bad arguments");
  Status s = agn::fill_commit_inputs(theta_c, acc, replicas, P, ld, n, seed,
                                     static_cast<cudaStream_t>(stream));
  return s.ok() ? AGN_OK : fail(nullptr, s);
}

}  // extern "C"

namespace agn {
// Message returned by agn_last_error(NULL) for entry points defined in other files.
void set_global_error(const std::string& msg) { g_error = msg; }
}  // namespace agn
