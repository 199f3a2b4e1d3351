// Host generation of the seeded inputs: dataset, teacher labels, initial
// parameters and the round-robin schedule (the same definitions as the
// generator header; host code is compiled with -ffp-contract=off).
#include <thread>
#include <vector>

#include "../../include/agn.h"
#include "generator.cuh"
#include "host_inputs.h"

#include <algorithm>

namespace agn {

namespace {

template <typename F>
void parallel_for(int64_t n, F&& f) {
  unsigned hw = std::thread::hardware_concurrency();
  int nt = (int)std::max<int64_t>(1, std::min<int64_t>(hw ? hw : 4, (n + 4095) / 4096));
  if (nt == 1) {
    f(0, n);
    return;
  }
  std::vector<std::thread> th;
  const int64_t chunk = (n + nt - 1) / nt;
  for (int t = 0; t < nt; ++t) {
    const int64_t b = t * chunk, e = std::min(n, b + chunk);
    if (b < e) th.emplace_back([&f, b, e] { f(b, e); });
  }
  for (auto& x : th) x.join();
}

}  // namespace

void gen_dataset_rows(uint64_t seed, int d0, int64_t row0, int64_t n_rows, int dist, float* X) {
  const uint64_t k = gen::key(seed, gen::kData);
  const int64_t base = row0 * d0;
  parallel_for(n_rows * d0, [&](int64_t b, int64_t e) {
    for (int64_t i = b; i < e; ++i) {
      const uint64_t j = (uint64_t)(base + i);
      X[i] = dist == AGN_DIST_UNIFORM ? gen::uniform_f32(gen::draw(k, j)) : (float)gen::normal(k, j);
    }
  });
}

void gen_dataset(uint64_t seed, int d0, int64_t N, int dist, float* X) {
  gen_dataset_rows(seed, d0, 0, N, dist, X);
}

std::vector<std::vector<double>> gen_teacher(uint64_t seed, const std::vector<int>& tdims) {
  const uint64_t k = gen::key(seed, gen::kTeacher);
  std::vector<std::vector<double>> Ws;
  uint64_t off = 0;
  for (size_t l = 1; l < tdims.size(); ++l) {
    const int fi = tdims[l - 1], fo = tdims[l];
    std::vector<double> W((size_t)fo * fi);
    const double sd = gen::dsqrt(gen::ddiv(2.0, (double)fi));
    for (int64_t i = 0; i < (int64_t)W.size(); ++i)
      W[i] = gen::dmul(gen::normal(k, off + (uint64_t)i), sd);
    if (l > 1) {  // centre the rows of layers fed by ReLU outputs
      for (int o = 0; o < fo; ++o) {
        double s = 0.0;
        for (int i = 0; i < fi; ++i) s = gen::dadd(s, W[(size_t)o * fi + i]);
        const double mu = gen::ddiv(s, (double)fi);
        for (int i = 0; i < fi; ++i) W[(size_t)o * fi + i] = gen::dsub(W[(size_t)o * fi + i], mu);
      }
    }
    Ws.push_back(std::move(W));
    off += (uint64_t)fo * fi;
  }
  return Ws;
}

void gen_teacher_labels(const float* X, int64_t N, int d0, int dist,
                        const std::vector<int>& tdims, const std::vector<std::vector<double>>& Ws,
                        int32_t* y) {
  const double centre = dist == AGN_DIST_UNIFORM ? 0.5 : 0.0;
  int maxd = 0;
  for (int d : tdims) maxd = std::max(maxd, d);
  parallel_for(N, [&](int64_t b, int64_t e) {
    std::vector<double> h(maxd), z(maxd);
    for (int64_t r = b; r < e; ++r) {
      for (int c = 0; c < d0; ++c) h[c] = (double)X[r * d0 + c] - centre;
      for (size_t l = 1; l < tdims.size(); ++l) {
        const int fi = tdims[l - 1], fo = tdims[l];
        const double* W = Ws[l - 1].data();
        for (int o = 0; o < fo; ++o) {
          double s = 0.0;
          for (int i = 0; i < fi; ++i) s += W[(size_t)o * fi + i] * h[i];
          z[o] = (l + 1 < tdims.size() && s < 0.0) ? 0.0 : s;
        }
        for (int o = 0; o < fo; ++o) h[o] = z[o];
      }
      const int C = tdims.back();
      int best = 0;
      for (int c = 1; c < C; ++c)
        if (h[c] > h[best]) best = c;
      y[r] = best;
    }
  });
}

void gen_init(uint64_t seed, const std::vector<int>& dims, float* theta) {
  const uint64_t k = gen::key(seed, gen::kInit);
  int64_t off = 0;
  for (size_t l = 1; l < dims.size(); ++l) {
    const int fi = dims[l - 1], fo = dims[l];
    const double r = gen::dsqrt(gen::ddiv(6.0, (double)(fi + fo)));
    const int64_t nw = (int64_t)fo * fi;
    const int64_t base = off;
    parallel_for(nw, [&](int64_t b, int64_t e) {
      for (int64_t i = b; i < e; ++i) {
        const double u = gen::uniform_f64(gen::draw(k, (uint64_t)(base + i)));
        theta[base + i] = (float)gen::dmul(gen::dsub(gen::dmul(2.0, u), 1.0), r);
      }
    });
    for (int o = 0; o < fo; ++o) theta[base + nw + o] = 0.f;
    off += nw + fo;
  }
}

void gen_schedule(int n, int64_t C, int lo, int hi, uint64_t seed, int32_t* w, int32_t* tau) {
  const uint64_t k = gen::key(seed, gen::kSchedule);
  const uint64_t span = (uint64_t)(hi - lo + 1);
  std::vector<int64_t> prev(n, -1);
  for (int64_t c = 0; c < C; ++c) {
    const int wk = (int)(c % n);
    int64_t t = lo + (int64_t)gen::bounded(gen::draw(k, (uint64_t)c), span);
    t = std::min<int64_t>(t, c - prev[wk] - 1);
    w[c] = wk;
    tau[c] = (int32_t)t;
    prev[wk] = c;
  }
}

}  // namespace agn
