// Host generation of the seeded inputs (see generator.cuh for the definitions).
#pragma once

#include <cstdint>
#include <vector>

namespace agn {

// X [N][d0] fp32: U[0,1) (top 24 bits of draw r*d0+c) or N(0,1) (number r*d0+c).
void gen_dataset(uint64_t seed, int d0, int64_t N, int dist, float* X);
// Rows [row0, row0 + n_rows) of the same dataset.
void gen_dataset_rows(uint64_t seed, int d0, int64_t row0, int64_t n_rows, int dist, float* X);
// Teacher ReLU MLP weights (double), W_l ~ N(0, 2/fan_in), rows of layers > 1 centred.
std::vector<std::vector<double>> gen_teacher(uint64_t seed, const std::vector<int>& tdims);
// y = argmax of the teacher on X - centre (lowest index on ties), in double.
void gen_teacher_labels(const float* X, int64_t N, int d0, int dist,
                        const std::vector<int>& tdims, const std::vector<std::vector<double>>& Ws,
                        int32_t* y);
// Glorot-uniform weights, zero biases, flat order.
void gen_init(uint64_t seed, const std::vector<int>& dims, float* theta);
// Round-robin schedule with clamped uniform staleness.
void gen_schedule(int n, int64_t C, int lo, int hi, uint64_t seed, int32_t* w, int32_t* tau);

}  // namespace agn
