// Host float64 construction of the block transform; see transform_host.cpp.
#pragma once
#include <cstdint>
#include <string>

namespace cat {
// kind: 0 identity, 1 randomized Hadamard, 2 CAT.  Returns 0 on success, 1 if a block is not
// positive definite (message in *err).  Arrays are [d_in/k][k][k] row-major.
int build_transform_host(int kind, int64_t d_in, int k, const double* sigma_x_sums, int64_t n_calib,
                         const double* sigma_w, const float* rht_signs, double* T_out, double* Tinv_out,
                         std::string* err);
}  // namespace cat
