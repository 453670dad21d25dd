// Host float64 construction of the block transform; see transform_host.cpp.
#pragma once
#include <cstdint>
#include <string>

namespace cat {
// kind: 0 identity, 1 randomized Hadamard, 2 CAT (H_k M_b), 3 diagonal CAT (k = 1 optimum in k-blocks),
// 4 the M_b blocks of CAT with the full-size Hadamard (H_d applied separately).  Returns 0 on success,
// 1 if a block is not positive definite (message in *err).  Arrays are [d_in/k][k][k] row-major.
int build_transform_host(int kind, int64_t d_in, int k, const double* sigma_x_sums, int64_t n_calib,
                         const double* sigma_w, const float* rht_signs, double* T_out, double* Tinv_out,
                         std::string* err);
// Eq. 9: A_max from full d x d Sigma_x (positive definite) and Sigma_w; false if not computable.
bool alignment_ceiling_host(const double* sigma_x, const double* sigma_w, int64_t d, double* a_max, double* sum_mu,
                            double* sum_sqrt_mu);
}  // namespace cat
