// Host (float64) construction of the block transform (Sec. 4, Eq. 7 and Eq. 10).
//
// For every k x k block b:
//   Sigma_x_b = (calibration sums) / n_calib,  Sigma_w_b = (W_b^T W_b)
//   G_b = Sigma_w_b # Sigma_x_b^{-1}                (matrix geometric mean, Eq. 7)
//       = Sigma_x_b^{-1/2} (Sigma_x_b^{1/2} Sigma_w_b Sigma_x_b^{1/2})^{1/2} Sigma_x_b^{-1/2}
//         (the mean is symmetric in its arguments, so it can be expanded around Sigma_x^{-1})
//   M_b = G_b^{1/2},  M_b^{-1} = G_b^{-1/2}
//   T_b = H_k M_b,    T_b^{-1} = M_b^{-1} H_k^T      (Eq. 10; H_k orthonormal Sylvester Hadamard)
// Randomized Hadamard: T_b = H_k Diag(sigma_b), T_b^{-1} = Diag(sigma_b) H_k^T.  Identity: T_b = I.
//
// Symmetric matrix functions come from a cyclic Jacobi eigen-decomposition written here; blocks
// are independent and are processed in parallel on host threads.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <string>
#include <thread>
#include <vector>

#include "transform_host.h"

namespace cat {
namespace {

// Eigen-decomposition of a symmetric k x k matrix (row-major, destroyed): A = V diag(w) V^T,
// eigenvectors in the columns of V.  Cyclic Jacobi rotations until the off-diagonal mass is
// below 1e-30 of the diagonal mass (or 60 sweeps).
void jacobi_eig(std::vector<double>& A, int k, std::vector<double>& w, std::vector<double>& V) {
  V.assign((size_t)k * k, 0.0);
  for (int i = 0; i < k; ++i) V[(size_t)i * k + i] = 1.0;
  auto a = [&](int r, int c) -> double& { return A[(size_t)r * k + c]; };
  auto v = [&](int r, int c) -> double& { return V[(size_t)r * k + c]; };
  for (int sweep = 0; sweep < 60; ++sweep) {
    double off = 0.0, dia = 0.0;
    for (int p = 0; p < k; ++p) {
      dia += a(p, p) * a(p, p);
      for (int q = p + 1; q < k; ++q) off += a(p, q) * a(p, q);
    }
    if (off <= 1e-30 * dia || off == 0.0) break;
    for (int p = 0; p < k - 1; ++p) {
      for (int q = p + 1; q < k; ++q) {
        const double apq = a(p, q);
        if (apq == 0.0) continue;
        const double app = a(p, p), aqq = a(q, q);
        if (std::fabs(apq) < 1e-18 * std::sqrt(std::fabs(app * aqq))) {
          a(p, q) = a(q, p) = 0.0;
          continue;
        }
        const double theta = (aqq - app) / (2.0 * apq);
        const double t = (theta >= 0.0 ? 1.0 : -1.0) / (std::fabs(theta) + std::sqrt(theta * theta + 1.0));
        const double c = 1.0 / std::sqrt(t * t + 1.0), s = t * c;
        for (int r = 0; r < k; ++r) {  // A <- A J
          const double arp = a(r, p), arq = a(r, q);
          a(r, p) = c * arp - s * arq;
          a(r, q) = s * arp + c * arq;
        }
        for (int r = 0; r < k; ++r) {  // A <- J^T A
          const double apr = a(p, r), aqr = a(q, r);
          a(p, r) = c * apr - s * aqr;
          a(q, r) = s * apr + c * aqr;
        }
        a(p, q) = a(q, p) = 0.0;
        for (int r = 0; r < k; ++r) {  // V <- V J
          const double vrp = v(r, p), vrq = v(r, q);
          v(r, p) = c * vrp - s * vrq;
          v(r, q) = s * vrp + c * vrq;
        }
      }
    }
  }
  w.resize(k);
  for (int i = 0; i < k; ++i) w[i] = a(i, i);
}

// out = V diag(f) V^T
void compose(const std::vector<double>& V, const std::vector<double>& f, int k, std::vector<double>& out) {
  out.assign((size_t)k * k, 0.0);
  for (int i = 0; i < k; ++i)
    for (int j = i; j < k; ++j) {
      double s = 0.0;
      for (int e = 0; e < k; ++e) s += V[(size_t)i * k + e] * f[e] * V[(size_t)j * k + e];
      out[(size_t)i * k + j] = out[(size_t)j * k + i] = s;
    }
}

// Powers p1 and p2 of a symmetric positive definite matrix.  Returns false if not SPD.
bool spd_powers(const std::vector<double>& S, int k, double p1, std::vector<double>& out1, double p2,
                std::vector<double>& out2) {
  std::vector<double> A(S.size()), w, V;
  for (int i = 0; i < k; ++i)
    for (int j = 0; j < k; ++j) A[(size_t)i * k + j] = 0.5 * (S[(size_t)i * k + j] + S[(size_t)j * k + i]);
  jacobi_eig(A, k, w, V);
  const double wmax = *std::max_element(w.begin(), w.end());
  const double wmin = *std::min_element(w.begin(), w.end());
  if (!(wmax > 0.0) || !(wmin > 1e-13 * wmax) || !std::isfinite(wmax)) return false;
  std::vector<double> f(k);
  for (int i = 0; i < k; ++i) f[i] = std::pow(w[i], p1);
  compose(V, f, k, out1);
  for (int i = 0; i < k; ++i) f[i] = std::pow(w[i], p2);
  compose(V, f, k, out2);
  return true;
}

void matmul(const std::vector<double>& A, const std::vector<double>& B, int k, std::vector<double>& C) {
  C.assign((size_t)k * k, 0.0);
  for (int i = 0; i < k; ++i)
    for (int e = 0; e < k; ++e) {
      const double aie = A[(size_t)i * k + e];
      if (aie == 0.0) continue;
      for (int j = 0; j < k; ++j) C[(size_t)i * k + j] += aie * B[(size_t)e * k + j];
    }
}

double hadamard_entry(int i, int j, double inv_sqrt_k) {
  return (__builtin_popcount((unsigned)(i & j)) & 1) ? -inv_sqrt_k : inv_sqrt_k;
}

// One CAT block: T = H M, Tinv = M^{-1} H^T (with_h), or T = M, Tinv = M^{-1} (the full-size
// Hadamard variant, whose H_d is applied across all blocks afterwards).  Returns false if a block is
// not positive definite.
bool cat_block(const double* sx_sum, double inv_n, const double* sw, int k, double* T, double* Ti, bool with_h = true) {
  const size_t kk = (size_t)k * k;
  std::vector<double> Sx(kk), Sw(sw, sw + kk);
  for (size_t e = 0; e < kk; ++e) Sx[e] = sx_sum[e] * inv_n;
  std::vector<double> Sxh, Sxih;   // Sigma_x^{1/2}, Sigma_x^{-1/2}
  if (!spd_powers(Sx, k, 0.5, Sxh, -0.5, Sxih)) return false;
  std::vector<double> tmp, C;
  matmul(Sxh, Sw, k, tmp);
  matmul(tmp, Sxh, k, C);          // Sigma_x^{1/2} Sigma_w Sigma_x^{1/2}
  std::vector<double> Ch, unused;
  if (!spd_powers(C, k, 0.5, Ch, 1.0, unused)) return false;
  std::vector<double> G;
  matmul(Sxih, Ch, k, tmp);
  matmul(tmp, Sxih, k, G);         // G = Sigma_w # Sigma_x^{-1}
  std::vector<double> M, Mi;
  if (!spd_powers(G, k, 0.5, M, -0.5, Mi)) return false;
  if (!with_h) {
    std::copy(M.begin(), M.end(), T);
    std::copy(Mi.begin(), Mi.end(), Ti);
    return true;
  }
  const double h = 1.0 / std::sqrt((double)k);
  for (int i = 0; i < k; ++i)
    for (int j = 0; j < k; ++j) {
      double t = 0.0, ti = 0.0;
      for (int e = 0; e < k; ++e) {
        t += hadamard_entry(i, e, h) * M[(size_t)e * k + j];       // (H M)_{ij}
        ti += Mi[(size_t)i * k + e] * hadamard_entry(j, e, h);     // (M^{-1} H^T)_{ij}
      }
      T[(size_t)i * k + j] = t;
      Ti[(size_t)i * k + j] = ti;
    }
  return true;
}

// The k = 1 optimum (end of Sec. 4): m_i = (Sigma_w_ii / Sigma_x_ii)^{1/4}, from the diagonals of the
// k x k blocks.  Returns false for a non-positive diagonal entry.
bool diag_block(const double* sx_sum, double inv_n, const double* sw, int k, double* T, double* Ti) {
  for (int i = 0; i < k; ++i) {
    const double sx = sx_sum[(size_t)i * k + i] * inv_n, swi = sw[(size_t)i * k + i];
    if (!(sx > 0.0) || !(swi > 0.0) || !std::isfinite(sx) || !std::isfinite(swi)) return false;
    const double m = std::pow(swi / sx, 0.25);
    for (int j = 0; j < k; ++j) {
      T[(size_t)i * k + j] = i == j ? m : 0.0;
      Ti[(size_t)i * k + j] = i == j ? 1.0 / m : 0.0;
    }
  }
  return true;
}

}  // namespace

int build_transform_host(int kind, int64_t d_in, int k, const double* sigma_x, int64_t n_calib, const double* sigma_w,
                         const float* rht_signs, double* T_out, double* Tinv_out, std::string* err) {
  const int64_t nb = d_in / k;
  const size_t kk = (size_t)k * k;
  const double h = 1.0 / std::sqrt((double)k);
  if (kind == 0 || kind == 1) {
    for (int64_t b = 0; b < nb; ++b) {
      double* T = T_out + b * kk;
      double* Ti = Tinv_out + b * kk;
      for (int i = 0; i < k; ++i)
        for (int j = 0; j < k; ++j) {
          if (kind == 0) {
            T[(size_t)i * k + j] = Ti[(size_t)i * k + j] = (i == j) ? 1.0 : 0.0;
          } else {
            const double si = rht_signs[b * k + i], sj = rht_signs[b * k + j];
            T[(size_t)i * k + j] = hadamard_entry(i, j, h) * sj;    // H Diag(sigma)
            Ti[(size_t)i * k + j] = si * hadamard_entry(j, i, h);   // Diag(sigma) H^T
          }
        }
    }
    return 0;
  }
  // CAT: independent blocks on a pool of host threads.
  const double inv_n = 1.0 / (double)n_calib;
  std::atomic<int64_t> next(0);
  std::atomic<int64_t> bad(-1);
  auto worker = [&]() {
    for (;;) {
      const int64_t b = next.fetch_add(1);
      if (b >= nb) return;
      const bool good = kind == 3 ? diag_block(sigma_x + b * kk, inv_n, sigma_w + b * kk, k, T_out + b * kk, Tinv_out + b * kk)
                                  : cat_block(sigma_x + b * kk, inv_n, sigma_w + b * kk, k, T_out + b * kk,
                                              Tinv_out + b * kk, kind != 4);
      if (!good) {
        int64_t expected = -1;
        bad.compare_exchange_strong(expected, b);
      }
    }
  };
  unsigned hw = std::thread::hardware_concurrency();
  int64_t nthreads = std::min<int64_t>(nb, std::max(1u, std::min(hw, 64u)));
  std::vector<std::thread> pool;
  for (int64_t i = 1; i < nthreads; ++i) pool.emplace_back(worker);
  worker();
  for (auto& th : pool) th.join();
  if (bad.load() >= 0) {
    if (err) *err = "calibration or weight autocorrelation block " + std::to_string(bad.load()) + " is not positive definite";
    return 1;
  }
  return 0;
}

// A_max = Tr(P) / Tr(P^{1/2})^2, P = Sigma_x^{1/2} Sigma_w Sigma_x^{1/2} (Eq. 9, R11): the eigenvalues mu of
// P are those of W Sigma_x W^T.  Full d x d matrices; Sigma_x must be positive definite, Sigma_w
// positive semi-definite.  Returns false if not.
bool alignment_ceiling_host(const double* sigma_x, const double* sigma_w, int64_t d, double* a_max, double* sum_mu,
                            double* sum_sqrt_mu) {
  const int k = (int)d;
  std::vector<double> Sx(sigma_x, sigma_x + (size_t)k * k), Sw(sigma_w, sigma_w + (size_t)k * k);
  std::vector<double> Sxh, unused;
  if (!spd_powers(Sx, k, 0.5, Sxh, 1.0, unused)) return false;
  std::vector<double> tmp, P;
  matmul(Sxh, Sw, k, tmp);
  matmul(tmp, Sxh, k, P);
  std::vector<double> A((size_t)k * k), w, V;
  for (int i = 0; i < k; ++i)
    for (int j = 0; j < k; ++j) A[(size_t)i * k + j] = 0.5 * (P[(size_t)i * k + j] + P[(size_t)j * k + i]);
  jacobi_eig(A, k, w, V);
  double s = 0.0, r = 0.0;
  for (double m : w) {
    const double mu = m > 0.0 ? m : 0.0;   // rounding can leave tiny negative eigenvalues of a PSD P
    s += mu;
    r += std::sqrt(mu);
  }
  if (!(r > 0.0)) return false;
  *a_max = s / (r * r);
  if (sum_mu) *sum_mu = s;
  if (sum_sqrt_mu) *sum_sqrt_mu = r;
  return true;
}

}  // namespace cat
