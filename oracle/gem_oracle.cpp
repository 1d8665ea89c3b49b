// ORACLE -- test infrastructure, not part of the product.
//
// A plain, slow restatement of Gradient Energy Matching (Hermans & Louppe, "Gradient
// Energy Matching for Distributed Asynchronous Gradient Descent", arXiv 1805.08469).  Only
// the tests, the smoke check and the CPU-baseline leg of the benchmark may load it.  It
// shares no source, header or constant with the CUDA path.
//
// It runs on one thread unless oracle_set_commit_threads asks for more.  Then the
// coordinates of each commit are split across threads: every step of Psi_GEM and of the
// update is elementwise (Algorithm 1 uses the elementwise product), so coordinate j's
// result depends only on element j of each input, and the split changes no result.
//
// Build with -O2 -ffp-contract=off: every floating-point operation below is one IEEE
// operation with its own rounding (no fused multiply-add), in the precision of T.
//
// Readings taken where the paper is silent or loose (each one is listed with its reason
// in the design notes of the repository):
//   * the snapshot a worker computes its next gradient at is the central variable right
//     after its own commit (s <- theta after Commit, Algorithm 1); the literal "pulled
//     before the commit" reading is available as a contrast flag only;
//   * the scaling factor is clamped at zero: pi = max(0, .);
//   * the moment accumulates the raw update Delta-theta (Algorithm 1, Psi_GEM), not the
//     scaled one;
//   * |.| is the elementwise absolute value (notation table) and sqrt(2) sqrt(E_k)
//     equals |m| by Eq. proxy_estimate, so no square root is taken;
//   * fp32 state and arithmetic for the commit (the paper's implementation is PyTorch
//     with its default fp32 tensors); a double instantiation serves the pins.
#include <cmath>
#include <cstdint>
#include <cstring>
#ifdef _OPENMP
#include <omp.h>
#endif

namespace {

int g_commit_threads = 1;  // threads over the coordinates of one commit

// Commit modes.  GEM is Algorithm 1; the others are the comparison rules of the
// experiments section and the high-energy proxies of Appendix B.
enum Mode : int {
  MODE_GEM = 0,            // Algorithm 1: pi = (|m| - |theta - s|) / (|dtheta| + eps)
  MODE_DOWNPOUR = 1,       // commit dtheta unscaled (pi = 1)
  MODE_ADAPTIVE = 2,       // commit dtheta / (tau + 1)
  MODE_KAPPA_SQRT = 3,     // App. B, Eq. pi_with_kappa: sqrt(kappa) |m|
  MODE_KAPPA_LINEAR = 4,   // App. B, the modified form used in that study: kappa |m|
  MODE_MOMENTUM = 5,       // the proxy itself, Eq. momentum_update: theta += (m <- mu m + dtheta)
};

// One worker's commit on one coordinate (Algorithm 1, procedures Worker and Psi_GEM,
// followed by the master's update of Eq. update_psi).  Returns the scaling factor pi the
// commit applied to this coordinate (the per-parameter value whose median the experiments
// section reports).
template <typename T>
inline T commit_coordinate(T& theta, T& m, T& s, T g, T eta, T mu, T eps, int mode,
                              T kappa, int tau, int precommit_snapshot) {
  // Worker: the update is plain SGD on the snapshot, dtheta = -eta * grad L(s).
  const T dtheta = -(eta * g);
  // theta <- Pull(): the value of the central variable the commit is applied to.
  const T theta_pulled = theta;
  T pi;
  if (mode == MODE_MOMENTUM) {
    // The target dynamics of the proxy (sequential momentum SGD with the worker's moment):
    // the commit adds the moment itself; no scaling factor is formed (NaN is recorded).
    m = mu * m + dtheta;
    theta = theta_pulled + m;
    s = precommit_snapshot ? theta_pulled : theta;
    return T(NAN);
  }
  if (mode == MODE_DOWNPOUR) {
    pi = T(1);
  } else if (mode == MODE_ADAPTIVE) {
    pi = T(1) / (T(tau) + T(1));
  } else {
    // Psi_GEM, first step: m <- mu m + dtheta (Eq. moment_estimate, local first moment).
    m = mu * m + dtheta;
    // sqrt(2) sqrt(E_k(t+1)) with the proxy energy of Eq. proxy_estimate is |m|.
    T energy_root = std::fabs(m);
    if (mode == MODE_KAPPA_SQRT) energy_root = std::sqrt(kappa) * energy_root;
    if (mode == MODE_KAPPA_LINEAR) energy_root = kappa * energy_root;
    // Psi_GEM, second step (Eq. new_pi with eps added to |dtheta|): the factor that
    // matches the central variable's energy 1/2 (theta - s + pi dtheta)^2 to the proxy.
    const T drift = std::fabs(theta_pulled - s);
    pi = (energy_root - drift) / (std::fabs(dtheta) + eps);
    if (!(pi > T(0))) pi = T(0);
  }
  // Commit(pi (.) dtheta): theta_{t+1} = theta_t + Psi(dtheta_t) (Eq. update_psi).
  theta = theta_pulled + pi * dtheta;
  // s <- theta: the worker's next gradient is taken at the post-commit central variable.
  s = precommit_snapshot ? theta_pulled : theta;
  return pi;
}

template <typename T>
int run(int64_t P, int n, int T_commits, const int32_t* order, const int32_t* tau,
        const T* grads, int64_t grad_stride, const int32_t* grad_index, T* theta, T* m,
        T* s, int64_t state_stride, double eta_d, double mu_d, double eps_d, int mode,
        double kappa_d, int precommit_snapshot, const int64_t* record_cols, int n_record,
        T* record, T* pi_record) {
  if (P < 0 || n < 1 || T_commits < 0 || !order || !grads || !theta || !m || !s) return -1;
  if (state_stride < P) return -1;
  const T eta = T(eta_d), mu = T(mu_d), eps = T(eps_d), kappa = T(kappa_d);
  for (int t = 0; t < T_commits; ++t) {
    const int w = order[t];
    if (w < 0 || w >= n) return -1;
    const int64_t row = grad_index ? grad_index[t] : t;
    const T* g = grads + row * grad_stride;
    T* mw = m + int64_t(w) * state_stride;
    T* sw = s + int64_t(w) * state_stride;
    const int tw = tau ? tau[t] : 0;
    T* pi_row = pi_record ? pi_record + int64_t(t) * P : nullptr;
#pragma omp parallel for schedule(static) num_threads(g_commit_threads) if (g_commit_threads > 1)
    for (int64_t j = 0; j < P; ++j) {
      const T pi = commit_coordinate<T>(theta[j], mw[j], sw[j], g[j], eta, mu, eps, mode, kappa,
                                        tw, precommit_snapshot);
      if (pi_row) pi_row[j] = pi;
    }
    if (record && n_record > 0)
      for (int r = 0; r < n_record; ++r) record[int64_t(t) * n_record + r] = theta[record_cols[r]];
  }
  return 0;
}

}  // namespace

extern "C" {

// Threads that split the coordinates of each commit (1, the default, runs the loop on the
// calling thread; values below 1 are taken as 1).  Returns the previous value.
int oracle_set_commit_threads(int threads) {
  const int prev = g_commit_threads;
  g_commit_threads = threads < 1 ? 1 : threads;
  return prev;
}

// Apply T_commits commits in schedule order.  Commit t is made by worker order[t] with
// the gradient row grads[grad_index[t] * grad_stride .. + P) (row t when grad_index is
// NULL).  theta [P], m and s [n][state_stride] are updated in place.  When record is not
// NULL, theta at the n_record columns record_cols is written after every commit into
// record[t][r].  Returns 0, or -1 on an invalid argument.
int oracle_gem_run_f32(int64_t P, int n, int T, const int32_t* order, const int32_t* tau,
                       const float* grads, int64_t grad_stride, const int32_t* grad_index,
                       float* theta, float* m, float* s, int64_t state_stride, double eta,
                       double mu, double eps, int mode, double kappa,
                       int precommit_snapshot, const int64_t* record_cols, int n_record,
                       float* record) {
  return run<float>(P, n, T, order, tau, grads, grad_stride, grad_index, theta, m, s,
                    state_stride, eta, mu, eps, mode, kappa, precommit_snapshot,
                    record_cols, n_record, record, nullptr);
}

int oracle_gem_run_f64(int64_t P, int n, int T, const int32_t* order, const int32_t* tau,
                       const double* grads, int64_t grad_stride, const int32_t* grad_index,
                       double* theta, double* m, double* s, int64_t state_stride,
                       double eta, double mu, double eps, int mode, double kappa,
                       int precommit_snapshot, const int64_t* record_cols, int n_record,
                       double* record) {
  return run<double>(P, n, T, order, tau, grads, grad_stride, grad_index, theta, m, s,
                     state_stride, eta, mu, eps, mode, kappa, precommit_snapshot,
                     record_cols, n_record, record, nullptr);
}

// As oracle_gem_run_f32 / _f64, and when pi_record is not NULL the scaling factor pi of
// every coordinate of commit t is written to pi_record[t][0..P).
int oracle_gem_run_pi_f32(int64_t P, int n, int T, const int32_t* order, const int32_t* tau,
                          const float* grads, int64_t grad_stride, const int32_t* grad_index,
                          float* theta, float* m, float* s, int64_t state_stride, double eta,
                          double mu, double eps, int mode, double kappa,
                          int precommit_snapshot, float* pi_record) {
  return run<float>(P, n, T, order, tau, grads, grad_stride, grad_index, theta, m, s,
                    state_stride, eta, mu, eps, mode, kappa, precommit_snapshot, nullptr, 0,
                    nullptr, pi_record);
}

int oracle_gem_run_pi_f64(int64_t P, int n, int T, const int32_t* order, const int32_t* tau,
                          const double* grads, int64_t grad_stride, const int32_t* grad_index,
                          double* theta, double* m, double* s, int64_t state_stride,
                          double eta, double mu, double eps, int mode, double kappa,
                          int precommit_snapshot, double* pi_record) {
  return run<double>(P, n, T, order, tau, grads, grad_stride, grad_index, theta, m, s,
                     state_stride, eta, mu, eps, mode, kappa, precommit_snapshot, nullptr, 0,
                     nullptr, pi_record);
}

}  // extern "C"
