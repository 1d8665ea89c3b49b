// ORACLE -- test infrastructure, not part of the product.
//
// Gradients of the workers' model and the end-to-end asynchronous simulation that feeds
// them to GEM.  A worker computes dtheta = -eta grad L(s) at its snapshot s (notation
// table; Algorithm 1, procedure Worker).  The model is a fully connected ReLU network
// with a softmax cross-entropy loss averaged over the worker's minibatch; its
// parameters are one flat vector [W_1, b_1, W_2, b_2, ...] with W_l stored out x in,
// row-major.
//
// Precision: the gradient is computed in double from the fp32 snapshot and rounded once
// to fp32 for the commit.  With tf32 != 0 every operand of every matrix product is first
// rounded to TF32 (10 explicit mantissa bits, round to nearest, ties away from zero),
// the input precision of a TF32 tensor-core product; products and sums stay in double.
//
// The matrix products are plain loops.  An OpenMP "parallel for" over their output rows
// only splits independent outputs across threads: each output is still summed by one
// thread in index order, so the result does not depend on the thread count.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>
#ifdef _OPENMP
#include <omp.h>
#endif

extern "C" int oracle_gem_run_f32(int64_t P, int n, int T, const int32_t* order,
                                  const int32_t* tau, const float* grads,
                                  int64_t grad_stride, const int32_t* grad_index,
                                  float* theta, float* m, float* s, int64_t state_stride,
                                  double eta, double mu, double eps, int mode, double kappa,
                                  int precommit_snapshot, const int64_t* record_cols,
                                  int n_record, float* record);
extern "C" int oracle_gem_run_pi_f32(int64_t P, int n, int T, const int32_t* order,
                                     const int32_t* tau, const float* grads,
                                     int64_t grad_stride, const int32_t* grad_index,
                                     float* theta, float* m, float* s, int64_t state_stride,
                                     double eta, double mu, double eps, int mode, double kappa,
                                     int precommit_snapshot, float* pi_record);

namespace {

// Round an fp32 value to TF32: keep 10 explicit mantissa bits, round to nearest with
// ties away from zero (add half of the dropped range to the magnitude, then truncate).
float tf32_rna(float x) {
  uint32_t u;
  std::memcpy(&u, &x, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) return x;  // inf and NaN pass through
  u += 0x00001000u;
  u &= 0xFFFFE000u;
  std::memcpy(&x, &u, 4);
  return x;
}

inline double operand(double v, int tf32) {
  return tf32 ? double(tf32_rna(float(v))) : v;
}

struct Layer {
  int64_t w, b;  // offsets of W (out x in) and bias (out) in the flat vector
  int out, in;
};

std::vector<Layer> layout(int L, const int32_t* dims) {
  std::vector<Layer> lay(L);
  int64_t off = 0;
  for (int l = 0; l < L; ++l) {
    lay[l].in = dims[l];
    lay[l].out = dims[l + 1];
    lay[l].w = off;
    lay[l].b = off + int64_t(dims[l + 1]) * dims[l];
    off = lay[l].b + dims[l + 1];
  }
  return lay;
}

// Mean softmax cross-entropy over the b rows of X and its gradient with respect to the
// flat parameter vector.  X is [b][dims[0]], labels y in [0, dims[L]).
double loss_and_grad(int L, const int32_t* dims, const double* theta, const double* X,
                     const int32_t* y, int b, double* grad, int tf32) {
  const std::vector<Layer> lay = layout(L, dims);
  // a[l] is the input of layer l ([b][in]); z[l] its pre-activation ([b][out]).
  std::vector<std::vector<double>> a(L + 1), z(L);
  a[0].assign(X, X + int64_t(b) * dims[0]);
  for (int l = 0; l < L; ++l) {
    const Layer& ly = lay[l];
    z[l].assign(int64_t(b) * ly.out, 0.0);
    const double* W = theta + ly.w;
    const double* bias = theta + ly.b;
#pragma omp parallel for schedule(static)
    for (int i = 0; i < b; ++i)
      for (int o = 0; o < ly.out; ++o) {
        double acc = 0.0;
        for (int k = 0; k < ly.in; ++k)
          acc += operand(a[l][int64_t(i) * ly.in + k], tf32) *
                 operand(W[int64_t(o) * ly.in + k], tf32);
        z[l][int64_t(i) * ly.out + o] = acc + bias[o];
      }
    if (l + 1 < L) {
      a[l + 1].resize(z[l].size());
      for (size_t q = 0; q < z[l].size(); ++q) a[l + 1][q] = z[l][q] > 0.0 ? z[l][q] : 0.0;
    }
  }
  // Softmax cross-entropy: loss_i = log sum_c exp(z_ic) - z_{i, y_i}; the gradient of the
  // batch mean with respect to z is (softmax(z_i) - onehot(y_i)) / b.
  const int C = dims[L];
  std::vector<double> delta(int64_t(b) * C);
  double loss = 0.0;
  for (int i = 0; i < b; ++i) {
    const double* zi = &z[L - 1][int64_t(i) * C];
    double zmax = zi[0];
    for (int c = 1; c < C; ++c) zmax = zi[c] > zmax ? zi[c] : zmax;
    double sum = 0.0;
    for (int c = 0; c < C; ++c) sum += std::exp(zi[c] - zmax);
    loss += (std::log(sum) + zmax) - zi[y[i]];
    for (int c = 0; c < C; ++c) {
      const double p = std::exp(zi[c] - zmax) / sum;
      delta[int64_t(i) * C + c] = (p - (c == y[i] ? 1.0 : 0.0)) / double(b);
    }
  }
  loss /= double(b);
  // Backward pass, last layer first.
  for (int l = L - 1; l >= 0; --l) {
    const Layer& ly = lay[l];
    const double* W = theta + ly.w;
    double* dW = grad + ly.w;
    double* db = grad + ly.b;
#pragma omp parallel for schedule(static)
    for (int o = 0; o < ly.out; ++o) {
      for (int k = 0; k < ly.in; ++k) {
        double acc = 0.0;
        for (int i = 0; i < b; ++i)
          acc += operand(delta[int64_t(i) * ly.out + o], tf32) *
                 operand(a[l][int64_t(i) * ly.in + k], tf32);
        dW[int64_t(o) * ly.in + k] = acc;
      }
      double acc = 0.0;
      for (int i = 0; i < b; ++i) acc += delta[int64_t(i) * ly.out + o];
      db[o] = acc;
    }
    if (l == 0) break;
    // delta of the previous layer: (delta W) masked by the ReLU derivative.
    std::vector<double> prev(int64_t(b) * ly.in);
#pragma omp parallel for schedule(static)
    for (int i = 0; i < b; ++i)
      for (int k = 0; k < ly.in; ++k) {
        double acc = 0.0;
        for (int o = 0; o < ly.out; ++o)
          acc += operand(delta[int64_t(i) * ly.out + o], tf32) *
                 operand(W[int64_t(o) * ly.in + k], tf32);
        prev[int64_t(i) * ly.in + k] = z[l - 1][int64_t(i) * ly.in + k] > 0.0 ? acc : 0.0;
      }
    delta.swap(prev);
  }
  return loss;
}

int64_t param_count(int L, const int32_t* dims) {
  int64_t P = 0;
  for (int l = 0; l < L; ++l) P += int64_t(dims[l + 1]) * dims[l] + dims[l + 1];
  return P;
}

}  // namespace

extern "C" {

float oracle_tf32_rna(float x) { return tf32_rna(x); }

int oracle_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

// Mean loss and gradient in double.  theta [P], X [b][dims[0]], y [b], grad [P].
double oracle_mlp_loss_grad_f64(int L, const int32_t* dims, const double* theta,
                                const double* X, const int32_t* y, int b, double* grad,
                                int tf32) {
  return loss_and_grad(L, dims, theta, X, y, b, grad, tf32);
}

// End-to-end simulation: for t = 0..T-1, worker w = order[t] computes the gradient of
// the mean loss over rows batch_rows[t][0..b) of X at its snapshot s_w (double, then
// rounded to fp32) and commits it with GEM (oracle_gem_run_f32, one commit).
// theta [P], m and s [n][state_stride] fp32 are updated in place.  X [x_rows][dims[0]],
// labels [x_rows].  After commit t = record_at[r] theta is copied to record[r][0..P).
// losses[t] (optional) receives the minibatch loss of commit t.
int oracle_mlp_sim_run_pi(int L, const int32_t* dims, int n, int T, const int32_t* order,
                          const int32_t* tau, const float* X, int64_t x_rows,
                          const int32_t* labels, const int32_t* batch_rows, int b,
                          float* theta, float* m, float* s, int64_t state_stride, double eta,
                          double mu, double eps, int mode, double kappa, int tf32,
                          int n_record, const int32_t* record_at, float* record,
                          double* losses, float* pi_record);

int oracle_mlp_sim_run(int L, const int32_t* dims, int n, int T, const int32_t* order,
                       const int32_t* tau, const float* X, int64_t x_rows,
                       const int32_t* labels, const int32_t* batch_rows, int b,
                       float* theta, float* m, float* s, int64_t state_stride, double eta,
                       double mu, double eps, int mode, double kappa, int tf32,
                       int n_record, const int32_t* record_at, float* record,
                       double* losses) {
  return oracle_mlp_sim_run_pi(L, dims, n, T, order, tau, X, x_rows, labels, batch_rows, b,
                               theta, m, s, state_stride, eta, mu, eps, mode, kappa, tf32,
                               n_record, record_at, record, losses, nullptr);
}

// As oracle_mlp_sim_run; when pi_record is not NULL, the scaling factors of commit t are
// written to pi_record[t][0..P).
int oracle_mlp_sim_run_pi(int L, const int32_t* dims, int n, int T, const int32_t* order,
                          const int32_t* tau, const float* X, int64_t x_rows,
                          const int32_t* labels, const int32_t* batch_rows, int b,
                          float* theta, float* m, float* s, int64_t state_stride, double eta,
                          double mu, double eps, int mode, double kappa, int tf32,
                          int n_record, const int32_t* record_at, float* record,
                          double* losses, float* pi_record) {
  if (L < 1 || n < 1 || T < 0 || b < 1 || !order || !X || !labels || !batch_rows) return -1;
  const int64_t P = param_count(L, dims);
  if (state_stride < P) return -1;
  const int d0 = dims[0];
  std::vector<double> params(P), grad(P), xb(int64_t(b) * d0);
  std::vector<float> g32(P);
  std::vector<int32_t> yb(b);
  int r = 0;
  for (int t = 0; t < T; ++t) {
    const int w = order[t];
    if (w < 0 || w >= n) return -1;
    const float* sw = s + int64_t(w) * state_stride;
    for (int64_t j = 0; j < P; ++j) params[j] = double(sw[j]);
    for (int i = 0; i < b; ++i) {
      const int64_t row = batch_rows[int64_t(t) * b + i];
      if (row < 0 || row >= x_rows) return -1;
      for (int k = 0; k < d0; ++k) xb[int64_t(i) * d0 + k] = double(X[row * d0 + k]);
      yb[i] = labels[row];
    }
    const double loss = loss_and_grad(L, dims, params.data(), xb.data(), yb.data(), b,
                                      grad.data(), tf32);
    if (losses) losses[t] = loss;
    for (int64_t j = 0; j < P; ++j) g32[j] = float(grad[j]);
    const int32_t one_w = w;
    const int32_t one_tau = tau ? tau[t] : 0;
    const int rc = oracle_gem_run_pi_f32(P, n, 1, &one_w, &one_tau, g32.data(), P, nullptr,
                                         theta, m, s, state_stride, eta, mu, eps, mode, kappa,
                                         0, pi_record ? pi_record + int64_t(t) * P : nullptr);
    if (rc) return rc;
    while (record && r < n_record && record_at[r] == t) {
      std::memcpy(record + int64_t(r) * P, theta, size_t(P) * sizeof(float));
      ++r;
    }
  }
  return 0;
}

}  // extern "C"
