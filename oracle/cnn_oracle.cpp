// ORACLE -- test infrastructure, not part of the product.
//
// The convolutional network of the MNIST experiments (Appendix A) as the workers' model,
// and the asynchronous simulation that feeds its gradients to GEM.  Plain loops in double,
// in the order the appendix lists the layers:
//
//   conv1: c1 output channels from 1 input channel, 5 x 5 kernel, no padding, stride 1
//   2 x 2 max-pooling (stride 2), then ReLU
//   conv2: c2 output channels from c1, 5 x 5, no padding, stride 1
//   dropout on the last convolutional layer: channel i of sample r is multiplied by the
//       given scale drop[r][i] (0 for a dropped channel, 1 / (1 - p) for a kept one)
//   2 x 2 max-pooling, then ReLU; flattened in (channel, row, column) order
//   three fully connected layers (f1, f2, C outputs), ReLU after the first two
//   log-softmax and the mean negative log-likelihood over the minibatch
//
// Max-pooling takes the first maximum of its window in the order (0,0), (0,1), (1,0),
// (1,1); its gradient goes to that element.  ReLU's gradient is 1 where its input is > 0.
//
// Parameters are one flat vector in the order conv1.W [c1][1][5][5], conv1.b [c1],
// conv2.W [c2][c1][5][5], conv2.b [c2], fc1.W [f1][F], fc1.b [f1], fc2.W [f2][f1], fc2.b,
// fc3.W [C][f2], fc3.b, with F = c2 * P2 * P2 the flattened feature count.
//
// shape = {H, c1, c2, f1, f2, C}: H x H inputs with H - 4 even and (H - 4) / 2 - 4 even
// and positive (H = 28: 24 -> 12 -> 8 -> 4, F = 16 c2).
#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

extern "C" int oracle_gem_run_pi_f32(int64_t P, int n, int T, const int32_t* order,
                                     const int32_t* tau, const float* grads,
                                     int64_t grad_stride, const int32_t* grad_index,
                                     float* theta, float* m, float* s, int64_t state_stride,
                                     double eta, double mu, double eps, int mode, double kappa,
                                     int precommit_snapshot, float* pi_record);

namespace {

constexpr int kK = 5;  // kernel side

struct Net {
  int H, c1, c2, f1, f2, C;
  int H1, P1, H2, P2, F;  // conv1 side, pool1 side, conv2 side, pool2 side, features
  int64_t w1, b1, w2, b2, wf1, bf1, wf2, bf2, wf3, bf3, P;
};

bool make_net(const int32_t* shape, Net& n) {
  n.H = shape[0];
  n.c1 = shape[1];
  n.c2 = shape[2];
  n.f1 = shape[3];
  n.f2 = shape[4];
  n.C = shape[5];
  if (n.H < 5 || n.c1 < 1 || n.c2 < 1 || n.f1 < 1 || n.f2 < 1 || n.C < 2) return false;
  n.H1 = n.H - (kK - 1);
  if (n.H1 % 2) return false;
  n.P1 = n.H1 / 2;
  n.H2 = n.P1 - (kK - 1);
  if (n.H2 < 2 || n.H2 % 2) return false;
  n.P2 = n.H2 / 2;
  n.F = n.c2 * n.P2 * n.P2;
  int64_t off = 0;
  auto take = [&](int64_t count) {
    const int64_t o = off;
    off += count;
    return o;
  };
  n.w1 = take(int64_t(n.c1) * kK * kK);
  n.b1 = take(n.c1);
  n.w2 = take(int64_t(n.c2) * n.c1 * kK * kK);
  n.b2 = take(n.c2);
  n.wf1 = take(int64_t(n.f1) * n.F);
  n.bf1 = take(n.f1);
  n.wf2 = take(int64_t(n.f2) * n.f1);
  n.bf2 = take(n.f2);
  n.wf3 = take(int64_t(n.C) * n.f2);
  n.bf3 = take(n.C);
  n.P = off;
  return true;
}

// First maximum of the 2 x 2 window at (2py, 2px) of an s x s map; returns its flat index.
int argmax2x2(const double* map, int s, int py, int px) {
  int best = (2 * py) * s + 2 * px;
  const int cand[3] = {(2 * py) * s + 2 * px + 1, (2 * py + 1) * s + 2 * px,
                       (2 * py + 1) * s + 2 * px + 1};
  for (int q = 0; q < 3; ++q)
    if (map[cand[q]] > map[best]) best = cand[q];
  return best;
}

// Forward and backward for one minibatch; returns the mean loss and, when grad is not
// null, writes the gradient of the mean loss with respect to theta.  logits (optional)
// receives [b][C].
double cnn_loss_grad(const Net& n, const double* th, const double* X, const int32_t* y,
                     const double* drop, int b, double* grad, double* logits) {
  const int H = n.H, H1 = n.H1, P1 = n.P1, H2 = n.H2, P2 = n.P2, F = n.F;
  if (grad) std::memset(grad, 0, sizeof(double) * size_t(n.P));
  double loss = 0.0;
  // per-sample buffers
  std::vector<double> z1(size_t(n.c1) * H1 * H1), a1(size_t(n.c1) * P1 * P1);
  std::vector<double> z2(size_t(n.c2) * H2 * H2), a2(F);
  std::vector<double> h1(n.f1), h2(n.f2), zo(n.C);
  std::vector<double> dzo(n.C), dh2(n.f2), dh1(n.f1), da2(F), dz2(z2.size()), da1(a1.size()),
      dz1(z1.size());
  for (int r = 0; r < b; ++r) {
    const double* x = X + int64_t(r) * H * H;
    // conv1
    for (int co = 0; co < n.c1; ++co)
      for (int yy = 0; yy < H1; ++yy)
        for (int xx = 0; xx < H1; ++xx) {
          double acc = th[n.b1 + co];
          for (int ky = 0; ky < kK; ++ky)
            for (int kx = 0; kx < kK; ++kx)
              acc += th[n.w1 + (int64_t(co) * kK + ky) * kK + kx] * x[(yy + ky) * H + xx + kx];
          z1[(size_t(co) * H1 + yy) * H1 + xx] = acc;
        }
    // pool1, ReLU
    for (int co = 0; co < n.c1; ++co)
      for (int py = 0; py < P1; ++py)
        for (int px = 0; px < P1; ++px) {
          const double* map = &z1[size_t(co) * H1 * H1];
          const double v = map[argmax2x2(map, H1, py, px)];
          a1[(size_t(co) * P1 + py) * P1 + px] = v > 0.0 ? v : 0.0;
        }
    // conv2, dropout
    for (int co = 0; co < n.c2; ++co)
      for (int yy = 0; yy < H2; ++yy)
        for (int xx = 0; xx < H2; ++xx) {
          double acc = th[n.b2 + co];
          for (int ci = 0; ci < n.c1; ++ci)
            for (int ky = 0; ky < kK; ++ky)
              for (int kx = 0; kx < kK; ++kx)
                acc += th[n.w2 + ((int64_t(co) * n.c1 + ci) * kK + ky) * kK + kx] *
                       a1[(size_t(ci) * P1 + yy + ky) * P1 + xx + kx];
          z2[(size_t(co) * H2 + yy) * H2 + xx] = acc * drop[int64_t(r) * n.c2 + co];
        }
    // pool2, ReLU, flatten (channel, row, column)
    for (int co = 0; co < n.c2; ++co)
      for (int py = 0; py < P2; ++py)
        for (int px = 0; px < P2; ++px) {
          const double* map = &z2[size_t(co) * H2 * H2];
          const double v = map[argmax2x2(map, H2, py, px)];
          a2[(size_t(co) * P2 + py) * P2 + px] = v > 0.0 ? v : 0.0;
        }
    // fully connected layers
    for (int o = 0; o < n.f1; ++o) {
      double acc = th[n.bf1 + o];
      for (int k = 0; k < F; ++k) acc += th[n.wf1 + int64_t(o) * F + k] * a2[k];
      h1[o] = acc > 0.0 ? acc : 0.0;
    }
    for (int o = 0; o < n.f2; ++o) {
      double acc = th[n.bf2 + o];
      for (int k = 0; k < n.f1; ++k) acc += th[n.wf2 + int64_t(o) * n.f1 + k] * h1[k];
      h2[o] = acc > 0.0 ? acc : 0.0;
    }
    for (int o = 0; o < n.C; ++o) {
      double acc = th[n.bf3 + o];
      for (int k = 0; k < n.f2; ++k) acc += th[n.wf3 + int64_t(o) * n.f2 + k] * h2[k];
      zo[o] = acc;
      if (logits) logits[int64_t(r) * n.C + o] = acc;
    }
    // log-softmax and negative log-likelihood
    double zmax = zo[0];
    for (int c = 1; c < n.C; ++c) zmax = zo[c] > zmax ? zo[c] : zmax;
    double sum = 0.0;
    for (int c = 0; c < n.C; ++c) sum += std::exp(zo[c] - zmax);
    loss += (std::log(sum) + zmax) - zo[y[r]];
    if (!grad) continue;

    // backward: d(mean loss)/d logits = (softmax - onehot) / b
    for (int c = 0; c < n.C; ++c)
      dzo[c] = (std::exp(zo[c] - zmax) / sum - (c == y[r] ? 1.0 : 0.0)) / double(b);
    for (int o = 0; o < n.C; ++o) {
      grad[n.bf3 + o] += dzo[o];
      for (int k = 0; k < n.f2; ++k) grad[n.wf3 + int64_t(o) * n.f2 + k] += dzo[o] * h2[k];
    }
    for (int k = 0; k < n.f2; ++k) {
      double acc = 0.0;
      for (int o = 0; o < n.C; ++o) acc += dzo[o] * th[n.wf3 + int64_t(o) * n.f2 + k];
      dh2[k] = h2[k] > 0.0 ? acc : 0.0;
    }
    for (int o = 0; o < n.f2; ++o) {
      grad[n.bf2 + o] += dh2[o];
      for (int k = 0; k < n.f1; ++k) grad[n.wf2 + int64_t(o) * n.f1 + k] += dh2[o] * h1[k];
    }
    for (int k = 0; k < n.f1; ++k) {
      double acc = 0.0;
      for (int o = 0; o < n.f2; ++o) acc += dh2[o] * th[n.wf2 + int64_t(o) * n.f1 + k];
      dh1[k] = h1[k] > 0.0 ? acc : 0.0;
    }
    for (int o = 0; o < n.f1; ++o) {
      grad[n.bf1 + o] += dh1[o];
      for (int k = 0; k < F; ++k) grad[n.wf1 + int64_t(o) * F + k] += dh1[o] * a2[k];
    }
    for (int k = 0; k < F; ++k) {
      double acc = 0.0;
      for (int o = 0; o < n.f1; ++o) acc += dh1[o] * th[n.wf1 + int64_t(o) * F + k];
      da2[k] = a2[k] > 0.0 ? acc : 0.0;   // through the ReLU after pool2
    }
    // pool2 routes to its argmax, dropout scales, into conv2's output gradient
    std::fill(dz2.begin(), dz2.end(), 0.0);
    for (int co = 0; co < n.c2; ++co)
      for (int py = 0; py < P2; ++py)
        for (int px = 0; px < P2; ++px) {
          const double* map = &z2[size_t(co) * H2 * H2];
          const int q = argmax2x2(map, H2, py, px);
          dz2[size_t(co) * H2 * H2 + q] +=
              da2[(size_t(co) * P2 + py) * P2 + px] * drop[int64_t(r) * n.c2 + co];
        }
    // conv2: weights, bias, and input (a1) gradients
    std::fill(da1.begin(), da1.end(), 0.0);
    for (int co = 0; co < n.c2; ++co)
      for (int yy = 0; yy < H2; ++yy)
        for (int xx = 0; xx < H2; ++xx) {
          const double g = dz2[(size_t(co) * H2 + yy) * H2 + xx];
          grad[n.b2 + co] += g;
          for (int ci = 0; ci < n.c1; ++ci)
            for (int ky = 0; ky < kK; ++ky)
              for (int kx = 0; kx < kK; ++kx) {
                const int64_t wi = n.w2 + ((int64_t(co) * n.c1 + ci) * kK + ky) * kK + kx;
                const size_t ai = (size_t(ci) * P1 + yy + ky) * P1 + xx + kx;
                grad[wi] += g * a1[ai];
                da1[ai] += g * th[wi];
              }
        }
    // ReLU after pool1, pool1 routes to its argmax
    std::fill(dz1.begin(), dz1.end(), 0.0);
    for (int co = 0; co < n.c1; ++co)
      for (int py = 0; py < P1; ++py)
        for (int px = 0; px < P1; ++px) {
          const size_t ai = (size_t(co) * P1 + py) * P1 + px;
          if (!(a1[ai] > 0.0)) continue;
          const double* map = &z1[size_t(co) * H1 * H1];
          dz1[size_t(co) * H1 * H1 + argmax2x2(map, H1, py, px)] += da1[ai];
        }
    // conv1: weights and bias
    for (int co = 0; co < n.c1; ++co)
      for (int yy = 0; yy < H1; ++yy)
        for (int xx = 0; xx < H1; ++xx) {
          const double g = dz1[(size_t(co) * H1 + yy) * H1 + xx];
          if (g == 0.0) continue;
          grad[n.b1 + co] += g;
          for (int ky = 0; ky < kK; ++ky)
            for (int kx = 0; kx < kK; ++kx)
              grad[n.w1 + (int64_t(co) * kK + ky) * kK + kx] += g * x[(yy + ky) * H + xx + kx];
        }
  }
  return loss / double(b);
}

}  // namespace

extern "C" {

// Number of parameters of the network with shape {H, c1, c2, f1, f2, C}; -1 if invalid.
int64_t oracle_cnn_param_count(const int32_t* shape) {
  Net n;
  return make_net(shape, n) ? n.P : -1;
}

// Mean loss over the b samples X [b][H*H] with labels y and dropout scales drop [b][c2],
// at parameters theta [P] (double); grad [P] (may be NULL) receives its gradient and
// logits [b][C] (may be NULL) the network's outputs.  NaN on an invalid shape or label.
double oracle_cnn_loss_grad_f64(const int32_t* shape, const double* theta, const double* X,
                                const int32_t* y, const double* drop, int b, double* grad,
                                double* logits) {
  Net n;
  if (!make_net(shape, n) || b < 1) return NAN;
  for (int r = 0; r < b; ++r)
    if (y[r] < 0 || y[r] >= n.C) return NAN;
  return cnn_loss_grad(n, theta, X, y, drop, b, grad, logits);
}

// End-to-end simulation as oracle_mlp_sim_run, with the network above: for t = 0..T-1,
// worker order[t] computes the gradient of the mean loss over rows batch_rows[t][0..b)
// of X [x_rows][H*H] with dropout scales drop [t][b][c2] at its snapshot s_w (double,
// rounded to fp32) and commits it (oracle_gem_run_pi_f32, one commit).  theta [P],
// m and s [n][state_stride] fp32 are updated in place.  After commit record_at[r], theta
// is copied to record[r]; losses[t] (optional) receives commit t's minibatch loss.
int oracle_cnn_sim_run(const int32_t* shape, int n_workers, int T, const int32_t* order,
                       const int32_t* tau, const float* X, int64_t x_rows, const int32_t* labels,
                       const int32_t* batch_rows, int b, const float* drop, float* theta,
                       float* m, float* s, int64_t state_stride, double eta, double mu,
                       double eps, int mode, double kappa, int n_record,
                       const int32_t* record_at, float* record, double* losses) {
  Net n;
  if (!make_net(shape, n) || n_workers < 1 || T < 0 || b < 1 || !order || !X || !labels ||
      !batch_rows || !drop)
    return -1;
  if (state_stride < n.P) return -1;
  const int64_t P = n.P, HH = int64_t(n.H) * n.H;
  std::vector<double> params(P), grad(P), xb(size_t(b) * HH), db(size_t(b) * n.c2);
  std::vector<float> g32(P);
  std::vector<int32_t> yb(b);
  int rec = 0;
  for (int t = 0; t < T; ++t) {
    const int w = order[t];
    if (w < 0 || w >= n_workers) return -1;
    const float* sw = s + int64_t(w) * state_stride;
    for (int64_t j = 0; j < P; ++j) params[j] = double(sw[j]);
    for (int i = 0; i < b; ++i) {
      const int64_t row = batch_rows[int64_t(t) * b + i];
      if (row < 0 || row >= x_rows) return -1;
      for (int64_t k = 0; k < HH; ++k) xb[size_t(i) * HH + k] = double(X[row * HH + k]);
      yb[i] = labels[row];
      if (yb[i] < 0 || yb[i] >= n.C) return -1;
      for (int c = 0; c < n.c2; ++c)
        db[size_t(i) * n.c2 + c] = double(drop[(int64_t(t) * b + i) * n.c2 + c]);
    }
    const double loss = cnn_loss_grad(n, params.data(), xb.data(), yb.data(), db.data(), b,
                                      grad.data(), nullptr);
    if (losses) losses[t] = loss;
    for (int64_t j = 0; j < P; ++j) g32[j] = float(grad[j]);
    const int32_t one_w = w;
    const int32_t one_tau = tau ? tau[t] : 0;
    const int rc = oracle_gem_run_pi_f32(P, n_workers, 1, &one_w, &one_tau, g32.data(), P,
                                         nullptr, theta, m, s, state_stride, eta, mu, eps, mode,
                                         kappa, 0, nullptr);
    if (rc) return rc;
    while (record && rec < n_record && record_at[rec] == t) {
      std::memcpy(record + int64_t(rec) * P, theta, size_t(P) * sizeof(float));
      ++rec;
    }
  }
  return 0;
}

}  // extern "C"
