// Internal declarations shared by the MLP and CNN drivers (not installed, not part of the
// ABI): the dense-network engine that computes the workers' gradients of a segment.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/gem_sim.h"
#include "gem_internal.h"

namespace gem {
namespace mlp {

constexpr int kMaxLayers = 8;
constexpr int kMaxGroups = 128;
constexpr int kMaxClasses = 32;
constexpr int kMaxBatch = 1024;

}  // namespace mlp
}  // namespace gem

struct gem_mlp {
  gem_t* gem = nullptr;
  int L = 0;
  int dims[gem::mlp::kMaxLayers + 1] = {};
  long long w_off[gem::mlp::kMaxLayers] = {}, b_off[gem::mlp::kMaxLayers] = {};
  int batch = 0;
  int precision = 0;
  // use inside a larger network: parameters start at param_base in theta; the caller
  // fills the input rows (off_x) instead of the gather; input_grad asks for the gradient
  // with respect to the input, D_0 [b x d0] at off_delta[0]
  long long param_base = 0;
  bool external_input = false;
  bool input_grad = false;
  const float* X = nullptr;
  const int32_t* labels = nullptr;
  int64_t rows = 0;
  // per-slot scratch: X_s [b x d0], A_l [b x d_l] (l = 1..L-1), logits [b x C],
  // D_l [b x d_l] (l = 1..L, and l = 0 with input_grad)
  long long off_x = 0, off_act[gem::mlp::kMaxLayers + 1] = {}, off_logits = 0, off_delta[gem::mlp::kMaxLayers + 1] = {};
  long long off_row_loss = 0;   // per-row losses of the minibatch [b] (fused loss)
  // TF32 engine: TF32-rounded transposes of the minibatch panels that the weight-gradient
  // products dW_l = D_{l+1}^T A_l read K-major: A_l^T [d_l x b] (X^T for l = 0) and
  // D_{l+1}^T [d_{l+1} x b] (has_t: the layout holds them)
  bool has_t = false;
  long long off_actT[gem::mlp::kMaxLayers + 1] = {};
  long long off_deltaT[gem::mlp::kMaxLayers + 1] = {};
  long long slot_stride = 0;
  int slots = 0;
  float* scratch = nullptr;
  float* scratch_end = nullptr;   // one past the scratch (bounds of the tensor-core reads)
  unsigned* tc_status = nullptr;  // error word of the tensor-core products (TF32), 0 = none
  float* grads = nullptr;  // [n][gem stride]
  float* ws = nullptr;     // split-K partial sums
  float* pi_rows = nullptr;  // [n][gem stride] scaling factors of a segment's commits
  long long ws_floats = 0;
  // second stream for the weight-gradient products, which nothing waits for until the
  // commit; ev_delta[l] marks D_l ready on the main stream, ev_side the side stream's end
  cudaStream_t side = nullptr;
  cudaEvent_t ev_delta[gem::mlp::kMaxLayers + 1] = {};
  cudaEvent_t ev_side = nullptr;
  // ev_x: the minibatch rows gathered (main stream), for X^T on the side stream
  cudaEvent_t ev_x = nullptr;
  int32_t* rows_dev = nullptr;  // minibatch rows uploaded from the host
  size_t rows_cap = 0;
  uint64_t launches = 0;
};

namespace gem {
namespace mlp {

// A dense network of n_layers layers (dims[0..n_layers]) bound to the GEM handle g, with
// per-slot scratch for min(n, kMaxGroups) workers.  Its parameters start at param_base in
// theta (the whole of theta for gem_mlp_create).  own_grads allocates one gradient row per
// worker for gem_mlp_run / gem_mlp_grad.  Returns a gem_status.
int mlp_build(gem_t* g, int n_layers, const int32_t* dims, int batch, int precision,
              long long param_base, bool external_input, bool input_grad, bool own_grads,
              gem_mlp** out);

// Free everything mlp_build allocated (after the handle's pending work).
void mlp_free(gem_mlp* M);

// Forward and backward for groups [0, G) of one chunk: workers[g] (snapshots s_w),
// minibatch rows batch_rows[g][0..b) (device; labels, and the gather unless the input is
// external), gradient of group g written at grads + g * grad_stride (whole-theta indexing),
// losses[g] (device, may be null) the minibatch losses.  Stream-ordered on the handle's
// stream.  Returns a gem_status.
int mlp_chunk(gem_mlp* M, const int32_t* workers, int G, const int32_t* batch_rows,
              float* grads, long long grad_stride, float* losses);

inline float* mlp_input(gem_mlp* M, int g) { return M->scratch + g * M->slot_stride + M->off_x; }
inline float* mlp_input_grad(gem_mlp* M, int g) {
  return M->scratch + g * M->slot_stride + M->off_delta[0];
}

}  // namespace mlp
}  // namespace gem
