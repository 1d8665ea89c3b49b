/* gem_cnn.h -- the convolutional network of the paper's MNIST experiments as the workers'
 * model (C ABI, sm_103a).
 *
 * Appendix A of Hermans & Louppe (arXiv 1805.08469) trains, with GEM, a network of two
 * 5 x 5 convolutional layers (no padding, stride 1; 1 -> 10 and 10 -> 20 channels), each
 * followed by 2 x 2 max-pooling and ReLU, with dropout (PyTorch's default, p = 0.5, by
 * channel) on the second convolution, then three fully connected layers with ReLU and a
 * log-softmax.  The appendix does not give the fully connected sizes; this library takes
 * them, with the input side and the channel counts, as a shape
 *
 *   shape = {H, c1, c2, f1, f2, C}      (the paper's network: {28, 10, 20, 128, 64, 10})
 *
 * with H - 4 even and (H - 4) / 2 - 4 even and positive; F = c2 ((H - 4) / 2 - 4)^2 / 4
 * features reach the first fully connected layer (320 for H = 28).  The loss is the mean
 * negative log-likelihood of the minibatch.  Max-pooling routes its gradient to the first
 * maximum of each window (row-major order).
 *
 * Parameters are one flat fp32 vector of gem_cnn_param_count(shape) values, in the order
 * conv1.W [c1][1][5][5], conv1.b [c1], conv2.W [c2][c1][5][5], conv2.b [c2], fc1.W [f1][F],
 * fc1.b [f1], fc2.W [f2][f1], fc2.b [f2], fc3.W [C][f2], fc3.b [C]; the GEM handle's P must
 * equal that count.  Arithmetic is fp32 on the CUDA cores (the fully connected products
 * through the MLP engine of gem_sim.h), with fixed summation orders: results do not depend
 * on timing.
 *
 * Dropout draws random numbers; they are inputs here: drop [..][b][c2] holds, per commit,
 * sample and channel of conv2, the scale of that channel (0 for a dropped channel, 2 for a
 * kept one with p = 0.5; gem_synth_dropout generates them).  Conventions of gem.h apply.
 */
#ifndef GEM_CNN_H
#define GEM_CNN_H

#include <stddef.h>
#include <stdint.h>

#include "gem.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gem_cnn gem_cnn_t;

/* Number of parameters of the network with this shape, or -1 if the shape is invalid. */
int64_t gem_cnn_param_count(const int32_t* shape);

/* Bind the network to a GEM handle (P must equal gem_cnn_param_count(shape)).  batch is the
 * per-worker minibatch b (1..1024); C <= 32 classes.  Allocates per-worker scratch for
 * min(n, 128) workers at a time and one gradient buffer per worker on the handle's
 * device. */
int gem_cnn_create(gem_t* gem, const int32_t* shape, int batch, gem_cnn_t** out);

/* Training set: X [rows][H * H] fp32 and labels [rows] int32 in device memory, borrowed. */
int gem_cnn_set_data(gem_cnn_t* cnn, const float* X, const int32_t* labels, int64_t rows);

/* Gradients of the mean loss at the snapshots of workers[0..L) on minibatches batch_rows
 * [L][batch] (host array, checked against the data set and copied before the call returns)
 * with dropout scales drop [L][batch][c2] (device), written to grads[i] (device, P floats,
 * 16-byte aligned).  losses (device [L], may be NULL) receives the minibatch losses. */
int gem_cnn_grad(gem_cnn_t* cnn, const int32_t* workers, int L, const int32_t* batch_rows,
                 const float* drop, float* const* grads, float* losses);

/* End-to-end asynchronous GEM on the network, as gem_mlp_run: commit t by worker order[t]
 * on minibatch batch_rows[t] (host [T][batch]) with dropout scales drop[t] (device
 * [T][batch][c2]); segments of distinct workers get their gradients in one batched
 * forward/backward, then the fused commit.  losses (device [T], may be NULL). */
int gem_cnn_run(gem_cnn_t* cnn, const int32_t* order, int T, const int32_t* batch_rows,
                const float* drop, float* losses);

/* gem_cnn_run that also follows the scaling factors, as the experiments section does for
 * this network: for each commit t, the lower and upper medians (gem_pi_median) of the
 * factors pi that the commit applied to each of the 10 tensors of the flat layout are
 * written to pi_lo[t][10] and pi_hi[t][10] (device arrays of 10 T floats, tensors in
 * layout order).  The commits are the same, bit for bit.  The first call allocates a
 * factor buffer of n rows of the handle's stride and the select scratch. */
int gem_cnn_run_pi(gem_cnn_t* cnn, const int32_t* order, int T, const int32_t* batch_rows,
                   const float* drop, float* losses, float* pi_lo, float* pi_hi);

/* Wait for the network's work; GEM_ECUDA if device work failed. */
int gem_cnn_status(gem_cnn_t* cnn);

/* Kernels launched by the network (the commits are counted by gem_launch_count). */
uint64_t gem_cnn_launch_count(const gem_cnn_t* cnn);

/* Free the network's scratch (after its pending work).  NULL is a no-op. */
void gem_cnn_destroy(gem_cnn_t* cnn);

#ifdef __cplusplus
}
#endif

#endif /* GEM_CNN_H */
