/* gem_sim.h -- the asynchronous-system simulator around the GEM commit path.
 *
 * The paper's workers commit asynchronously; which worker commits at each tick of the
 * global clock, and with what staleness, follows from an implicit queueing model
 * (Introduction, Eq. staleness: s_t = theta_{t - tau_t}, expected staleness n - 1 under
 * a homogeneous model).  On one GPU that behaviour is simulated: a seeded schedule fixes
 * the commit order, and a segment planner groups consecutive commits by distinct workers,
 * whose gradients can then be computed together because none of their snapshots changes
 * inside the group.
 *
 * Random numbers: SplitMix64 (Steele, Lea & Flood, OOPSLA 2014).  The stream for
 * (seed, id) starts at mix64(seed * 0x9E3779B97F4A7C15 + id) and its c-th output is
 * mix64(start + 0x9E3779B97F4A7C15 (c + 1)).  The schedule functions are host-only and
 * return 0, or -1 on an invalid argument; the MLP calls return a gem_status.
 */
#ifndef GEM_SIM_H
#define GEM_SIM_H

#include <stddef.h>
#include <stdint.h>

#include "gem.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Uniform tick (stream id 10): at tick t the worker floor(n u / 2^32) commits, u the top
 * 32 bits of output t.  order [T] receives the workers; tau [T] (may be NULL) the
 * staleness of each commit, t minus the tick of the worker's previous commit minus one
 * (t for its first commit: it pulled theta_0).  Requires n >= 1, T >= 0. */
int gem_schedule_uniform(uint64_t seed, int n, int T, int32_t* order, int32_t* tau);

/* Exponential-service queue (stream id 10 + 1): worker w's j-th gradient takes
 * -ln(1 - u) / rate time units, u = (output (w << 32) | j) >> 11 times 2^-53; the worker
 * that finishes first commits next (ties to the lower id) and starts its next gradient.
 * Same outputs as gem_schedule_uniform.  Requires rate > 0. */
int gem_schedule_queue(uint64_t seed, int n, int T, double rate, int32_t* order,
                       int32_t* tau);

/* Segment planner: cuts order [T] into maximal runs of consecutive commits by distinct
 * workers.  seg_start [T + 1] receives the first commit of each segment followed by T;
 * returns the number of segments S (seg_start[0..S]), or -1 on an invalid argument. */
int gem_plan_segments(const int32_t* order, int T, int n, int32_t* seg_start);

/* ---------------------------------------------------------------------------------
 * Worker gradients of a fully connected ReLU network, batched over stale snapshots.
 *
 * A worker computes dtheta = -eta grad L(s) at its snapshot s (notation table; Algorithm 1,
 * Worker).  The model here is an MLP dims[0] -> dims[1] -> ... -> dims[L] with ReLU on the
 * hidden layers and the mean softmax cross-entropy over the worker's minibatch as L.  Its
 * parameters are GEM's flat vector [W_1, b_1, W_2, b_2, ...], W_l stored dims[l] x
 * dims[l-1] row-major (out x in).  The gradients of a segment's workers (distinct workers,
 * so every snapshot is fixed for the whole segment) are computed together: each GEMM of
 * the forward and backward pass is one grouped launch over the segment.
 */
typedef struct gem_mlp gem_mlp_t;

enum gem_mlp_precision {
  GEM_MLP_FP32 = 0, /* fp32 products and sums */
  GEM_MLP_TF32 = 1  /* TF32 operands (10 explicit mantissa bits, round to nearest, ties
                       away from zero), products exact in fp32, fp32 sums: on the
                       tcgen05 tensor cores where both operands are K-major (forward
                       products; weight gradients through transposed minibatch panels),
                       on warp-level mma.sync for the input gradients, and on the CUDA
                       cores, with the same rounding, below 32 rows or a K of 32 */
};

/* Bind an MLP to a GEM handle (its P must equal the MLP's parameter count).  batch is the
 * per-worker minibatch b (1..1024); dims[L] <= 32 classes.  Allocates per-worker scratch
 * (activations and deltas, and for GEM_MLP_TF32 their TF32 transposes) and one gradient
 * buffer per worker on the handle's device. */
int gem_mlp_create(gem_t* gem, int n_layers, const int32_t* dims, int batch, int precision,
                   gem_mlp_t** out);

/* Training set: X [rows][dims[0]] fp32 and labels [rows] int32 in device memory, borrowed
 * (they must stay valid while the MLP is used). */
int gem_mlp_set_data(gem_mlp_t* mlp, const float* X, const int32_t* labels, int64_t rows);

/* Gradients of the mean loss at the snapshots of workers[0..L) (any workers, repeats
 * allowed) on minibatches batch_rows [L][batch] (host array of row indices into X, checked
 * against the data set and copied to the device before the call returns), written to
 * grads[i] (device, P floats, 16-byte aligned, caller-owned).  losses (device [L], may be
 * NULL) receives each minibatch's mean loss.  Asynchronous on the GEM handle's stream. */
int gem_mlp_grad(gem_mlp_t* mlp, const int32_t* workers, int L, const int32_t* batch_rows,
                 float* const* grads, float* losses);

/* End-to-end asynchronous GEM: commits t = 0..T-1 by workers order[t] (host array), commit
 * t using the minibatch batch_rows[t][0..batch) (host array, checked and copied to the
 * device before the call returns; an index outside the data set is GEM_EINVAL).  A label
 * outside [0, dims[L]) yields a NaN loss and gradient.  The schedule is cut into
 * segments of distinct workers (gem_plan_segments); per segment the workers' gradients
 * are computed at their snapshots in one batched forward/backward, then committed in
 * order with the fused commit kernel (so each snapshot is refreshed to the post-commit
 * theta).  losses (device [T], may be NULL) receives each commit's minibatch loss. */
int gem_mlp_run(gem_mlp_t* mlp, const int32_t* order, int T, const int32_t* batch_rows,
                float* losses);

/* gem_mlp_run that also follows the scaling factors, as the experiments section does: for
 * each commit t, the lower and upper medians (gem_pi_median) of the factors pi that the
 * commit applied to each tensor of the flat layout [W_1, b_1, ..., W_L, b_L] are written
 * to pi_lo[t][2L] and pi_hi[t][2L] (device arrays of T * 2 * n_layers floats; tensor 2l is
 * W_(l+1), 2l + 1 is b_(l+1)).  The commits are the same, bit for bit.  The first call
 * allocates a factor buffer of n rows of `stride` floats (the size of the gradient
 * buffers) and the select scratch. */
int gem_mlp_run_pi(gem_mlp_t* mlp, const int32_t* order, int T, const int32_t* batch_rows,
                   float* losses, float* pi_lo, float* pi_hi);

/* Wait for the MLP's work on the handle's stream (and its second stream); GEM_ECUDA if
 * device work failed or a tensor-core product reported an error: a wait on the tensor cores
 * that gave up after its time limit, or a read or write outside its buffers that it
 * skipped.  The handle is then unusable (GEM_ESTATE). */
int gem_mlp_status(gem_mlp_t* mlp);

/* Number of kernels the MLP has launched (gather, forward, loss, backward; the commits are
 * counted by gem_launch_count). */
uint64_t gem_mlp_launch_count(const gem_mlp_t* mlp);

/* The gradient of gem_mlp_grad for one set of parameters, for callers that cannot allocate
 * device memory: code that runs under a framework owning all device memory through its own
 * pool (an allocation outside it breaks the pool's budget), or in a loop where cudaMalloc's
 * device-wide synchronisation is not allowed.  Nothing is allocated and no handle is needed:
 * the caller passes the inputs (theta [P] in device memory, the data set X [rows][dims[0]]
 * and labels [rows] in device memory, the minibatch batch_rows [batch] as a host array,
 * checked and passed by value in a kernel's argument block, so the host array may be reused
 * as soon as the call returns) and the outputs (grad [P], device, 16-byte aligned; loss,
 * device, may be NULL).  The scratch is one file-scope device array of 4 MiB (1,048,576
 * floats) held by every GPU that loads the library until the process exits; a network whose
 * per-minibatch activations and deltas (plus the batch's row indices) do not fit in it is
 * rejected with GEM_EINVAL.  The first call on a device looks up the array's device
 * address, so make it before any stream capture; the address is looked up again if the
 * device's current context changes (after a reset of its primary context, say).  Calls
 * share the array and keep nothing in it between calls: calls queued one after another on
 * one stream are ordered, while calls that overlap on the GPU (other streams, other host
 * threads) race; order them on one stream.  The paper has no counterpart to this entry
 * point. */
int gem_mlp_grad_static(int n_layers, const int32_t* dims, int batch, int precision,
                        const float* theta, const float* X, const int32_t* labels,
                        int64_t rows, const int32_t* batch_rows, float* grad, float* loss,
                        void* stream);

/* Free the MLP's scratch (after its pending work).  NULL is a no-op. */
void gem_mlp_destroy(gem_mlp_t* mlp);

#ifdef __cplusplus
}
#endif

#endif /* GEM_SIM_H */
