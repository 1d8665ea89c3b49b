/* gem.h -- C ABI of the Gradient Energy Matching commit path for GB300 (sm_103a).
 *
 * Gradient Energy Matching (GEM; Hermans & Louppe, "Gradient Energy Matching for
 * Distributed Asynchronous Gradient Descent", arXiv 1805.08469) lets n asynchronous
 * workers update a central variable theta.  Each commit is rescaled elementwise so the
 * kinetic energy the workers put into theta together stays at or below the energy of
 * momentum SGD.  This library keeps theta, every worker's first moment m_w and its
 * snapshot s_w in the memory of one GPU.  A commit by worker w with gradient g
 * (computed by the caller at s_w) does, for every coordinate j:
 *
 *   dtheta = -(eta * g)                    worker update (notation table; Algorithm 1, Worker)
 *   m_w    = mu * m_w + dtheta             Psi_GEM, first step (Eq. moment_estimate)
 *   pi     = (|m_w| - |theta - s_w|) / (|dtheta| + eps),  clamped to pi >= 0
 *                                          Psi_GEM, second step (Eq. new_pi; |m_w| is
 *                                          sqrt(2) sqrt(E_k) by Eq. proxy_estimate)
 *   theta  = theta + pi * dtheta           Commit (Eqs. traditional_async_update, update_psi)
 *   s_w    = theta                         the worker's pull for its next gradient
 *
 * Every step is one IEEE-754 fp32 operation rounded to nearest: no fused multiply-add
 * and an IEEE division.  This order is part of the contract; it makes each commit
 * reproducible bit for bit.
 *
 * Conventions shared by every call:
 *   - Return value: GEM_OK (0) or a negative gem_status.  Arguments are checked on the
 *     host; a call that fails a check changes nothing and launches nothing.
 *   - Device work is asynchronous and ordered on the handle's stream (gem_set_stream;
 *     the legacy default stream until set).  A CUDA error raised by device work is
 *     reported by a later call, at the latest by gem_sync, as GEM_ECUDA.  Kernels are
 *     launched as programmatic dependents of the previous kernel in the stream: each
 *     waits, before it touches memory, until that kernel has completed and its writes
 *     are visible, so stream order holds as for plain launches (also when captured
 *     into a CUDA graph), while the launch itself overlaps the previous kernel.
 *   - Caller buffers are fp32, 16-byte aligned, and must stay valid and unmodified until
 *     the work that reads them has completed on the stream.  The library never keeps a
 *     caller pointer beyond that work.
 *   - State is library-owned device memory: theta [P] and m, s [n][stride] fp32, row w of
 *     m and s belonging to worker w.  stride is P rounded up to a multiple of 32 floats
 *     (128 bytes).  Elements past P hold 0 and stay 0.
 *   - A handle is not thread-safe; separate handles are independent.
 */
#ifndef GEM_H
#define GEM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gem_ctx gem_t;

enum gem_status {
  GEM_OK = 0,
  GEM_EINVAL = -1, /* an argument failed a host-side check */
  GEM_ENOMEM = -2, /* device or pinned-host allocation failed */
  GEM_ECUDA = -3,  /* a CUDA call failed, or device work raised an error */
  GEM_ESTATE = -4  /* the handle is unusable after an earlier CUDA error */
};

/* Create a handle for P parameters and n workers on the current CUDA device.
 * Hyper-parameters follow Algorithm 1: learning rate eta > 0, momentum 0 <= mu < 1,
 * eps > 0 (the term that keeps pi finite when dtheta = 0; the paper's default is 1e-16).
 * Allocates theta [P] and m, s [n][stride] on the device; theta = 0, m = 0, s = 0.
 * Requires P >= 1 and n >= 1.  On success *out receives the handle. */
int gem_create(size_t P, int n, float eta, float mu, float eps, gem_t** out);

/* Free every resource of the handle after finishing its pending work.  NULL is a no-op. */
void gem_destroy(gem_t* h);

/* Order all later device work of the handle on `stream` (a cudaStream_t of the handle's
 * device; NULL selects the legacy default stream).  Work already issued is not moved. */
int gem_set_stream(gem_t* h, void* stream);

/* Initial pull (Algorithm 1, Worker: m <- 0, s <- Pull()): theta = theta0, s_w = theta0
 * and m_w = 0 for every worker.  theta0 holds P fp32 values in device memory or in host
 * memory (any pointer the CUDA runtime can copy from). */
int gem_set_theta(gem_t* h, const float* theta0);

/* Pull (Algorithm 1, Worker): *snapshot receives the device address of s_w, the central
 * variable as it was right after worker w's last commit (theta0 before its first).  The
 * memory is borrowed: read-only for the caller, and valid, with that content, until the
 * next commit of worker w is issued.  Requires 0 <= worker < n. */
int gem_pull(gem_t* h, int worker, const float** snapshot);

/* One commit by worker w (Algorithm 1, Psi_GEM then Commit, then s <- theta): the five
 * steps listed at the top of this file, over all P coordinates, in one kernel that
 * reads grad, m_w, s_w, theta and writes m_w, s_w, theta once each.  grad is P fp32
 * values in device memory (the gradient of the loss at s_w; the call forms
 * dtheta = -eta grad itself).  Requires 0 <= worker < n and grad 16-byte aligned. */
int gem_commit(gem_t* h, int worker, const float* grad);

/* K commits in order: commit k is made by worker order[k] with gradient grads[k].  The
 * result equals K calls of gem_commit in that order, bit for bit, including repeated
 * workers.  order and grads are host arrays of length K, read before the call returns;
 * each grads[k] is P fp32 values in device memory, 16-byte aligned.  theta is read and
 * written once per batch instead of once per commit.  Requires K >= 0 (K = 0 is a
 * no-op) and 0 <= order[k] < n. */
int gem_commit_batch(gem_t* h, const int* order, const float* const* grads, int K);

/* As gem_commit_batch, with each grads[k] in host memory instead.  When every gradient is
 * page-locked (cudaHostAlloc / cudaHostRegister) and 16-byte aligned, the commit kernel
 * reads them in place over the host link and nothing is copied.  Otherwise the gradients
 * are copied to library-owned device staging buffers on a second stream, in chunks that
 * overlap with the commits of earlier chunks; those buffers are allocated by the first such
 * call (16 gradients of `stride` floats).  Either way the host buffers must stay valid and
 * unmodified until the handle's stream has finished the batch. */
int gem_commit_batch_host(gem_t* h, const int* order, const float* const* grads, int K);

/* *theta receives the device address of theta [P] (borrowed, read-only, valid until
 * gem_destroy; its content changes with every commit). */
int gem_theta(gem_t* h, const float** theta);

/* *moment receives the device address of m_w [P] (borrowed, read-only). */
int gem_moment(gem_t* h, int worker, const float** moment);

/* Checkpoint: stream-ordered copies of the whole state into theta [P], m [n][P] and s [n][P]
 * (dense rows of P floats; host or device memory).  Any of the three may be NULL. */
int gem_save_state(gem_t* h, float* theta, float* m, float* s);

/* Resume: replace the whole state with theta [P], m [n][P] and s [n][P] (dense rows of P
 * floats; host or device memory; NULL leaves that part unchanged).  The snapshot s_w is the
 * central variable as worker w last pulled it and m_w its first moment (Algorithm 1). */
int gem_load_state(gem_t* h, const float* theta, const float* m, const float* s);

/* Stream-ordered copy of theta [P] into `out` (host or device memory). */
int gem_read_theta(gem_t* h, float* out);

/* Block until the handle's stream has finished; GEM_ECUDA if device work failed. */
int gem_sync(gem_t* h);

/* Layout query: P, n and the row stride (in floats) of m and s.  Any output may be NULL. */
int gem_shape(const gem_t* h, size_t* P, int* n, size_t* stride);

/* Commit rules.  GEM_MODE_GEM is the rule at the top of this file and the default; the
 * others are the comparison rules of the paper's experiments and the high-energy proxies
 * of its Appendix B.  Each is computed in fp32, one IEEE operation per step:
 *
 *   GEM_MODE_GEM           Algorithm 1: the five steps above.
 *   GEM_MODE_DOWNPOUR      the DOWNPOUR rule: theta = theta + dtheta (pi = 1), s_w = theta;
 *                          m_w is not read or changed.
 *   GEM_MODE_ADAPTIVE      adaptive staleness (experiments section): the update is rescaled
 *                          by 1 / (tau + 1), pi = 1 / (tau + 1) rounded to fp32 and
 *                          theta = theta + pi * dtheta, s_w = theta; m_w is not read or
 *                          changed.  tau is the commit's staleness on the handle's clock
 *                          (gem_staleness).
 *   GEM_MODE_KAPPA_SQRT    App. B, Eq. pi_with_kappa: as GEM with |m_w| replaced by
 *                          sqrt(kappa) * |m_w| (sqrt(kappa) rounded to fp32 first).
 *   GEM_MODE_KAPPA_LINEAR  App. B, the modified form used in its study: as GEM with |m_w|
 *                          replaced by kappa * |m_w|.
 *   GEM_MODE_MOMENTUM      the proxy itself, as a reference run (Eq. momentum_update):
 *                          m_w = mu * m_w + dtheta, theta = theta + m_w, s_w = theta; no
 *                          scaling factor is formed (gem_commit_batch_pi records NaN).  With
 *                          one worker this is sequential momentum SGD. */
enum gem_mode {
  GEM_MODE_GEM = 0,
  GEM_MODE_DOWNPOUR = 1,
  GEM_MODE_ADAPTIVE = 2,
  GEM_MODE_KAPPA_SQRT = 3,
  GEM_MODE_KAPPA_LINEAR = 4,
  GEM_MODE_MOMENTUM = 5
};

/* Select the rule of every later commit.  kappa is the proxy's energy factor: required
 * finite and > 0 for the two kappa modes, ignored (and reported as 1) for the others.
 * Host-side only: takes effect for commits issued after the call. */
int gem_set_mode(gem_t* h, int mode, float kappa);

/* Current rule and kappa.  Either output may be NULL. */
int gem_get_mode(const gem_t* h, int* mode, float* kappa);

/* Staleness bookkeeping.  The handle numbers commits 0, 1, 2, ... in the order they are
 * issued (its clock, reset to 0 by gem_set_theta).  A worker pulls right after its own
 * commit, so the staleness of a commit by w at clock t is the number of commits by the
 * other workers since then: tau = t - last_w - 1, with last_w the clock value of w's
 * previous commit, or -1 before its first.  *tau receives the staleness that w's next
 * commit will have. */
int gem_staleness(const gem_t* h, int worker, int64_t* tau);

/* The clock and last[w] for each of the n workers (last may be NULL); with gem_save_state
 * this is the whole of a checkpoint. */
int gem_get_clock(const gem_t* h, int64_t* clock, int64_t* last);

/* Restore the clock: clock >= 0 and -1 <= last[w] < clock for every worker (last NULL: -1
 * for all).  Returns GEM_EINVAL and changes nothing if a value is out of range. */
int gem_set_clock(gem_t* h, int64_t clock, const int64_t* last);

/* Scaling-factor statistics.  The experiments section follows the median per-parameter
 * value of pi over time (and, in the appendix, per tensor) to show how GEM rescales the
 * commits as workers are added.  These two calls record pi and take exact medians.
 *
 * gem_commit_batch_pi: gem_commit_batch, and when pi is not NULL and pi[k] is not NULL,
 * the scaling factor that commit k applied to each coordinate is written to pi[k] [P]
 * (device memory, 16-byte aligned): the clamped pi of the GEM and kappa rules, 1 for
 * DOWNPOUR, 1 / (tau + 1) for adaptive staleness.  The commits themselves are unchanged,
 * bit for bit.  pi and its entries are host data read before the call returns. */
int gem_commit_batch_pi(gem_t* h, const int* order, const float* const* grads, int K,
                        float* const* pi);

/* Exact medians of K rows of P floats (typically recorded by gem_commit_batch_pi), per
 * segment: segment i of row k is pi[k][seg[i] .. seg[i+1]).  With its N elements sorted
 * ascending, lo[k * nseg + i] receives element (N - 1) / 2 and hi[k * nseg + i] element
 * N / 2 (the same for odd N; their mean is the usual median); NaN for an empty segment.
 * pi is a host array of K device pointers (4-byte aligned); seg is a host array of nseg + 1
 * offsets with 0 <= seg[0] <= ... <= seg[nseg] <= P, 1 <= nseg <= 64; lo and hi are device
 * arrays of K * nseg floats.  "Sorted" is the total order of the float bits: -0 below +0,
 * NaNs with the sign bit set below everything, other NaNs above.  Stream-ordered: up to
 * three passes over the rows (radix selection, 11 + 11 + 10 bits of an order-preserving
 * key; a median that falls in a run of exact +0, as clamped factors give, is resolved by
 * the first pass).  The first call, and any call with more rows or segments than before
 * (up to 200 rows per pass), allocates the select scratch: 16 KB per row and segment. */
int gem_pi_median(gem_t* h, const float* const* pi, int K, const int64_t* seg, int nseg,
                  float* lo, float* hi);

/* gem_commit_batch_pi with every factor recorded (each pi[k] set, 16-byte aligned), followed
 * by gem_pi_median of the K recorded rows with segments seg[0..nseg], in one call, with the
 * same results bit for bit (commits, recorded rows, lo and hi).  The commit kernel also
 * counts, for every row and segment, the factors below +0 and equal to +0 as it writes them
 * (the median of the experiments section is often +0 at many workers, where most clamped
 * factors are exactly 0): a middle element inside the run of +0 is then known without a
 * selection pass, and a row and segment whose two middle elements both lie there is never
 * read back.  Commits are taken in chunks of at most 200 (at most 2048 / nseg), each a
 * commit launch followed by the selection of its rows.  The first call, and any call with
 * more rows per chunk or segments than before, allocates the select scratch. */
int gem_commit_batch_pi_median(gem_t* h, const int* order, const float* const* grads, int K,
                               float* const* pi, const int64_t* seg, int nseg, float* lo,
                               float* hi);

/* Parameter sharding.  Every step of a commit is elementwise (Algorithm 1 applies Psi_GEM
 * with an elementwise product, and pi is a per-parameter vector), so coordinate j of theta,
 * m_w and s_w depends only on coordinate j of the gradients.  A parameter vector can
 * therefore be split into contiguous shards, each held by its own handle (one per GPU, or
 * several on one GPU), and committing the matching slice of every gradient to every shard
 * gives, shard by shard, the same bits as one handle over all P: no data is exchanged
 * between shards on the commit path.  This call gives shard `rank` of `world`:
 * [*begin, *end) with boundaries on multiples of 32 floats (128 bytes), so the slice of a
 * 16-byte-aligned gradient stays 16-byte aligned; shards differ in size by at most 32
 * floats, and the last non-empty one ends at P.  A shard with *begin == *end holds nothing
 * (world larger than P / 32, rounded up).  Host-only; needs no GPU. */
int gem_shard_range(size_t P, int world, int rank, size_t* begin, size_t* end);

/* Number of kernels this handle has launched since it was created. */
uint64_t gem_launch_count(const gem_t* h);

/* Human-readable name of a gem_status value (static storage). */
const char* gem_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* GEM_H */
