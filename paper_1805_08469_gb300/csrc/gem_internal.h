// Internal declarations of the GEM commit library (not installed, not part of the ABI).
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <vector>

#include "../../include/gem.h"

namespace gem {

// Commits carried by one launch of the batched commit kernel.  They travel in the
// kernel's parameter block (2.4 KB + header), so a launch needs no device-side
// descriptor; longer batches are split into several launches, in order.
constexpr int kMaxBatchPerLaunch = 200;

// Row stride of m and s (and length of theta): P rounded up to 32 floats = 128 bytes.
constexpr size_t kStrideAlign = 32;

// Host-gradient staging for gem_commit_batch_host: two halves of kStageChunk slots.
constexpr int kStageChunk = 8;

// How a launch scales each commit.
enum RuleKind : int {
  kRuleGem = 0,     // pi from energy matching with the proxy |m_w| (Algorithm 1)
  kRuleScaled = 1,  // the same with the proxy energy_scale |m_w| (App. B, high-energy proxies)
  kRuleFixed = 2,   // pi[k] given per commit; m_w untouched (DOWNPOUR, adaptive staleness)
  kRuleMomentum = 3,  // the proxy itself: theta += (m_w <- mu m_w + dtheta); no factor
};

// Arguments of one launch of the fused commit kernel, for up to KCAP commits.  Launches of
// at most kSmallBatch commits (single commits, the segments of the simulators) pass the
// small form: the kernel parameters then take about 1 KB instead of 5.5 KB.
template <int KCAP>
struct BatchArgsT {
  float* theta;                            // [stride]
  float* m;                                // [n][stride]
  float* s;                                // [n][stride]
  size_t P;
  size_t stride;
  float eta, mu, eps;
  int K;                                   // commits in this launch, 1..KCAP
  int rule;                                // RuleKind
  float energy_scale;                      // kRuleScaled: factor on |m_w|
  const float* grad[KCAP];                 // gradient of commit k, P floats
  int worker[KCAP];                        // worker of commit k
  float pi[KCAP];                          // kRuleFixed: scaling factor of commit k
  int record_pi;                           // 1: pi_out[k] (when not null) receives pi
  float* pi_out[KCAP];                     // scaling factors of commit k, P floats, or null
  // Factor counts of a recording launch (null: none).  For every commit k with pi_out[k]
  // set and every segment s = [pi_seg[s], pi_seg[s + 1]) of the coordinates, the number of
  // recorded factors whose sign bit is set (below +0 in the total order of the medians) is
  // added to pi_counts[2 (k pi_nseg + s)] and the number equal to +0 to the word after it.
  // The block keeps its counts in dynamic shared memory from float4 count_smem_at on.
  unsigned* pi_counts;
  const long long* pi_seg;                 // device array [pi_nseg + 1], non-decreasing
  int pi_nseg;
  int count_smem_at;
  // On-chip reuse of a worker that commits again later in the launch (energy rules):
  // commit k keeps its m_w, s_w lanes in shared-memory slot slot_out[k] instead of writing
  // them to global memory, and the worker's next commit reads them from slot_in[k];
  // -1 means global memory.  Fixed-factor rules: keep_s[k] = 0 skips the store of s_w
  // when the worker commits again in the launch (nothing reads it before that).
  int8_t slot_in[KCAP];
  int8_t slot_out[KCAP];
  uint8_t keep_s[KCAP];
  // L2 policy of commit k's stores of m_w and s_w to global memory (launches of more than
  // kSmallBatch commits, energy rules): kL2Keep when a later commit of the launch reads
  // them back from global memory (no slot), kL2Stream at the worker's last commit of the
  // launch, kL2Normal otherwise.
  uint8_t l2[KCAP];
};
using BatchArgs = BatchArgsT<kMaxBatchPerLaunch>;
enum L2Hint : uint8_t { kL2Normal = 0, kL2Keep = 1, kL2Stream = 2 };
constexpr int kSmallBatch = 32;

// Shared-memory slots of the commit kernel (m_w and s_w lanes of one worker per slot), and
// the shortest repeat distance (in commits) given a slot: shorter repeats are served by L2.
#ifndef GEM_COMMIT_SLOTS
#define GEM_COMMIT_SLOTS 6
#endif
#ifndef GEM_COMMIT_SLOT_MIN_DISTANCE
#define GEM_COMMIT_SLOT_MIN_DISTANCE 4
#endif
#ifndef GEM_COMMIT_REG_SLOTS
#define GEM_COMMIT_REG_SLOTS 1
#endif
constexpr int kCommitSlots = GEM_COMMIT_SLOTS;
// Slots held in registers: ids kCommitSlots .. kCommitSlots + kRegSlots - 1 (one measured
// best: a second pushes the kernel past 64 registers into a spill).
constexpr int kRegSlots = GEM_COMMIT_REG_SLOTS;
constexpr int kTotalSlots = kCommitSlots + kRegSlots;
constexpr int kSlotMinDistance = GEM_COMMIT_SLOT_MIN_DISTANCE;

// Fill slot_in, slot_out, keep_s and l2 of a launch from its a.K workers.
void plan_slots(BatchArgs& a);

// Launch the fused commit kernel for a.K commits on `stream`.
cudaError_t launch_commit_batch(const BatchArgs& a, int sm_count, cudaStream_t stream);

// Shared-memory words a recording launch may use for its factor counts (2 per commit and
// segment); callers split their commits so that K * pi_nseg * 2 stays within it.
constexpr int kMaxCountWords = 4096;

}  // namespace gem

struct gem_ctx {
  int device = 0;
  int sm_count = 0;
  size_t P = 0;
  size_t stride = 0;
  int n = 0;
  float eta = 0.f, mu = 0.f, eps = 0.f;
  float* theta = nullptr;
  float* m = nullptr;
  float* s = nullptr;
  cudaStream_t stream = nullptr;
  uint64_t launches = 0;
  bool broken = false;
  // commit rule (gem_set_mode) and the commit clock the staleness is counted on
  int mode = GEM_MODE_GEM;
  float kappa = 1.f;
  int64_t clock = 0;           // commits issued since gem_set_theta
  std::vector<int64_t> last;   // [n] clock value of worker w's last commit, -1 before its first
  // scratch of the pi median select: histograms and per-problem state, grown on demand
  void* select_scratch = nullptr;
  size_t select_bytes = 0;
  // staging of host gradients (gem_commit_batch_host), allocated on first use
  float* stage = nullptr;
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t stage_filled[2] = {nullptr, nullptr};
  cudaEvent_t stage_free[2] = {nullptr, nullptr};
};

namespace gem {

// Launch commits [0, K) of the handle in order, in chunks of kMaxBatchPerLaunch, with the
// handle's commit rule; advances the commit clock and counts the launches.  The arguments
// must have been checked.
// With pi_counts set (K * pi_nseg * 2 <= kMaxCountWords, one launch), the recording launch
// also adds the factor counts of every commit and segment to pi_counts (see BatchArgsT).
cudaError_t commit_ordered(gem_ctx* h, const int* order, const float* const* grads, int K,
                           float* const* pi_out = nullptr, unsigned* pi_counts = nullptr,
                           const long long* pi_seg = nullptr, int pi_nseg = 0);

// Segments per median call and commits per select launch.
constexpr int kMaxPiSegments = 64;
constexpr int kMaxPiBatch = 200;

// Exact lower and upper medians of each segment of each of K scaling-factor rows
// (segments seg[0..nseg] shared by all rows), written to lo/hi [K][nseg] on the handle's
// stream.  Uses the handle's select scratch (grown on demand).  Arguments checked by the
// caller.
cudaError_t pi_median_ordered(gem_ctx* h, const float* const* pi, int K, const int64_t* seg,
                              int nseg, float* lo, float* hi);

// Commits [0, K) in order with every factor recorded in pi[k] (all set), then the lower and
// upper medians of each row and segment as pi_median_ordered.  The recording launches also
// count each row's factors below and equal to +0 per segment, so a middle element that lies
// in the run of zeros is known before any selection pass, and a row and segment whose two
// middle elements both lie there is never read again.  Arguments checked by the caller.
cudaError_t commit_pi_median_ordered(gem_ctx* h, const int* order, const float* const* grads,
                                     int K, float* const* pi, const int64_t* seg, int nseg,
                                     float* lo, float* hi);

}  // namespace gem
