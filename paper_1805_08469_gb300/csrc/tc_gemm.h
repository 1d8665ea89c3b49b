// Grouped TF32 matrix products on the 5th-generation tensor cores (tcgen05), internal to the
// library: the worker products of the batched MLP forward/backward (Algorithm 1, Worker:
// the gradient of each worker at its own snapshot).
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

namespace gem {
namespace tc {

constexpr int kMaxGroups = 128;

// Epilogues (the same values as the MLP engine's): plain store, + bias[n], ReLU(+ bias[n]),
// and keep where mask(m, n) > 0.
enum Epi : int { kStore = 0, kBias = 1, kBiasRelu = 2, kMask = 3 };

// A K-major operand of group g: its elements start at base + gidx * group_stride, gidx = g
// or workers[g] (by_worker); A is indexed (m, k), B (n, k), element (r, k) at [r * ld + k].
// extent: floats addressable from base (every read is checked against it).
struct Operand {
  const float* base;
  long long group_stride;
  long long ld;
  long long extent;
  int by_worker;
  int rounded;   // its values are TF32 already (the kernel then does not round them again)
};

// C[g] (M x N, row-major with ldc) = epilogue(sum_k A(m, k) B(n, k)) with every operand
// value rounded to TF32 (round to nearest, ties away from zero) and fp32 accumulation.
// bias and mask are indexed like the MLP engine's: bias by worker, bias[n]; mask by group,
// mask[m * ldmask + n].  The operands are read by tensor copies whose maps cover exactly the
// rows x K x groups (or workers) that supported() checked against the operands' extents;
// every other global read and every write is checked against its extent, and an access
// outside it is skipped and reported in *status (which stays 0 on success), as is a wait on
// the tensor cores that gave up.
struct Args {
  int M, N, K;
  Operand A, B;
  float* C;
  long long c_group_stride, ldc, c_extent;
  int round_c;        // store C rounded to TF32 (for outputs that are only used as operands)
  // optional transposed copy: CT[g] (N x M, row-major with ldct) = the epilogue's output
  // rounded to TF32, at ct + g * ct_group_stride (null: none)
  float* ct;
  long long ct_group_stride, ldct, ct_extent;
  const float* bias;
  long long bias_group_stride, bias_extent;
  const float* mask;
  long long mask_group_stride, ldmask, mask_extent;
  unsigned* status;
  int workers[kMaxGroups];
};

// Error codes written to *status (the first one wins).
enum Status : unsigned {
  kOk = 0,
  kWaitStage = 1,    // a wait for a stage's MMAs to finish gave up
  kWaitDone = 2,     // the wait for the accumulator gave up
  kOutOfRange = 3,   // an access outside an operand's extent was skipped
};

// Whether launch() takes this product over `groups` groups: both operands K-major and
// 16-byte aligned (base, ld and group stride in multiples of 4 floats), every element of
// rows x K x groups (or x the workers named, for an operand indexed by worker) inside the
// operand's extent, and any of the epilogues.
bool supported(const Args& a, bool a_kmajor, bool b_kmajor, int epi, int groups);

// Launch over `groups` groups (a persistent grid of one CTA per SM over the N tiles x M
// tiles x groups), as a programmatic dependent of the previous kernel in `stream`.
// a_kmajor / b_kmajor give the operands' layouts; epi an Epi value.  Returns the launch error
// (cudaErrorInvalidValue for a product supported() does not take).
cudaError_t launch(const Args& a, int groups, bool a_kmajor, bool b_kmajor, int epi,
                   cudaStream_t stream);

}  // namespace tc
}  // namespace gem
