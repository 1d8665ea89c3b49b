// Exact medians of the scaling factors pi, per commit and per segment (the statistic of the
// experiments section: the median per-parameter value of pi, over time, and per tensor in
// the ImageNet figures of the appendix).
//
// Selection by radix on an order-preserving 32-bit key of each float, most significant
// digit first, in three passes of 11, 11 and 10 bits.  Every problem (commit k, segment s)
// has two targets, the lower and upper middle elements (ranks (N - 1) / 2 and N / 2 of the
// N elements sorted ascending).  A target is a (prefix, mask, rank) triple: the key bits
// fixed so far and the rank of the target among the elements that share them.
//   - select_hist_kernel: blocks of 16,384 elements of one segment count, in shared memory,
//     the next digit of every element that matches a target's prefix, and add their
//     counts to the problem's histogram in global memory.  Counts are aggregated per warp
//     (one shared-memory atomic per distinct digit), because clamped factors put many
//     equal keys (pi = 0) into one bin.  While both targets share their prefix, which is
//     always true in the first pass, one histogram serves both.
//   - select_pick_kernel: one block per problem scans the histogram, finds the bin that
//     holds each target's rank, extends the prefix and reduces the rank, then clears the
//     histogram for the next pass.
// After the third pass the prefix is the target's key, which maps back to its float.
// Each pass reads the factors once (4 bytes per element), so 12 bytes per element.
// Runs of exact zeros: pi = max(0, .) makes +0 common (at P = 25M often more than half of
// a commit's factors), and then every pass funnels those elements into one bin.  The first
// pass therefore counts the elements equal to +0 apart (in word kBins of the histogram,
// which the first pass does not otherwise use); every smaller key lies in the bins below
// +0's first-pass bin, so a target whose rank falls in the run of zeros is resolved after
// one pass (its mask becomes full), and later passes skip it, and skip a problem whose
// targets are both resolved.
// Fused with the commit (commit_pi_median_ordered): the recording commit kernel counts, per
// row and segment, the factors below +0 and equal to +0 while it writes them.  With those
// counts the init kernel resolves every target whose rank lies in the run of zeros before
// any pass, and a problem with both targets resolved is never read.
#include <cmath>

#include "gem_internal.h"
#include "pdl.h"

namespace gem {
namespace {

constexpr int kThreads = 256;
constexpr int kBins = 2048;                 // 11-bit digits (the last pass uses 1024)
constexpr int kUnroll = 8;                  // independent loads per thread and step
constexpr int kChunk = kThreads * kUnroll * 8;   // elements per histogram block
constexpr int kPasses = 3;
constexpr int kState = 6;                   // per problem: two (prefix, mask, rank)
constexpr unsigned kZeroKey = 0x80000000u;  // order_key(+0.0f)

__host__ __device__ constexpr int digit_shift(int pass) { return pass == 0 ? 21 : (pass == 1 ? 10 : 0); }
__host__ __device__ constexpr int digit_bits(int pass) { return pass == 2 ? 10 : 11; }

struct SelectArgs {
  const float* pi[kMaxPiBatch];             // row k: P floats
  long long seg[kMaxPiSegments + 1];        // segment offsets, shared by all rows
  int block_start[kMaxPiSegments + 1];      // first histogram block of each segment
  int K, nseg, pass;
  unsigned* hist;                           // [K][nseg][2][kBins]
  unsigned* state;                          // [K][nseg][kState]: 2 x (prefix, mask, rank)
  const unsigned* counts;                   // [K][nseg][2]: factors below +0, equal to +0; or null
  float* lo;                                // [K][nseg]
  float* hi;                                // [K][nseg]
};

// Unsigned order of the keys equals the order of the floats (-0 below +0, NaNs outermost).
__device__ __forceinline__ unsigned order_key(float x) {
  const unsigned u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float key_value(unsigned k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

__global__ void select_init_kernel(const __grid_constant__ SelectArgs a) {
  gem::pdl_entry();
  const int q = blockIdx.x * blockDim.x + threadIdx.x;     // problem k * nseg + s
  if (q >= a.K * a.nseg) return;
  const int s = q % a.nseg;
  const long long N = a.seg[s + 1] - a.seg[s];
  unsigned* st = a.state + size_t(q) * kState;
  st[0] = 0u;
  st[1] = 0u;
  st[2] = N > 0 ? unsigned((N - 1) / 2) : 0u;
  st[3] = 0u;
  st[4] = 0u;
  st[5] = unsigned(N / 2);
  if (a.counts && N > 0) {
    // elements below +0 come first in the order, then the run of +0: a target whose rank
    // falls in that run is +0, resolved without a pass
    const unsigned below = a.counts[2 * q], zeros = a.counts[2 * q + 1];
    for (int t = 0; t < 2; ++t) {
      const unsigned r = st[3 * t + 2];
      if (r >= below && r - below < zeros) {
        st[3 * t] = kZeroKey;
        st[3 * t + 1] = 0xffffffffu;
        st[3 * t + 2] = r - below;
        (t == 0 ? a.lo : a.hi)[q] = 0.0f;
      }
    }
  }
}

// Counts of a fused commit: clears them and stores the segment offsets where the commit
// kernel reads them.
struct CountInitArgs {
  unsigned* counts;                         // [K][nseg][2]
  int words;
  long long* seg_dev;                       // [nseg + 1]
  long long seg[kMaxPiSegments + 1];
  int nseg;
};

__global__ void count_init_kernel(const __grid_constant__ CountInitArgs a) {
  gem::pdl_entry();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < a.words) a.counts[i] = 0u;
  if (i <= a.nseg) a.seg_dev[i] = a.seg[i];
}

// Adds one element's digit to a shared histogram when its key matches the prefix; every
// lane of the warp must call it (the match is warp-wide).  FIRST: the first pass, whose
// prefix is empty, so that every element matches.
template <bool FIRST>
__device__ __forceinline__ void count_digit(unsigned* h, bool valid, unsigned key, unsigned prefix,
                                            unsigned mask, unsigned digit, int lane) {
  const unsigned bin = (valid && (FIRST || (key & mask) == prefix)) ? digit : 0xffffffffu;
  const unsigned peers = __match_any_sync(0xffffffffu, bin);
  if (bin != 0xffffffffu && lane == __ffs(peers) - 1) atomicAdd(h + bin, unsigned(__popc(peers)));
}

template <bool FIRST>
__global__ void __launch_bounds__(kThreads) select_hist_kernel(const __grid_constant__ SelectArgs a) {
  gem::pdl_entry();
  __shared__ unsigned h[2 * kBins];
  const int b = blockIdx.x, k = blockIdx.y;
  int s = 0;
  while (b >= a.block_start[s + 1]) ++s;
  const int q = k * a.nseg + s;
  const unsigned* st = a.state + size_t(q) * kState;
  const unsigned p0 = st[0], m0 = st[1], p1 = st[3], m1 = st[4];
  const bool done0 = m0 == 0xffffffffu, done1 = m1 == 0xffffffffu;
  if (done0 && done1) return;               // both targets resolved: nothing to count
  const bool two = p0 != p1 || m0 != m1;
  const bool need0 = !done0, need1 = two && !done1;
  for (int i = threadIdx.x; i < 2 * kBins; i += kThreads) h[i] = 0u;
  __syncthreads();

  const int shift = digit_shift(a.pass);
  const unsigned dmask = (1u << digit_bits(a.pass)) - 1u;
  const long long beg = a.seg[s] + (long long)(b - a.block_start[s]) * kChunk;
  const long long end = beg + kChunk < a.seg[s + 1] ? beg + kChunk : a.seg[s + 1];
  const float* x = a.pi[k];
  const int lane = threadIdx.x & 31;
  // the loop bounds are uniform across the block, so whole warps reach count_digit
  for (long long base = beg; base < end; base += kThreads * kUnroll) {
    unsigned key[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const long long i = base + u * kThreads + threadIdx.x;
      key[u] = i < end ? order_key(x[i]) : 0u;
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const bool valid = base + u * kThreads + threadIdx.x < end;
      const unsigned d = (key[u] >> shift) & dmask;
      if (FIRST) {
        count_digit<true>(h, valid, key[u], 0u, 0u, key[u] == kZeroKey ? unsigned(kBins) : d, lane);
      } else {
        if (need0) count_digit<false>(h, valid, key[u], p0, m0, d, lane);
        if (need1) count_digit<false>(h + kBins, valid, key[u], p1, m1, d, lane);
      }
    }
  }
  __syncthreads();
  unsigned* g = a.hist + size_t(q) * 2 * kBins;
  const int used = FIRST ? kBins + 1 : (two ? 2 * kBins : kBins);
  for (int i = threadIdx.x; i < used; i += kThreads) {
    const unsigned c = h[i];
    if (c) atomicAdd(g + i, c);
  }
}

__global__ void __launch_bounds__(kThreads) select_pick_kernel(const __grid_constant__ SelectArgs a) {
  gem::pdl_entry();
  constexpr int kPer = kBins / kThreads;     // bins per thread (8)
  __shared__ unsigned wsum[kThreads / 32];
  __shared__ unsigned sst[kState];
  __shared__ unsigned zeros;                // first pass: elements equal to +0
  const int q = blockIdx.x;
  const int s = q % a.nseg;
  const long long N = a.seg[s + 1] - a.seg[s];
  unsigned* st = a.state + size_t(q) * kState;
  unsigned* g = a.hist + size_t(q) * 2 * kBins;
  if (threadIdx.x < kState) sst[threadIdx.x] = st[threadIdx.x];
  if (threadIdx.x == 0) zeros = a.pass == 0 ? g[kBins] : 0u;
  __syncthreads();
  const int zero_bin = int(kZeroKey >> digit_shift(0));   // +0's first-pass bin
  // the first pass fills one histogram for both targets (a target resolved by the fused
  // counts is skipped below, so their prefixes may differ then)
  const bool two = a.pass > 0 && (sst[0] != sst[3] || sst[1] != sst[4]);
  const int shift = digit_shift(a.pass);
  const unsigned nb = 1u << digit_bits(a.pass);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  for (int t = 0; t < 2; ++t) {
    const unsigned* hh = g + (two ? t : 0) * kBins;
    unsigned local[kPer];
    unsigned sum = 0;
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      local[j] = hh[threadIdx.x * kPer + j];
      if (a.pass == 0 && threadIdx.x * kPer + j == zero_bin) local[j] += zeros;   // counted apart
      sum += local[j];
    }
    unsigned incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const unsigned v = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += v;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    unsigned before = 0;
    for (int w = 0; w < warp; ++w) before += wsum[w];
    const unsigned excl = before + incl - sum;
    const unsigned r = sst[3 * t + 2];
    const bool active = sst[3 * t + 1] != 0xffffffffu;   // not resolved in an earlier pass
    if (active && N > 0 && r >= excl && r - excl < sum) {
      unsigned c = excl;
      int d = 0;
#pragma unroll
      for (int j = 0; j < kPer; ++j) {
        if (r - c < local[j]) {
          d = threadIdx.x * kPer + j;
          break;
        }
        c += local[j];
      }
      if (a.pass == 0 && d == zero_bin && r - c < zeros) {
        // +0 is the smallest key of its bin, so the bin's first `zeros` ranks are exact
        // zeros: the target is +0, resolved now
        st[3 * t] = kZeroKey;
        st[3 * t + 1] = 0xffffffffu;
        st[3 * t + 2] = r - c;
        (t == 0 ? a.lo : a.hi)[q] = 0.0f;
      } else {
        const unsigned prefix = sst[3 * t] | (unsigned(d) << shift);
        st[3 * t] = prefix;
        st[3 * t + 1] = sst[3 * t + 1] | ((nb - 1u) << shift);
        st[3 * t + 2] = r - c;
        if (a.pass == kPasses - 1) (t == 0 ? a.lo : a.hi)[q] = key_value(prefix);
      }
    }
    __syncthreads();   // wsum is reused by the next target
  }
  for (int i = threadIdx.x; i < 2 * kBins; i += kThreads) g[i] = 0u;
  if (N == 0 && a.pass == kPasses - 1 && threadIdx.x == 0) {
    a.lo[q] = __int_as_float(0x7fc00000);
    a.hi[q] = __int_as_float(0x7fc00000);
  }
}

}  // namespace

namespace {

// The handle's select scratch for chunks of up to kc rows of nseg segments: histograms,
// per-problem state, factor counts and the segment offsets (grown on demand).
struct SelectScratch {
  unsigned* hist;
  unsigned* state;
  unsigned* counts;
  long long* seg;
};

cudaError_t select_scratch(gem_ctx* h, int kc, int nseg, SelectScratch* out) {
  const size_t problems = size_t(kc) * nseg;
  const size_t hist_bytes = problems * 2 * kBins * sizeof(unsigned);
  const size_t state_bytes = problems * kState * sizeof(unsigned);
  const size_t count_bytes = (problems * 2 * sizeof(unsigned) + 15) / 16 * 16;
  const size_t seg_bytes = size_t(kMaxPiSegments + 1) * sizeof(long long);
  const size_t need = hist_bytes + state_bytes + count_bytes + seg_bytes;
  if (need > h->select_bytes) {
    cudaFree(h->select_scratch);   // waits for work still using the old buffer
    h->select_scratch = nullptr;
    h->select_bytes = 0;
    cudaError_t e = cudaMalloc(&h->select_scratch, need);
    if (e != cudaSuccess) return e;
    h->select_bytes = need;
  }
  char* base = static_cast<char*>(h->select_scratch);
  out->hist = reinterpret_cast<unsigned*>(base);
  out->state = reinterpret_cast<unsigned*>(base + hist_bytes);
  out->counts = reinterpret_cast<unsigned*>(base + hist_bytes + state_bytes);
  out->seg = reinterpret_cast<long long*>(base + hist_bytes + state_bytes + count_bytes);
  return cudaSuccess;
}

// Segment offsets and histogram blocks of a select.
int prepare_args(SelectArgs& a, const int64_t* seg, int nseg) {
  a.nseg = nseg;
  a.block_start[0] = 0;
  for (int s = 0; s <= nseg; ++s) a.seg[s] = seg[s];
  for (int s = 0; s < nseg; ++s) {
    const long long N = seg[s + 1] - seg[s];
    a.block_start[s + 1] = a.block_start[s] + int((N + kChunk - 1) / kChunk);
  }
  return a.block_start[nseg];
}

// The select of rows a.pi[0 .. kc) (a.lo, a.hi, a.counts set by the caller).
cudaError_t select_rows(gem_ctx* h, SelectArgs& a, int kc, int blocks) {
  a.K = kc;
  a.pass = 0;
  cudaError_t e = cudaMemsetAsync(a.hist, 0, size_t(kc) * a.nseg * 2 * kBins * sizeof(unsigned),
                                  h->stream);
  if (e != cudaSuccess) return e;
  gem::launch_pdl(select_init_kernel, (kc * a.nseg + 127) / 128, 128, 0, h->stream, a);
  h->launches += 1;
  for (int p = 0; p < kPasses; ++p) {
    a.pass = p;
    if (blocks > 0) {
      if (p == 0)
        gem::launch_pdl(select_hist_kernel<true>, dim3(unsigned(blocks), unsigned(kc)), kThreads, 0, h->stream, a);
      else
        gem::launch_pdl(select_hist_kernel<false>, dim3(unsigned(blocks), unsigned(kc)), kThreads, 0, h->stream, a);
      h->launches += 1;
    }
    gem::launch_pdl(select_pick_kernel, unsigned(kc * a.nseg), kThreads, 0, h->stream, a);
    h->launches += 1;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t pi_median_ordered(gem_ctx* h, const float* const* pi, int K, const int64_t* seg,
                              int nseg, float* lo, float* hi) {
  if (K <= 0) return cudaSuccess;
  const int kc_max = K < kMaxPiBatch ? K : kMaxPiBatch;
  SelectScratch sc;
  cudaError_t e = select_scratch(h, kc_max, nseg, &sc);
  if (e != cudaSuccess) return e;
  SelectArgs a;
  const int blocks = prepare_args(a, seg, nseg);
  a.hist = sc.hist;
  a.state = sc.state;
  a.counts = nullptr;
  for (int k0 = 0; k0 < K; k0 += kMaxPiBatch) {
    const int kc = (K - k0) < kMaxPiBatch ? (K - k0) : kMaxPiBatch;
    for (int k = 0; k < kc; ++k) a.pi[k] = pi[k0 + k];
    a.lo = lo + size_t(k0) * nseg;
    a.hi = hi + size_t(k0) * nseg;
    e = select_rows(h, a, kc, blocks);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t commit_pi_median_ordered(gem_ctx* h, const int* order, const float* const* grads,
                                     int K, float* const* pi, const int64_t* seg, int nseg,
                                     float* lo, float* hi) {
  if (K <= 0) return cudaSuccess;
  // commits per chunk: one commit launch, one select, and the counters in shared memory
  int per = kMaxCountWords / (2 * nseg);
  if (per > kMaxBatchPerLaunch) per = kMaxBatchPerLaunch;
  if (per > kMaxPiBatch) per = kMaxPiBatch;
  const int kc_max = K < per ? K : per;
  SelectScratch sc;
  cudaError_t e = select_scratch(h, kc_max, nseg, &sc);
  if (e != cudaSuccess) return e;
  SelectArgs a;
  const int blocks = prepare_args(a, seg, nseg);
  a.hist = sc.hist;
  a.state = sc.state;
  a.counts = sc.counts;
  CountInitArgs ci;
  ci.counts = sc.counts;
  ci.seg_dev = sc.seg;
  ci.nseg = nseg;
  for (int s = 0; s <= nseg; ++s) ci.seg[s] = seg[s];
  for (int k0 = 0; k0 < K; k0 += per) {
    const int kc = (K - k0) < per ? (K - k0) : per;
    ci.words = kc * nseg * 2;
    const int n_init = ci.words > nseg + 1 ? ci.words : nseg + 1;
    gem::launch_pdl(count_init_kernel, (n_init + 255) / 256, 256, 0, h->stream, ci);
    h->launches += 1;
    e = commit_ordered(h, order + k0, grads + k0, kc, pi + k0, sc.counts, sc.seg, nseg);
    if (e != cudaSuccess) return e;
    for (int k = 0; k < kc; ++k) a.pi[k] = pi[k0 + k];
    a.lo = lo + size_t(k0) * nseg;
    a.hi = hi + size_t(k0) * nseg;
    e = select_rows(h, a, kc, blocks);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace gem
