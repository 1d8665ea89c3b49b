// Fused GEM commit kernel (Algorithm 1: Psi_GEM, Commit, and the worker's next pull).
//
// Every step of a commit is elementwise over the P coordinates (the scaling factor pi is
// a per-parameter vector, applied with a Hadamard product), so coordinate j of theta,
// m_w and s_w depends only on coordinate j of the gradients.  The kernel therefore
// gives each thread a few 16-byte lanes of coordinates and walks *all* commits of the
// launch, in order, on those lanes: commit order is preserved without any lock or
// inter-block communication, repeated workers inside a batch see their own earlier
// results by program order, and theta stays in registers across the batch (read and
// written once per launch instead of once per commit).
//
// Per coordinate and commit the kernel streams 12 bytes in (g, m_w, s_w) and 8 bytes
// out (m_w, s_w); theta adds 8 bytes per launch.  The path is HBM-bound (about 0.5 flop
// per byte), so the design goals are coalesced 128-bit accesses and enough independent
// loads in flight per SM (one 16-byte lane per thread, 512 threads per block).  The
// gradients are read with an evict-first hint (a gradient is used once per batch); the
// rows of m_w and s_w are cached normally, so a worker that commits again a few commits
// later in the same batch finds them in L2 and DRAM traffic drops below the algorithmic
// 20 bytes per parameter and commit.
#include "gem_internal.h"

// Launch shape: threads per block, 16-byte lanes per thread, and a minimum number of
// resident blocks per SM (0: let the compiler choose registers freely).
#ifndef GEM_COMMIT_THREADS
#define GEM_COMMIT_THREADS 512
#endif
#ifndef GEM_COMMIT_LANES
#define GEM_COMMIT_LANES 1
#endif
#ifndef GEM_COMMIT_MIN_BLOCKS
#define GEM_COMMIT_MIN_BLOCKS 0
#endif
// Cache policy of the moment and snapshot rows: 1 streams them (evict-first), 0 caches them
// normally so that a worker that commits again soon finds its rows in L2.
#ifndef GEM_COMMIT_STREAM_STATE
#define GEM_COMMIT_STREAM_STATE 0
#endif
// Resident blocks per SM used to size the grid, at most (0: as many as fit).
#ifndef GEM_COMMIT_MAX_BLOCKS_PER_SM
#define GEM_COMMIT_MAX_BLOCKS_PER_SM 0
#endif

namespace gem {
namespace {

constexpr int kThreads = GEM_COMMIT_THREADS;

// One coordinate of one commit.  One IEEE fp32 operation per step, rounded to nearest,
// no contraction into FMA (the __f*_rn intrinsics are never fused), IEEE division.
// RULE kRuleGem takes |m_w| as the root of twice the proxy energy (Eq. proxy_estimate);
// kRuleScaled multiplies it by `scale` first (sqrt(kappa) or kappa, App. B).
template <int RULE>
__device__ __forceinline__ float commit_coord(float& theta, float& m, float& s, float g,
                                              float eta, float mu, float eps, float scale) {
  const float dtheta = -__fmul_rn(eta, g);                       // -eta grad L(s)
  const float m_new = __fadd_rn(__fmul_rn(mu, m), dtheta);       // m <- mu m + dtheta
  const float drift = fabsf(__fsub_rn(theta, s));                // |theta - s|
  const float energy = RULE == kRuleScaled ? __fmul_rn(scale, fabsf(m_new)) : fabsf(m_new);
  float pi = __fdiv_rn(__fsub_rn(energy, drift),                 // (|m| - |theta - s|)
                       __fadd_rn(fabsf(dtheta), eps));           //   / (|dtheta| + eps)
  pi = pi > 0.0f ? pi : 0.0f;                                    // pi >= 0
  theta = __fadd_rn(theta, __fmul_rn(pi, dtheta));               // theta + pi dtheta
  m = m_new;
  s = theta;                                                     // s <- theta
  return pi;
}

// A commit with a given scaling factor (kRuleFixed): theta + pi dtheta, s <- theta; the
// moment is not part of these rules.
__device__ __forceinline__ void commit_coord_fixed(float& theta, float& s, float g, float eta,
                                                   float pi) {
  const float dtheta = -__fmul_rn(eta, g);
  theta = __fadd_rn(theta, __fmul_rn(pi, dtheta));
  s = theta;
}

__device__ __forceinline__ float4 load_state(const float4* p) {
#if GEM_COMMIT_STREAM_STATE
  return __ldcs(p);
#else
  return *p;
#endif
}

__device__ __forceinline__ void store_state(float4* p, float4 v) {
#if GEM_COMMIT_STREAM_STATE
  __stcs(p, v);
#else
  *p = v;
#endif
}

// A store of m_w or s_w with the launch's L2 policy for it: kept in L2 ahead of other lines
// (evict-last, `keep` the access policy made by createpolicy) when a later commit of the
// launch reads it back, streamed (evict-first) at the worker's last commit of the launch.
__device__ __forceinline__ void store_state_hint(float4* p, float4 v, int hint, uint64_t keep) {
  if (hint == kL2Keep) {
    asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x),
                 "f"(v.y), "f"(v.z), "f"(v.w), "l"(keep)
                 : "memory");
  } else if (hint == kL2Stream) {
    __stcs(p, v);
  } else {
    store_state(p, v);
  }
}

// The momentum-SGD proxy committed as is (Eq. momentum_update): m <- mu m + dtheta,
// theta <- theta + m, s <- theta.
__device__ __forceinline__ void commit_coord_momentum(float& theta, float& m, float& s, float g,
                                                      float eta, float mu) {
  const float dtheta = -__fmul_rn(eta, g);
  m = __fadd_rn(__fmul_rn(mu, m), dtheta);
  theta = __fadd_rn(theta, m);
  s = theta;
}

// Segment s with seg[s] <= j < seg[s + 1] (the last such s when segments are empty), or -1
// when j lies outside [seg[0], seg[nseg]).
__device__ __forceinline__ int segment_of(const long long* seg, int nseg, long long j) {
  if (j < seg[0] || j >= seg[nseg]) return -1;
  int lo = 0, hi = nseg;   // seg[lo] <= j < seg[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (seg[mid] <= j) lo = mid;
    else hi = mid;
  }
  return lo;
}

// Factors below +0 (sign bit set: negatives, -0, negative NaN) and equal to +0.
__device__ __forceinline__ void count_factor(float x, unsigned& below, unsigned& zero) {
  const unsigned u = __float_as_uint(x);
  below += u >> 31;
  zero += u == 0u ? 1u : 0u;
}

template <int RULE>
__device__ __forceinline__ float4 commit_vec(float4& th, float4& m, float4& s, const float4 g,
                                             float eta, float mu, float eps, float scale) {
  float4 pi;
  pi.x = commit_coord<RULE>(th.x, m.x, s.x, g.x, eta, mu, eps, scale);
  pi.y = commit_coord<RULE>(th.y, m.y, s.y, g.y, eta, mu, eps, scale);
  pi.z = commit_coord<RULE>(th.z, m.z, s.z, g.z, eta, mu, eps, scale);
  pi.w = commit_coord<RULE>(th.w, m.w, s.w, g.w, eta, mu, eps, scale);
  return pi;
}

__device__ __forceinline__ void commit_vec_fixed(float4& th, float4& s, const float4 g, float eta,
                                                 float pi) {
  commit_coord_fixed(th.x, s.x, g.x, eta, pi);
  commit_coord_fixed(th.y, s.y, g.y, eta, pi);
  commit_coord_fixed(th.z, s.z, g.z, eta, pi);
  commit_coord_fixed(th.w, s.w, g.w, eta, pi);
}

// L independent 16-byte lanes per thread, strided by the grid so that each warp
// touches 512 contiguous bytes per lane and array.  The fixed-factor rules read only the
// gradient and write only s_w (12 bytes less per coordinate and commit).
// The scaled rule asks for two resident blocks per SM: left free, the compiler fits it in
// 40 registers for three blocks and spills, which costs about 4% of its bandwidth.  The
// energy rules' launches of more than kSmallBatch commits also carry the register slot and
// ask for two blocks (at most 64 registers); the smaller launches keep the compiler's
// choice, which measured faster for single commits.
// REC: the commits whose pi_out[k] is set also store their scaling factors there (4 more
// bytes per coordinate), and with pi_counts set count them per segment (factors below +0
// and equal to +0): per warp with one reduction, into the block's counters in shared
// memory, added to pi_counts when the block ends.  The lane loop of these launches runs
// while any lane of the warp has coordinates, so the warp reductions see every lane.
// A worker that commits again later in the launch can keep its m_w, s_w lanes on chip:
// each thread owns lanes slot_mem[(2 slot + {0: m, 1: s}) L kThreads + l kThreads + tid]
// of dynamic shared memory, so no synchronisation is needed.
template <int L, int RULE, bool REC, int KCAP>
__global__ void __launch_bounds__(kThreads, (RULE == kRuleScaled || (RULE != kRuleFixed && KCAP > kSmallBatch))
                                                 ? 2 : GEM_COMMIT_MIN_BLOCKS)
commit_batch_kernel(const __grid_constant__ BatchArgsT<KCAP> a) {
  extern __shared__ float4 slot_mem[];
  // Launched as a programmatic dependent of the previous kernel in the stream: wait until
  // that grid has completed and its writes are visible (theta, m_w and s_w may be the ones
  // it wrote).  The next launch is scheduled when this grid's blocks have exited.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const size_t nvec = a.P >> 2;
  const size_t nthreads = size_t(gridDim.x) * kThreads;
  const size_t tid = size_t(blockIdx.x) * kThreads + threadIdx.x;
  float4* theta4 = reinterpret_cast<float4*>(a.theta);
  const unsigned lane = threadIdx.x & 31u;
  // L2 hints on the stores of m_w and s_w: launches of more than kSmallBatch commits
  constexpr bool kHints = KCAP > kSmallBatch && RULE != kRuleFixed;
  uint64_t keep_policy = 0;
  if constexpr (kHints)
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep_policy));
  // factor counters of this block (recording launches with counts only)
  unsigned* cnt = nullptr;
  if constexpr (REC) {
    if (a.pi_counts) {
      cnt = reinterpret_cast<unsigned*>(slot_mem + a.count_smem_at);
      for (int q = threadIdx.x; q < a.K * a.pi_nseg * 2; q += kThreads) cnt[q] = 0u;
      __syncthreads();
    }
  }
  auto slot_m = [&](int slot, int l) -> float4& {
    return slot_mem[(2 * slot) * L * kThreads + l * kThreads + threadIdx.x];
  };
  auto slot_s = [&](int slot, int l) -> float4& {
    return slot_mem[(2 * slot + 1) * L * kThreads + l * kThreads + threadIdx.x];
  };

  for (size_t base = tid; (REC ? base - lane : base) < nvec; base += nthreads * L) {
    float4 th[L];
    // segment of each lane's four coordinates: >= 0 one segment, -1 outside every segment
    // (or no coordinates), -2 the four straddle a boundary; uni: the warp's lanes share one
    int sid[L];
    bool uni[L];
    if constexpr (REC) {
#pragma unroll
      for (int l = 0; l < L; ++l) {
        const size_t i = base + size_t(l) * nthreads;
        sid[l] = -1;
        if (cnt && i < nvec) {
          sid[l] = segment_of(a.pi_seg, a.pi_nseg, (long long)(4 * i));
          if (segment_of(a.pi_seg, a.pi_nseg, (long long)(4 * i + 3)) != sid[l]) sid[l] = -2;
        }
        uni[l] = __all_sync(0xffffffffu, sid[l] == __shfl_sync(0xffffffffu, sid[l], 0));
      }
    }
    // Register slots, in launches of more than kSmallBatch commits only (smaller launches
    // are planned without them, and compile to the shared-memory slots alone); get / put
    // reach a slot by its id, the register slots through static indices.
    constexpr int kR = KCAP > kSmallBatch ? kRegSlots : 0;
    float4 rm[kR > 0 ? kR : 1][L], rs[kR > 0 ? kR : 1][L];
    auto get = [&](int sid, int l, float4& mv, float4* sv) {
      if (sid < kCommitSlots) {
        mv = slot_m(sid, l);
        if (sv) *sv = slot_s(sid, l);
        return;
      }
#pragma unroll
      for (int r = 0; r < kR; ++r)
        if (sid == kCommitSlots + r) {
          mv = rm[r][l];
          if (sv) *sv = rs[r][l];
        }
    };
    auto put = [&](int sid, int l, const float4& mv, const float4* sv) {
      if (sid < kCommitSlots) {
        slot_m(sid, l) = mv;
        if (sv) slot_s(sid, l) = *sv;
        return;
      }
#pragma unroll
      for (int r = 0; r < kR; ++r)
        if (sid == kCommitSlots + r) {
          rm[r][l] = mv;
          if (sv) rs[r][l] = *sv;
        }
    };
#pragma unroll
    for (int l = 0; l < L; ++l) {
      const size_t i = base + size_t(l) * nthreads;
      if (i < nvec) th[l] = theta4[i];
    }
    for (int k = 0; k < a.K; ++k) {
      const float4* g4 = reinterpret_cast<const float4*>(a.grad[k]);
      const size_t row = size_t(a.worker[k]) * a.stride;
      float4* m4 = reinterpret_cast<float4*>(a.m + row);
      float4* s4 = reinterpret_cast<float4*>(a.s + row);
      const int sin = a.slot_in[k], sout = a.slot_out[k];
      float4 g[L], m[L], s[L];
      float4 pi_l[L];   // the factors of this commit (recording launches)
#pragma unroll
      for (int l = 0; l < L; ++l) {
        const size_t i = base + size_t(l) * nthreads;
        if (i < nvec) {
          g[l] = __ldcs(g4 + i);
          if (RULE == kRuleMomentum) {
            if constexpr (kR > 0) {
              if (sin >= 0) get(sin, l, m[l], nullptr);
              else m[l] = load_state(m4 + i);
            } else {
              m[l] = sin >= 0 ? slot_m(sin, l) : load_state(m4 + i);
            }
          } else if (RULE != kRuleFixed) {
            if (sin >= 0) {
              if constexpr (kR > 0) {
                get(sin, l, m[l], &s[l]);
              } else {
                m[l] = slot_m(sin, l);
                s[l] = slot_s(sin, l);
              }
            } else {
              m[l] = load_state(m4 + i);
              s[l] = load_state(s4 + i);
            }
          }
        }
      }
#pragma unroll
      for (int l = 0; l < L; ++l) {
        const size_t i = base + size_t(l) * nthreads;
        if (i < nvec) {
          float4 pi;
          if (RULE == kRuleFixed) {
            commit_vec_fixed(th[l], s[l], g[l], a.eta, a.pi[k]);
            pi = make_float4(a.pi[k], a.pi[k], a.pi[k], a.pi[k]);
            if (a.keep_s[k]) store_state(s4 + i, s[l]);
          } else if (RULE == kRuleMomentum) {
            commit_coord_momentum(th[l].x, m[l].x, s[l].x, g[l].x, a.eta, a.mu);
            commit_coord_momentum(th[l].y, m[l].y, s[l].y, g[l].y, a.eta, a.mu);
            commit_coord_momentum(th[l].z, m[l].z, s[l].z, g[l].z, a.eta, a.mu);
            commit_coord_momentum(th[l].w, m[l].w, s[l].w, g[l].w, a.eta, a.mu);
            const float nan = __int_as_float(0x7fc00000);
            pi = make_float4(nan, nan, nan, nan);
            if constexpr (kR > 0) {
              if (sout >= 0) put(sout, l, m[l], nullptr);
              else if constexpr (kHints) store_state_hint(m4 + i, m[l], a.l2[k], keep_policy);
              else store_state(m4 + i, m[l]);
            } else {
              if (sout >= 0) slot_m(sout, l) = m[l];
              else store_state(m4 + i, m[l]);
            }
            if (a.keep_s[k]) store_state(s4 + i, s[l]);
          } else {
            pi = commit_vec<RULE>(th[l], m[l], s[l], g[l], a.eta, a.mu, a.eps, a.energy_scale);
            if (sout >= 0) {
              if constexpr (kR > 0) {
                put(sout, l, m[l], &s[l]);
              } else {
                slot_m(sout, l) = m[l];
                slot_s(sout, l) = s[l];
              }
            } else if constexpr (kHints) {
              store_state_hint(m4 + i, m[l], a.l2[k], keep_policy);
              store_state_hint(s4 + i, s[l], a.l2[k], keep_policy);
            } else {
              store_state(m4 + i, m[l]);
              store_state(s4 + i, s[l]);
            }
          }
          if (REC && a.pi_out[k]) reinterpret_cast<float4*>(a.pi_out[k])[i] = pi;
          if constexpr (REC) pi_l[l] = pi;
        }
      }
      if constexpr (REC) {
        if (cnt && a.pi_out[k]) {
#pragma unroll
          for (int l = 0; l < L; ++l) {
            const size_t i = base + size_t(l) * nthreads;
            unsigned below = 0u, zero = 0u;
            if (i < nvec && sid[l] != -1) {
              count_factor(pi_l[l].x, below, zero);
              count_factor(pi_l[l].y, below, zero);
              count_factor(pi_l[l].z, below, zero);
              count_factor(pi_l[l].w, below, zero);
            }
            if (uni[l]) {
              // one segment (or none) for the whole warp: one reduction, one lane adds
              below = __reduce_add_sync(0xffffffffu, below);
              zero = __reduce_add_sync(0xffffffffu, zero);
              if (lane == 0 && sid[l] >= 0) {
                unsigned* c = cnt + 2 * (k * a.pi_nseg + sid[l]);
                if (below) atomicAdd(c, below);
                if (zero) atomicAdd(c + 1, zero);
              }
            } else if (sid[l] >= 0) {
              unsigned* c = cnt + 2 * (k * a.pi_nseg + sid[l]);
              if (below) atomicAdd(c, below);
              if (zero) atomicAdd(c + 1, zero);
            } else if (sid[l] == -2) {
              // the four coordinates straddle a segment boundary: one by one
              const float v[4] = {pi_l[l].x, pi_l[l].y, pi_l[l].z, pi_l[l].w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int se = segment_of(a.pi_seg, a.pi_nseg, (long long)(4 * i + e));
                unsigned b1 = 0u, z1 = 0u;
                count_factor(v[e], b1, z1);
                if (se >= 0 && (b1 | z1)) atomicAdd(cnt + 2 * (k * a.pi_nseg + se) + (b1 ? 0 : 1), 1u);
              }
            }
          }
        }
      }
    }
#pragma unroll
    for (int l = 0; l < L; ++l) {
      const size_t i = base + size_t(l) * nthreads;
      if (i < nvec) theta4[i] = th[l];
    }
  }

  // Ragged tail: the last P mod 4 coordinates, one thread each, scalar accesses (the
  // caller's gradient holds exactly P floats).
  const size_t tail0 = nvec << 2;
  if (tid < a.P - tail0) {
    const size_t j = tail0 + tid;
    float th = a.theta[j];
    for (int k = 0; k < a.K; ++k) {
      const size_t row = size_t(a.worker[k]) * a.stride;
      float s, pi;
      if (RULE == kRuleFixed) {
        commit_coord_fixed(th, s, a.grad[k][j], a.eta, a.pi[k]);
        pi = a.pi[k];
      } else if (RULE == kRuleMomentum) {
        float m = a.m[row + j];
        commit_coord_momentum(th, m, s, a.grad[k][j], a.eta, a.mu);
        a.m[row + j] = m;
        pi = __int_as_float(0x7fc00000);
      } else {
        float m = a.m[row + j];
        s = a.s[row + j];
        pi = commit_coord<RULE>(th, m, s, a.grad[k][j], a.eta, a.mu, a.eps, a.energy_scale);
        a.m[row + j] = m;
      }
      a.s[row + j] = s;
      if (REC && a.pi_out[k]) {
        a.pi_out[k][j] = pi;
        if (cnt) {
          const int se = segment_of(a.pi_seg, a.pi_nseg, (long long)j);
          unsigned b1 = 0u, z1 = 0u;
          count_factor(pi, b1, z1);
          if (se >= 0 && (b1 | z1)) atomicAdd(cnt + 2 * (k * a.pi_nseg + se) + (b1 ? 0 : 1), 1u);
        }
      }
    }
    a.theta[j] = th;
  }
  if constexpr (REC) {
    if (cnt) {
      __syncthreads();
      for (int q = threadIdx.x; q < a.K * a.pi_nseg * 2; q += kThreads)
        if (cnt[q]) atomicAdd(a.pi_counts + q, cnt[q]);
    }
  }
}

constexpr int kLanes = GEM_COMMIT_LANES;

// One launch of the kernel instantiation for KCAP commits.  The slot shared memory is
// requested only when the launch keeps a worker on chip; without it more blocks fit on an
// SM.  Occupancy is computed once per instantiation and shared-memory size.
template <int RULE, bool REC, int KCAP>
cudaError_t launch_kernel(BatchArgsT<KCAP> a, bool slots, int sm_count, cudaStream_t stream) {
  const int slot_bytes = slots ? kCommitSlots * 2 * kLanes * kThreads * 16 : 0;
  // factor counters after the slots, in whole float4 (recording launches with counts)
  const int count_bytes = (REC && a.pi_counts) ? (a.K * a.pi_nseg * 2 * 4 + 15) / 16 * 16 : 0;
  a.count_smem_at = slot_bytes / 16;
  const int smem = slot_bytes + count_bytes;
  static int blocks_per_sm[2] = {0, 0};
  int counted_bps = 0;
  int& bps = count_bytes ? counted_bps : blocks_per_sm[slots ? 1 : 0];
  if (bps == 0) {
    static bool attr_set = false;
    if (!attr_set) {
      // the most any launch of this instantiation asks for: every slot and the largest
      // counter block
      const int most = kCommitSlots * 2 * kLanes * kThreads * 16 + (REC ? kMaxCountWords * 4 : 0);
      if (most > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(commit_batch_kernel<kLanes, RULE, REC, KCAP>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, most);
        if (e != cudaSuccess) return e;
      }
      attr_set = true;
    }
    int b = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &b, commit_batch_kernel<kLanes, RULE, REC, KCAP>, kThreads, smem);
    if (e != cudaSuccess) return e;
    if (GEM_COMMIT_MAX_BLOCKS_PER_SM > 0 && b > GEM_COMMIT_MAX_BLOCKS_PER_SM)
      b = GEM_COMMIT_MAX_BLOCKS_PER_SM;
    bps = b < 1 ? 1 : b;
  }
  const size_t nvec = a.P >> 2;
  const size_t per_block = size_t(kThreads) * kLanes;
  const size_t max_grid = size_t(sm_count) * size_t(bps);
  size_t grid = (nvec + per_block - 1) / per_block;
  if (grid > max_grid) {
    // Same number of rounds per thread as the full resident grid, with the grid trimmed
    // so that the last round is as full as possible.
    const size_t rounds = (nvec + max_grid * per_block - 1) / (max_grid * per_block);
    grid = (nvec + rounds * per_block - 1) / (rounds * per_block);
  }
  if (grid < 1) grid = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = size_t(smem);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, commit_batch_kernel<kLanes, RULE, REC, KCAP>, a);
}

template <int RULE, bool REC>
cudaError_t launch_rule(const BatchArgs& a, int sm_count, cudaStream_t stream) {
  bool slots = false;
  if (RULE != kRuleFixed)
    for (int k = 0; k < a.K; ++k) slots = slots || (a.slot_out[k] >= 0 && a.slot_out[k] < kCommitSlots);
  if (a.K > kSmallBatch) return launch_kernel<RULE, REC, kMaxBatchPerLaunch>(a, slots, sm_count, stream);
  BatchArgsT<kSmallBatch> b;
  b.theta = a.theta;
  b.m = a.m;
  b.s = a.s;
  b.P = a.P;
  b.stride = a.stride;
  b.eta = a.eta;
  b.mu = a.mu;
  b.eps = a.eps;
  b.K = a.K;
  b.rule = a.rule;
  b.energy_scale = a.energy_scale;
  b.record_pi = a.record_pi;
  b.pi_counts = a.pi_counts;
  b.pi_seg = a.pi_seg;
  b.pi_nseg = a.pi_nseg;
  b.count_smem_at = 0;
  for (int k = 0; k < kSmallBatch; ++k) {
    const bool in = k < a.K;
    b.grad[k] = in ? a.grad[k] : nullptr;
    b.worker[k] = in ? a.worker[k] : 0;
    b.pi[k] = in ? a.pi[k] : 0.f;
    b.pi_out[k] = in ? a.pi_out[k] : nullptr;
    b.slot_in[k] = in ? a.slot_in[k] : int8_t(-1);
    b.slot_out[k] = in ? a.slot_out[k] : int8_t(-1);
    b.keep_s[k] = in ? a.keep_s[k] : uint8_t(1);
    b.l2[k] = kL2Normal;   // no hints below kSmallBatch + 1 commits
  }
  return launch_kernel<RULE, REC, kSmallBatch>(b, slots, sm_count, stream);
}

}  // namespace

void plan_slots(BatchArgs& a) {
  // next occurrence of each commit's worker within the launch
  int next[kMaxBatchPerLaunch];
  {
    int last_seen[kMaxBatchPerLaunch];   // commit index per distinct worker, via search
    int seen_worker[kMaxBatchPerLaunch];
    int n_seen = 0;
    for (int k = a.K - 1; k >= 0; --k) {
      next[k] = -1;
      for (int q = 0; q < n_seen; ++q)
        if (seen_worker[q] == a.worker[k]) {
          next[k] = last_seen[q];
          last_seen[q] = k;
          goto found;
        }
      seen_worker[n_seen] = a.worker[k];
      last_seen[n_seen] = k;
      ++n_seen;
    found:;
    }
  }
  for (int k = 0; k < a.K; ++k) {
    a.slot_in[k] = -1;
    a.slot_out[k] = -1;
    a.keep_s[k] = next[k] < 0 ? 1 : 0;
    a.l2[k] = next[k] < 0 ? kL2Stream : kL2Keep;   // a slot below makes it irrelevant
  }
  const int total = a.K > kSmallBatch ? kTotalSlots : kCommitSlots;   // see the kernel
  if (a.rule == kRuleFixed || total == 0) return;
  // Choose repeat intervals (k, next[k]) longer than kSlotMinDistance, at most kTotalSlots
  // (shared-memory and register slots) open at a time, as many as possible: by increasing end, each into the free slot that
  // became free last (greedy, optimal for interval graphs).
  int order[kMaxBatchPerLaunch], cnt = 0;
  for (int k = 0; k < a.K; ++k)
    if (next[k] >= 0 && next[k] - k > kSlotMinDistance) order[cnt++] = k;
  for (int x = 1; x < cnt; ++x)   // insertion sort by end point
    for (int y = x; y > 0 && next[order[y - 1]] > next[order[y]]; --y) {
      const int t = order[y];
      order[y] = order[y - 1];
      order[y - 1] = t;
    }
  int free_at[kTotalSlots > 0 ? kTotalSlots : 1];
  for (int q = 0; q < total; ++q) free_at[q] = -1;
  for (int x = 0; x < cnt; ++x) {
    const int k = order[x], e = next[k];
    int best = -1;
    for (int q = 0; q < total; ++q)
      if (free_at[q] <= k && (best < 0 || free_at[q] > free_at[best])) best = q;
    if (best < 0) continue;
    free_at[best] = e;
    a.slot_out[k] = int8_t(best);
    a.slot_in[e] = int8_t(best);
  }
}

cudaError_t launch_commit_batch(const BatchArgs& a, int sm_count, cudaStream_t stream) {
  if (a.record_pi) {
    switch (a.rule) {
      case kRuleGem: return launch_rule<kRuleGem, true>(a, sm_count, stream);
      case kRuleScaled: return launch_rule<kRuleScaled, true>(a, sm_count, stream);
      case kRuleFixed: return launch_rule<kRuleFixed, true>(a, sm_count, stream);
      case kRuleMomentum: return launch_rule<kRuleMomentum, true>(a, sm_count, stream);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (a.rule) {
    case kRuleGem: return launch_rule<kRuleGem, false>(a, sm_count, stream);
    case kRuleScaled: return launch_rule<kRuleScaled, false>(a, sm_count, stream);
    case kRuleFixed: return launch_rule<kRuleFixed, false>(a, sm_count, stream);
    case kRuleMomentum: return launch_rule<kRuleMomentum, false>(a, sm_count, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace gem
