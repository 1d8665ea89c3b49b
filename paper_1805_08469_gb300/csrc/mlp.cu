// Batched worker gradients of a ReLU MLP over stale snapshots, and the end-to-end
// asynchronous GEM loop built on them (include/gem_sim.h).
//
// A worker computes dtheta = -eta grad L(s) at its snapshot s (notation table; Algorithm
// 1, Worker).  Workers of one segment (distinct workers, see gem_plan_segments) have
// fixed snapshots, so each product of their forward and backward passes is one grouped
// launch over the segment: group g works on worker order[a + g]'s snapshot (weights read
// straight from s_w inside GEM's state) and on slot g of the scratch (activations,
// deltas, gradient).  The gradients are then committed in schedule order by the fused
// commit kernel.
//
// Products per layer l (dims d_l -> d_{l+1}, batch b), all written for row-major storage:
//   forward   Z_l  = A_l W_l^T + b_l     A_l [b x d_l],   W_l [d_{l+1} x d_l]
//   weights   dW_l = D_{l+1}^T A_l       D_{l+1} [b x d_{l+1}]
//   inputs    D_l  = (D_{l+1} W_l) * [A_l > 0]
//   biases    db_l = column sums of D_{l+1} (fixed order, no atomics)
// Every sum runs in a fixed order, so the gradients are deterministic.
//
// Precision.  Every product runs in one grouped SIMT GEMM kernel that reads either operand
// layout; with GEM_MLP_TF32 it rounds each operand to TF32 as it loads it (products of TF32
// values are exact in fp32; the sums stay fp32).
#include <cuda.h>

#include <cstdint>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "../../include/gem_sim.h"
#include "gem_internal.h"
#include "mlp_internal.h"
#include "pdl.h"
#include "tc_gemm.h"

namespace gem {
namespace mlp {


// SIMT tile: 128 (or 64) x 64 outputs per block of 256 (or 128) threads, 8 x 4 per thread,
// k-steps of 16 (also the split-K granularity).
constexpr int BN = 64, BK = 16;
constexpr long long kSmCountHint = 152;  // GB300
#ifndef GEM_MAX_SPLIT
#define GEM_MAX_SPLIT 4
#endif
#ifndef GEM_TF32_MIN_CHUNK
#define GEM_TF32_MIN_CHUNK 64
#endif
#ifndef GEM_TF32_BIG_TILE_BLOCKS   // large tensor-core tiles once a launch has this many per SM
#define GEM_TF32_BIG_TILE_BLOCKS 1
#endif
#ifndef GEM_SIMT_BIG_TILE_BLOCKS   // the same for the CUDA-core tiles
#define GEM_SIMT_BIG_TILE_BLOCKS 2
#endif
#ifndef GEM_SIMT_MIN_CHUNK         // shortest split of K on the CUDA cores
#define GEM_SIMT_MIN_CHUNK 64
#endif
constexpr int kMaxSplit = GEM_MAX_SPLIT;   // split-K factor at most

enum Epilogue : int { kStore = 0, kBias = 1, kBiasRelu = 2, kMask = 3 };

struct Operand {
  const float* base;
  long long group_stride;  // elements between the operands of consecutive groups
  long long ld;            // leading dimension of its row-major storage
  int by_worker;           // group g uses index workers[g] (GEM state) instead of g (scratch)
};

struct GemmArgs {
  int M, N, K;
  Operand A;  // element (m, k)
  Operand B;  // element (k, n)
  float* C;
  long long c_group_stride, ldc;
  const float* bias;  // by worker, bias[n]
  long long bias_group_stride;
  const float* mask;  // by group, keep C(m, n) where mask(m, n) > 0
  long long mask_group_stride, ldmask;
  // split-K: blockIdx.z = group * ksplit + split; split s sums k in [s kchunk, (s+1) kchunk)
  // and writes its raw partial sums to ws + (group * ksplit + s) * M * N (row-major, ld N)
  int ksplit;
  int kchunk;
  float* ws;            // null: no split
  long long ws_floats;  // capacity of ws
  // tensor-core path: floats addressable from each operand's base (0: unknown, which keeps
  // the product off that path) and the error word its kernels report to
  long long a_extent, b_extent, c_extent, bias_extent, mask_extent;
  unsigned* status;
  // tensor-core path only: operands already TF32 (not rounded again), C stored rounded,
  // and an optional TF32-rounded transposed copy of C (ct: [N x M] per group, ld ldct)
  int a_rounded, b_rounded, round_c;
  float* ct;
  long long ct_group_stride, ldct, ct_extent;
  int workers[kMaxGroups];
};

// TF32 operand: keep 10 explicit mantissa bits, round to nearest with ties away from zero
// (add half of the dropped range to the magnitude bits, then clear them); inf and NaN
// pass through.
__device__ __forceinline__ float to_tf32(float x) {
  uint32_t u = __float_as_uint(x);
  if ((u & 0x7F800000u) != 0x7F800000u) u = (u + 0x1000u) & 0xFFFFE000u;
  return __uint_as_float(u);
}

// Four consecutive elements (outer, inner .. inner + 3) of a row-major view with leading
// dimension ld: one 16-byte load when the rows are 16-byte aligned (vec) and the quad lies
// inside the operand, else element by element; zeros outside.  TF32: each value rounded.
template <bool TF32>
__device__ __forceinline__ float4 stage_quad(const float* base, long long ld, bool vec, int outer,
                                             int inner, int outer_end, int inner_end) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  if (outer < outer_end) {
    const float* q = base + (long long)outer * ld + inner;
    if (vec && inner + 3 < inner_end) {
      v = *reinterpret_cast<const float4*>(q);
    } else {
      if (inner < inner_end) v.x = q[0];
      if (inner + 1 < inner_end) v.y = q[1];
      if (inner + 2 < inner_end) v.z = q[2];
      if (inner + 3 < inner_end) v.w = q[3];
    }
  }
  if (TF32) {
    v.x = to_tf32(v.x);
    v.y = to_tf32(v.y);
    v.z = to_tf32(v.z);
    v.w = to_tf32(v.w);
  }
  return v;
}

// C[g] (M x N) = epilogue( op(A[g]) op(B[g]) ).  A_KMAJOR: A(m, k) at A[m*lda + k], else at
// A[k*lda + m].  B_KMAJOR: B(k, n) at B[n*ldb + k], else at B[k*ldb + n].
//
// TBM x 64 tile per block of 2 TBM threads; thread (tx, ty) = (tid % 16, tid / 16) owns
// rows 8 ty .. 8 ty + 7 and columns 4 tx .. 4 tx + 3.  Both tiles are kept m- (or n-) contiguous
// in shared memory, double-buffered, so one k-step is three 128-bit shared loads and 32
// FMAs.  The next k-tile is read from global memory into registers while the current one
// is multiplied; global reads are coalesced along whichever index is contiguous.
template <int TBM, bool A_KMAJOR, bool B_KMAJOR, int EPI, bool TF32>
__global__ void __launch_bounds__(2 * TBM)
gemm_grouped_kernel(const __grid_constant__ GemmArgs p) {
  gem::pdl_entry();
  constexpr int T = 2 * TBM;                 // threads: 16 columns x TBM / 8 rows of them
  constexpr int kPadA = TBM + 4, kPadB = BN + 4;  // row pitches (floats), 16-byte aligned
  __shared__ __align__(16) float As[2][BK][kPadA];
  __shared__ __align__(16) float Bs[2][BK][kPadB];
  const int split = p.ksplit > 1 ? p.ksplit : 1;
  const int g = blockIdx.z / split, sk = blockIdx.z - g * split;
  const int kbeg = sk * p.kchunk;
  const int kend = split > 1 ? min(p.K, kbeg + p.kchunk) : p.K;
  const int m0 = blockIdx.y * TBM, n0 = blockIdx.x * BN;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const float* A = p.A.base + (p.A.by_worker ? (long long)p.workers[g] : (long long)g) * p.A.group_stride;
  const float* B = p.B.base + (p.B.by_worker ? (long long)p.workers[g] : (long long)g) * p.B.group_stride;
  const long long lda = p.A.ld, ldb = p.B.ld;
  const int M = p.M, N = p.N;

  // staging: the k-tile's A (TBM x 16) and B (64 x 16) elements as quads along each
  // operand's contiguous index (k for a K-major operand, m or n otherwise), two quads of A
  // and one or two of B per thread; quads are read with 16-byte loads where the operand's
  // rows are 16-byte aligned (k0 and the tile origins are multiples of 4).
  constexpr int kAQ = TBM * BK / 4 / T, kBQ = BN * BK / 4 / T;
  const bool a_vec = (reinterpret_cast<uintptr_t>(A) & 15u) == 0 && (lda & 3) == 0;
  const bool b_vec = (reinterpret_cast<uintptr_t>(B) & 15u) == 0 && (ldb & 3) == 0;
  float4 ra[kAQ], rb[kBQ];
  auto load = [&](int k0) {
#pragma unroll
    for (int it = 0; it < kAQ; ++it) {
      const int q = tid + T * it;
      if (A_KMAJOR) ra[it] = stage_quad<TF32>(A, lda, a_vec, m0 + (q >> 2), k0 + 4 * (q & 3), M, kend);
      else ra[it] = stage_quad<TF32>(A, lda, a_vec, k0 + q / (TBM / 4), m0 + 4 * (q % (TBM / 4)), kend, M);
    }
#pragma unroll
    for (int it = 0; it < kBQ; ++it) {
      const int q = tid + T * it;
      if (B_KMAJOR) rb[it] = stage_quad<TF32>(B, ldb, b_vec, n0 + (q >> 2), k0 + 4 * (q & 3), N, kend);
      else rb[it] = stage_quad<TF32>(B, ldb, b_vec, k0 + q / (BN / 4), n0 + 4 * (q % (BN / 4)), kend, N);
    }
  };
  auto store = [&](int buf) {
#pragma unroll
    for (int it = 0; it < kAQ; ++it) {
      const int q = tid + T * it;
      if (A_KMAJOR) {
        const int m = q >> 2, k = 4 * (q & 3);
        As[buf][k][m] = ra[it].x;
        As[buf][k + 1][m] = ra[it].y;
        As[buf][k + 2][m] = ra[it].z;
        As[buf][k + 3][m] = ra[it].w;
      } else {
        *reinterpret_cast<float4*>(&As[buf][q / (TBM / 4)][4 * (q % (TBM / 4))]) = ra[it];
      }
    }
#pragma unroll
    for (int it = 0; it < kBQ; ++it) {
      const int q = tid + T * it;
      if (B_KMAJOR) {
        const int n = q >> 2, k = 4 * (q & 3);
        Bs[buf][k][n] = rb[it].x;
        Bs[buf][k + 1][n] = rb[it].y;
        Bs[buf][k + 2][n] = rb[it].z;
        Bs[buf][k + 3][n] = rb[it].w;
      } else {
        *reinterpret_cast<float4*>(&Bs[buf][q / (BN / 4)][4 * (q % (BN / 4))]) = rb[it];
      }
    }
  };

  float acc[8][4];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  load(kbeg);
  store(0);
  __syncthreads();
  int buf = 0;
  for (int k0 = kbeg; k0 < kend; k0 += BK) {
    const bool more = k0 + BK < kend;
    if (more) load(k0 + BK);
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      const float4 a0 = *reinterpret_cast<const float4*>(&As[buf][k][ty * 8]);
      const float4 a1 = *reinterpret_cast<const float4*>(&As[buf][k][ty * 8 + 4]);
      const float4 b4 = *reinterpret_cast<const float4*>(&Bs[buf][k][tx * 4]);
      const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float b[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) {
      store(buf ^ 1);   // the other buffer was last read before the previous barrier
      __syncthreads();
      buf ^= 1;
    }
  }

  if (split > 1) {  // raw partial sums; splitk_reduce_kernel applies the epilogue
    float* W = p.ws + (long long)blockIdx.z * M * N;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int m = m0 + ty * 8 + i;
      if (m >= M) continue;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int n = n0 + tx * 4 + j;
        if (n < N) W[(long long)m * N + n] = acc[i][j];
      }
    }
    return;
  }
  float* C = p.C + (long long)g * p.c_group_stride;
  const float* bias = (EPI == kBias || EPI == kBiasRelu)
                          ? p.bias + (long long)p.workers[g] * p.bias_group_stride : nullptr;
  const float* mask = EPI == kMask ? p.mask + (long long)g * p.mask_group_stride : nullptr;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = m0 + ty * 8 + i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= N) continue;
      float v = acc[i][j];
      if (EPI == kBias) v = v + bias[n];
      if (EPI == kBiasRelu) v = fmaxf(v + bias[n], 0.f);
      if (EPI == kMask) v = mask[m * p.ldmask + n] > 0.f ? v : 0.f;
      C[m * p.ldc + n] = v;
    }
  }
}

// The same products with TF32 operands on the tensor cores (warp-level mma.sync, m16n8k8,
// fp32 accumulation), used for GEM_MLP_TF32.  Operands are rounded to TF32 exactly as the
// CUDA-core path rounds them (to_tf32) while they are staged, so the tensor cores see the
// same operand values; products of TF32 values are exact, and the sums are fp32 in the
// tensor cores' order.
//
// 128 x TBN tile per block of 256 threads: 8 warps as 2 (m) x 4 (n), each owning a 64 x TBN/4
// sub-tile of m16n8 accumulators.  k-tiles of 16 are staged m- (n-) major in shared memory
// with a row pitch of 20 floats, so the fragment reads (rows gid, columns tig) of a warp hit
// 32 different banks; double-buffered, with the next k-tile read into registers while the
// current one is multiplied.
constexpr int kMmaBM = 128, kMmaBK = 16, kMmaPitch = kMmaBK + 4;

__device__ __forceinline__ void mma_tf32(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <int TBN, bool A_KMAJOR, bool B_KMAJOR, int EPI>
__global__ void __launch_bounds__(256)
gemm_mma_tf32_kernel(const __grid_constant__ GemmArgs p) {
  gem::pdl_entry();
  constexpr int kT = 256;
  constexpr int kWN = TBN / 4;            // columns per warp
  constexpr int kNT = kWN / 8;            // n8 tiles per warp
  constexpr int kAPer = kMmaBM * kMmaBK / kT;   // 8
  constexpr int kBPer = TBN * kMmaBK / kT;      // 4 or 8
  __shared__ __align__(16) float As[2][kMmaBM][kMmaPitch];
  __shared__ __align__(16) float Bs[2][TBN][kMmaPitch];
  const int split = p.ksplit > 1 ? p.ksplit : 1;
  const int g = blockIdx.z / split, sk = blockIdx.z - g * split;
  const int kbeg = sk * p.kchunk;
  const int kend = split > 1 ? min(p.K, kbeg + p.kchunk) : p.K;
  const int m0 = blockIdx.y * kMmaBM, n0 = blockIdx.x * TBN;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int wm = warp >> 2, wn = warp & 3;          // warp position: 2 x 4
  const int gid = lane >> 2, tig = lane & 3;        // mma fragment coordinates
  const float* A = p.A.base + (p.A.by_worker ? (long long)p.workers[g] : (long long)g) * p.A.group_stride;
  const float* B = p.B.base + (p.B.by_worker ? (long long)p.workers[g] : (long long)g) * p.B.group_stride;
  const long long lda = p.A.ld, ldb = p.B.ld;
  const int M = p.M, N = p.N;

  // staging coordinates: coalesced along k for K-major operands, along m (n) otherwise
  float ra[kAPer], rb[kBPer];
  auto a_coord = [&](int it, int& m, int& k) {
    const int idx = tid + kT * it;
    if (A_KMAJOR) { m = idx >> 4; k = idx & 15; }
    else          { m = idx & (kMmaBM - 1); k = idx / kMmaBM; }
  };
  auto b_coord = [&](int it, int& n, int& k) {
    const int idx = tid + kT * it;
    if (B_KMAJOR) { n = idx >> 4; k = idx & 15; }
    else          { n = idx % TBN; k = idx / TBN; }
  };
  auto load = [&](int k0) {
#pragma unroll
    for (int it = 0; it < kAPer; ++it) {
      int m, k;
      a_coord(it, m, k);
      const int gm = m0 + m, gk = k0 + k;
      float v = 0.f;
      if (gm < M && gk < kend) v = A_KMAJOR ? A[gm * lda + gk] : A[gk * lda + gm];
      ra[it] = to_tf32(v);
    }
#pragma unroll
    for (int it = 0; it < kBPer; ++it) {
      int n, k;
      b_coord(it, n, k);
      const int gn = n0 + n, gk = k0 + k;
      float v = 0.f;
      if (gn < N && gk < kend) v = B_KMAJOR ? B[gn * ldb + gk] : B[gk * ldb + gn];
      rb[it] = to_tf32(v);
    }
  };
  auto store = [&](int buf) {
#pragma unroll
    for (int it = 0; it < kAPer; ++it) {
      int m, k;
      a_coord(it, m, k);
      As[buf][m][k] = ra[it];
    }
#pragma unroll
    for (int it = 0; it < kBPer; ++it) {
      int n, k;
      b_coord(it, n, k);
      Bs[buf][n][k] = rb[it];
    }
  };

  float acc[4][kNT][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < kNT; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[i][j][e] = 0.f;

  load(kbeg);
  store(0);
  __syncthreads();
  int buf = 0;
  for (int k0 = kbeg; k0 < kend; k0 += kMmaBK) {
    const bool more = k0 + kMmaBK < kend;
    if (more) load(k0 + kMmaBK);
#pragma unroll
    for (int ks = 0; ks < kMmaBK; ks += 8) {
      uint32_t af[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int r = wm * 64 + i * 16 + gid;
        af[i][0] = __float_as_uint(As[buf][r][ks + tig]);
        af[i][1] = __float_as_uint(As[buf][r + 8][ks + tig]);
        af[i][2] = __float_as_uint(As[buf][r][ks + tig + 4]);
        af[i][3] = __float_as_uint(As[buf][r + 8][ks + tig + 4]);
      }
#pragma unroll
      for (int j = 0; j < kNT; ++j) {
        const int c = wn * kWN + j * 8 + gid;
        const uint32_t b0 = __float_as_uint(Bs[buf][c][ks + tig]);
        const uint32_t b1 = __float_as_uint(Bs[buf][c][ks + tig + 4]);
#pragma unroll
        for (int i = 0; i < 4; ++i) mma_tf32(acc[i][j], af[i], b0, b1);
      }
    }
    if (more) {
      store(buf ^ 1);   // the other buffer was last read before the previous barrier
      __syncthreads();
      buf ^= 1;
    }
  }

  // accumulator (i, j, e) holds C(row, col) with row = base + i*16 + gid + 8 (e >= 2),
  // col = base + j*8 + 2 tig + (e & 1)
  float* C = p.C + (long long)g * p.c_group_stride;
  float* W = split > 1 ? p.ws + (long long)blockIdx.z * M * N : nullptr;
  const float* bias = (EPI == kBias || EPI == kBiasRelu)
                          ? p.bias + (long long)p.workers[g] * p.bias_group_stride : nullptr;
  const float* mask = EPI == kMask ? p.mask + (long long)g * p.mask_group_stride : nullptr;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int m = m0 + wm * 64 + i * 16 + gid + (e >= 2 ? 8 : 0);
      if (m >= M) continue;
#pragma unroll
      for (int j = 0; j < kNT; ++j) {
        const int n = n0 + wn * kWN + j * 8 + 2 * tig + (e & 1);
        if (n >= N) continue;
        float v = acc[i][j][e];
        if (W) {  // raw partial sums; splitk_reduce_kernel applies the epilogue
          W[(long long)m * N + n] = v;
          continue;
        }
        if (EPI == kBias) v = v + bias[n];
        if (EPI == kBiasRelu) v = fmaxf(v + bias[n], 0.f);
        if (EPI == kMask) v = mask[m * p.ldmask + n] > 0.f ? v : 0.f;
        C[m * p.ldc + n] = v;
      }
    }
  }
}

// Pipelined variant for operands whose rows start on 16-byte boundaries (leading
// dimensions, group strides and bases multiples of 4 floats): k-tiles of 32 are copied
// global -> shared with cp.async (16-byte chunks, zero-filled past the operand's edge) into a
// 3-stage ring, so the copies of the next two k-tiles are in flight while the tensor cores
// work on the current one.  A K-major operand is staged [row][k] (pitch 36 floats), an
// m- (n-) contiguous one [k][row] (pitch rows + 8); both give conflict-free fragment reads.
// Each thread rounds the chunks it copied to TF32 (cvt.rna: nearest, ties away from zero, as
// to_tf32) once they have landed; K-major fragments are then read with ldmatrix.
#ifndef GEM_PIPE_BK
#define GEM_PIPE_BK 32
#endif
#ifndef GEM_PIPE_STAGES
#define GEM_PIPE_STAGES 3
#endif
constexpr int kPipeBK = GEM_PIPE_BK, kPipeStages = GEM_PIPE_STAGES;
static_assert(kPipeBK % 8 == 0 && (64 * kPipeBK / 4) % 256 == 0, "k-tile must split into 16-byte chunks");

__host__ __device__ constexpr int pipe_tile_floats(int rows, bool kmajor) {
  return kmajor ? rows * (kPipeBK + 4) : kPipeBK * (rows + 8);
}

__device__ __forceinline__ uint32_t tf32_bits(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src, int src_bytes) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem_dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(gmem_src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Stage the k-tile [k0, k0 + 32) of an operand tile of R rows (m or n) starting at row0:
// element (row, k) is at src[row * ld + k] (K-major) or src[k * ld + row].  Rows >= rows_end
// and k >= k_end are zero-filled (a chunk that straddles an edge copies its valid part).
template <int R, bool KMAJOR>
__device__ __forceinline__ void stage_tile(float* dst, const float* src, long long ld, int row0,
                                           int rows_end, int k0, int k_end, int tid) {
  constexpr int kChunks = R * kPipeBK / 4;
#pragma unroll
  for (int i = 0; i < kChunks / 256; ++i) {
    const int q = tid + 256 * i;
    int row, k, valid;
    float* d;
    if (KMAJOR) {
      row = q / (kPipeBK / 4);
      k = (q % (kPipeBK / 4)) * 4;
      d = dst + row * (kPipeBK + 4) + k;
      valid = (row0 + row < rows_end) ? min(4, max(0, k_end - (k0 + k))) : 0;
    } else {
      k = q / (R / 4);
      row = (q % (R / 4)) * 4;
      d = dst + k * (R + 8) + row;
      valid = (k0 + k < k_end) ? min(4, max(0, rows_end - (row0 + row))) : 0;
    }
    const float* g = valid ? (KMAJOR ? src + (long long)(row0 + row) * ld + (k0 + k)
                                     : src + (long long)(k0 + k) * ld + (row0 + row))
                           : src;
    cp_async16(d, g, valid * 4);
  }
}

// Round, in place, the chunks this thread copied with stage_tile (after they have landed):
// every staged element is rounded to TF32 once, by the thread that fetched it.
template <int R, bool KMAJOR>
__device__ __forceinline__ void round_tile(float* dst, int tid) {
  constexpr int kChunks = R * kPipeBK / 4;
#pragma unroll
  for (int i = 0; i < kChunks / 256; ++i) {
    const int q = tid + 256 * i;
    float* d = KMAJOR ? dst + (q / (kPipeBK / 4)) * (kPipeBK + 4) + (q % (kPipeBK / 4)) * 4
                      : dst + (q / (R / 4)) * (R + 8) + (q % (R / 4)) * 4;
    float4 v = *reinterpret_cast<float4*>(d);
    v.x = __uint_as_float(tf32_bits(v.x));
    v.y = __uint_as_float(tf32_bits(v.y));
    v.z = __uint_as_float(tf32_bits(v.z));
    v.w = __uint_as_float(tf32_bits(v.w));
    *reinterpret_cast<float4*>(d) = v;
  }
}

// Four 8 x 4 blocks of 32-bit words from shared memory in the register layout of an m16n8k8
// TF32 fragment: lane l supplies the address of row l % 8 of block l / 8; register i of
// lane t receives word (t / 4, t % 4) of block i.
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const float* row_addr) {
  const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(row_addr));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a));
}

template <int TBN, bool A_KMAJOR, bool B_KMAJOR, int EPI>
__global__ void __launch_bounds__(256)
gemm_mma_pipe_kernel(const __grid_constant__ GemmArgs p) {
  gem::pdl_entry();
  constexpr int kWN = TBN / 4, kNT = kWN / 8;
  constexpr int kAF = pipe_tile_floats(kMmaBM, A_KMAJOR), kBF = pipe_tile_floats(TBN, B_KMAJOR);
  constexpr int kStageF = kAF + kBF;
  extern __shared__ __align__(16) float pipe_smem[];
  const int split = p.ksplit > 1 ? p.ksplit : 1;
  const int g = blockIdx.z / split, sk = blockIdx.z - g * split;
  const int kbeg = sk * p.kchunk;
  const int kend = split > 1 ? min(p.K, kbeg + p.kchunk) : p.K;
  const int m0 = blockIdx.y * kMmaBM, n0 = blockIdx.x * TBN;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int wm = warp >> 2, wn = warp & 3;
  const int gid = lane >> 2, tig = lane & 3;
  const float* A = p.A.base + (p.A.by_worker ? (long long)p.workers[g] : (long long)g) * p.A.group_stride;
  const float* B = p.B.base + (p.B.by_worker ? (long long)p.workers[g] : (long long)g) * p.B.group_stride;
  const int M = p.M, N = p.N;
  const int nkt = kend > kbeg ? (kend - kbeg + kPipeBK - 1) / kPipeBK : 0;

  auto issue = [&](int kt) {
    float* st = pipe_smem + (kt % kPipeStages) * kStageF;
    const int k0 = kbeg + kt * kPipeBK;
    stage_tile<kMmaBM, A_KMAJOR>(st, A, p.A.ld, m0, M, k0, kend, tid);
    stage_tile<TBN, B_KMAJOR>(st + kAF, B, p.B.ld, n0, N, k0, kend, tid);
  };
  auto a_at = [&](const float* t, int row, int k) -> float {
    return A_KMAJOR ? t[row * (kPipeBK + 4) + k] : t[k * (kMmaBM + 8) + row];
  };
  auto b_at = [&](const float* t, int row, int k) -> float {
    return B_KMAJOR ? t[row * (kPipeBK + 4) + k] : t[k * (TBN + 8) + row];
  };

  float acc[4][kNT][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < kNT; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[i][j][e] = 0.f;

#pragma unroll
  for (int s = 0; s < kPipeStages - 1; ++s) {
    if (s < nkt) issue(s);
    cp_async_commit();
  }
  // ldmatrix row of this lane within a 16 x 8 (A) or 16 x 8 pair-of-n-tiles (B) block
  const int lrow = (lane & 7) + ((lane >> 3) & 1) * 8, lcol = (lane >> 4) * 4;
  const int brow = (lane & 7) + (lane >> 4) * 8, bcol = ((lane >> 3) & 1) * 4;
  for (int kt = 0; kt < nkt; ++kt) {
    cp_async_wait<kPipeStages - 2>();   // this thread's copies of k-tile kt have landed
    float* ta = pipe_smem + (kt % kPipeStages) * kStageF;
    float* tb = ta + kAF;
    round_tile<kMmaBM, A_KMAJOR>(ta, tid);
    round_tile<TBN, B_KMAJOR>(tb, tid);
    __syncthreads();                    // everyone's k-tile kt is rounded; stage kt - 1 is free
    if (kt + kPipeStages - 1 < nkt) issue(kt + kPipeStages - 1);
    cp_async_commit();
#pragma unroll
    for (int ks = 0; ks < kPipeBK; ks += 8) {
      uint32_t af[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int r = wm * 64 + i * 16;
        if (A_KMAJOR) {
          ldsm_x4(af[i], ta + (r + lrow) * (kPipeBK + 4) + ks + lcol);
        } else {
          af[i][0] = __float_as_uint(a_at(ta, r + gid, ks + tig));
          af[i][1] = __float_as_uint(a_at(ta, r + gid + 8, ks + tig));
          af[i][2] = __float_as_uint(a_at(ta, r + gid, ks + tig + 4));
          af[i][3] = __float_as_uint(a_at(ta, r + gid + 8, ks + tig + 4));
        }
      }
#pragma unroll
      for (int j = 0; j < kNT; j += 2) {
        uint32_t bf[4];   // b0, b1 of n-tile j, then of n-tile j + 1
        const int c = wn * kWN + j * 8;
        if (B_KMAJOR) {
          ldsm_x4(bf, tb + (c + brow) * (kPipeBK + 4) + ks + bcol);
        } else {
          bf[0] = __float_as_uint(b_at(tb, c + gid, ks + tig));
          bf[1] = __float_as_uint(b_at(tb, c + gid, ks + tig + 4));
          bf[2] = __float_as_uint(b_at(tb, c + 8 + gid, ks + tig));
          bf[3] = __float_as_uint(b_at(tb, c + 8 + gid, ks + tig + 4));
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          mma_tf32(acc[i][j], af[i], bf[0], bf[1]);
          mma_tf32(acc[i][j + 1], af[i], bf[2], bf[3]);
        }
      }
    }
  }
  cp_async_wait<0>();

  float* C = p.C + (long long)g * p.c_group_stride;
  float* W = split > 1 ? p.ws + (long long)blockIdx.z * M * N : nullptr;
  const float* bias = (EPI == kBias || EPI == kBiasRelu)
                          ? p.bias + (long long)p.workers[g] * p.bias_group_stride : nullptr;
  const float* mask = EPI == kMask ? p.mask + (long long)g * p.mask_group_stride : nullptr;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int m = m0 + wm * 64 + i * 16 + gid + (e >= 2 ? 8 : 0);
      if (m >= M) continue;
#pragma unroll
      for (int j = 0; j < kNT; ++j) {
        const int n = n0 + wn * kWN + j * 8 + 2 * tig + (e & 1);
        if (n >= N) continue;
        float v = acc[i][j][e];
        if (W) {
          W[(long long)m * N + n] = v;
          continue;
        }
        if (EPI == kBias) v = v + bias[n];
        if (EPI == kBiasRelu) v = fmaxf(v + bias[n], 0.f);
        if (EPI == kMask) v = mask[m * p.ldmask + n] > 0.f ? v : 0.f;
        C[m * p.ldc + n] = v;
      }
    }
  }
}

// Sum of the split-K partials of every output in split order (deterministic), then the
// epilogue of the product.
template <int EPI, int V>
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const __grid_constant__ GemmArgs p) {
  gem::pdl_entry();
  // one output row (g, m) per blockIdx.y; thread t of blockIdx.x covers V consecutive columns
  const int M = p.M, N = p.N;
  const int g = blockIdx.y / M, m = blockIdx.y - g * M;
  const int n0 = (blockIdx.x * blockDim.x + threadIdx.x) * V;
  if (n0 >= N) return;
  const long long MN = (long long)M * N;
  const float* W = p.ws + (long long)g * p.ksplit * MN + (long long)m * N + n0;
  const float* bias = (EPI == kBias || EPI == kBiasRelu)
                          ? p.bias + (long long)p.workers[g] * p.bias_group_stride + n0 : nullptr;
  const float* mask = EPI == kMask ? p.mask + (long long)g * p.mask_group_stride + (long long)m * p.ldmask + n0
                                   : nullptr;
  float* C = p.C + (long long)g * p.c_group_stride + (long long)m * p.ldc + n0;
  if (V == 4) {
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s = 0; s < p.ksplit; ++s) {
      const float4 w = *reinterpret_cast<const float4*>(W + s * MN);
      v.x += w.x;
      v.y += w.y;
      v.z += w.z;
      v.w += w.w;
    }
    float o[4] = {v.x, v.y, v.z, v.w};
    if (EPI == kBias || EPI == kBiasRelu) {
      const float4 b = *reinterpret_cast<const float4*>(bias);
      const float bb[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) o[j] = EPI == kBiasRelu ? fmaxf(o[j] + bb[j], 0.f) : o[j] + bb[j];
    }
    if (EPI == kMask) {
      const float4 k = *reinterpret_cast<const float4*>(mask);
      const float kk[4] = {k.x, k.y, k.z, k.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) o[j] = kk[j] > 0.f ? o[j] : 0.f;
    }
    *reinterpret_cast<float4*>(C) = make_float4(o[0], o[1], o[2], o[3]);
  } else {
    float v = 0.f;
    for (int s = 0; s < p.ksplit; ++s) v += W[s * MN];
    if (EPI == kBias) v = v + bias[0];
    if (EPI == kBiasRelu) v = fmaxf(v + bias[0], 0.f);
    if (EPI == kMask) v = mask[0] > 0.f ? v : 0.f;
    C[0] = v;
  }
}

// Products with few outputs per row (N <= kMaxClasses), used for the logits:
// C[g][m][n] = sum_k A[g][m][k] B[g][n][k] + bias[n], A and B K-major.  The block first
// copies the worker's B (N x K, TF32-rounded when asked) into shared memory; then each warp
// takes whole rows m: lane l accumulates k = l, l + 32, ... (coalesced A reads, conflict-free
// shared reads), a fixed butterfly adds the 32 lane sums, and lane 0 writes the N outputs
// of the row.  Deterministic.  rows_per_block rows per block; NC >= N classes compiled in
// (16 or 32), so that a network with few classes carries no idle class slots.
// The last layer's softmax cross-entropy, fused into the logits kernel (XENT): the lane
// that finishes a row's logits z goes on, with the operations and order of
// softmax_xent_kernel, to the row's loss gradient (softmax(z) - onehot(y)) / b and its
// loss; the row losses are summed in row order by bias_grad_kernel.
struct XentArgs {
  const int32_t* labels;        // [rows of the data set]
  const int32_t* batch_rows;    // [groups][b]
  float* delta;                 // D_L [b][C] of group g at delta + g * group_stride
  float* row_loss;              // [b] of group g at row_loss + g * group_stride
  long long group_stride;
  int b;
};

template <bool TF32, bool XENT, int NC>
__global__ void __launch_bounds__(256)
gemm_small_n_kernel(const __grid_constant__ GemmArgs p, int rows_per_block,
                    const __grid_constant__ XentArgs x) {
  gem::pdl_entry();
  extern __shared__ __align__(16) float Bsm[];
  const int g = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* A = p.A.base + (p.A.by_worker ? (long long)p.workers[g] : (long long)g) * p.A.group_stride;
  const float* B = p.B.base + (p.B.by_worker ? (long long)p.workers[g] : (long long)g) * p.B.group_stride;
  const int N = p.N, K = p.K;
  const bool vec = K % 4 == 0 && p.B.ld % 4 == 0 && (reinterpret_cast<uintptr_t>(B) & 15u) == 0;
  if (vec) {   // 16-byte asynchronous copies, all in flight at once, then rounded in place
    const int chunks = N * K / 4;
    for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
      const int n = (4 * c) / K, k = 4 * c - n * K;
      cp_async16(Bsm + 4 * c, B + (long long)n * p.B.ld + k, 16);
    }
    cp_async_commit();
    cp_async_wait<0>();
    if (TF32)
      for (int c = threadIdx.x; c < chunks; c += blockDim.x) {
        float4 v = *reinterpret_cast<float4*>(Bsm + 4 * c);
        v.x = to_tf32(v.x);
        v.y = to_tf32(v.y);
        v.z = to_tf32(v.z);
        v.w = to_tf32(v.w);
        *reinterpret_cast<float4*>(Bsm + 4 * c) = v;
      }
  } else {
#pragma unroll 8
    for (int i = threadIdx.x; i < N * K; i += blockDim.x) {
      const int n = i / K, k = i - n * K;
      const float v = B[(long long)n * p.B.ld + k];
      Bsm[i] = TF32 ? to_tf32(v) : v;
    }
  }
  __syncthreads();
  const float* bias = p.bias + (long long)p.workers[g] * p.bias_group_stride;
  const int r0 = blockIdx.x * rows_per_block;
  const int r1 = min(p.M, r0 + rows_per_block);
  for (int m = r0 + warp; m < r1; m += 8) {
    const float* a = A + (long long)m * p.A.ld;
    float acc[NC];
#pragma unroll
    for (int n = 0; n < NC; ++n) acc[n] = 0.f;
    constexpr int kUnroll = NC <= 16 ? 8 : 4;   // A loads in flight within the register budget
#pragma unroll kUnroll
    for (int k = lane; k < K; k += 32) {
      const float av = TF32 ? to_tf32(a[k]) : a[k];
#pragma unroll
      for (int n = 0; n < NC; ++n)
        if (n < N) acc[n] = fmaf(av, Bsm[n * K + k], acc[n]);
    }
#pragma unroll
    for (int n = 0; n < NC; ++n) {
      if (n < N) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc[n] += __shfl_xor_sync(0xffffffffu, acc[n], off);
      }
    }
    if (lane == 0) {
      float* c = p.C + (long long)g * p.c_group_stride + (long long)m * p.ldc;
#pragma unroll
      for (int n = 0; n < NC; ++n)
        if (n < N) {
          acc[n] = acc[n] + bias[n];   // the logit z_n
          c[n] = acc[n];
        }
      if (XENT) {
        int y = x.labels[x.batch_rows[(long long)g * x.b + m]];
        const bool bad_label = y < 0 || y >= N;   // reported as a NaN loss and gradient
        if (bad_label) y = 0;
        float zmax = acc[0];
#pragma unroll
        for (int n = 1; n < NC; ++n)
          if (n < N) zmax = fmaxf(zmax, acc[n]);
        float e[NC];
        float sum = 0.f;
#pragma unroll
        for (int n = 0; n < NC; ++n)
          if (n < N) {
            e[n] = expf(acc[n] - zmax);
            sum += e[n];
          }
        const float inv_b = 1.0f / float(x.b);
        const float poison = bad_label ? __int_as_float(0x7fc00000) : 0.f;
        float* d = x.delta + (long long)g * x.group_stride + (long long)m * N;
        float zy = acc[0];
#pragma unroll
        for (int n = 0; n < NC; ++n)
          if (n < N) {
            d[n] = (e[n] / sum - (n == y ? 1.f : 0.f)) * inv_b + poison;
            if (n == y) zy = acc[n];
          }
        x.row_loss[(long long)g * x.group_stride + m] = (logf(sum) + zmax) - zy + poison;
      }
    }
  }
}

// Launch the logits product when B fits in shared memory; false otherwise.
// xent: the fused loss (null for plain logits).
template <bool TF32>
bool launch_small_n(const GemmArgs& a, int groups, cudaStream_t st, cudaError_t* err,
                    const XentArgs* xent) {
  const size_t bytes = sizeof(float) * size_t(a.N) * size_t(a.K);
  constexpr size_t kMaxBytes = 200 * 1024;
  if (bytes > kMaxBytes) return false;
  static bool configured[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (bytes > 48 * 1024 && (dev < 0 || dev >= 64 || !configured[dev])) {
    *err = cudaFuncSetAttribute(gemm_small_n_kernel<TF32, false, 16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, int(kMaxBytes));
    if (*err == cudaSuccess)
      *err = cudaFuncSetAttribute(gemm_small_n_kernel<TF32, true, 16>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, int(kMaxBytes));
    if (*err == cudaSuccess)
      *err = cudaFuncSetAttribute(gemm_small_n_kernel<TF32, false, kMaxClasses>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, int(kMaxBytes));
    if (*err == cudaSuccess)
      *err = cudaFuncSetAttribute(gemm_small_n_kernel<TF32, true, kMaxClasses>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, int(kMaxBytes));
    if (*err != cudaSuccess) return true;
    if (dev >= 0 && dev < 64) configured[dev] = true;
  }
  // enough blocks to cover the SMs about twice, at least 8 rows (one per warp) each
  long long rows_per_block = (long long)a.M * groups / (2 * kSmCountHint);
  rows_per_block = rows_per_block < 8 ? 8 : (rows_per_block + 7) / 8 * 8;
  const int rpb = int(rows_per_block);
  dim3 grid(unsigned((a.M + rpb - 1) / rpb), unsigned(groups));
  const XentArgs xa = xent ? *xent : XentArgs{};
  if (a.N <= 16) {
    if (xent) gem::launch_pdl(gemm_small_n_kernel<TF32, true, 16>, grid, 256, bytes, st, a, rpb, xa);
    else gem::launch_pdl(gemm_small_n_kernel<TF32, false, 16>, grid, 256, bytes, st, a, rpb, xa);
  } else {
    if (xent) gem::launch_pdl(gemm_small_n_kernel<TF32, true, kMaxClasses>, grid, 256, bytes, st, a, rpb, xa);
    else gem::launch_pdl(gemm_small_n_kernel<TF32, false, kMaxClasses>, grid, 256, bytes, st, a, rpb, xa);
  }
  *err = cudaGetLastError();
  return true;
}

// Minibatch gather: slot g's rows X[batch_rows[g][r]] -> Xs[g][r][:].
__global__ void gather_rows_kernel(const float* X, int d0, const int32_t* batch_rows, int b,
                                   float* Xs, long long slot_stride, int round) {
  gem::pdl_entry();
  const int g = blockIdx.y, r = blockIdx.x;
  const long long row = batch_rows[(long long)g * b + r];
  const float* src = X + row * d0;
  float* dst = Xs + g * slot_stride + (long long)r * d0;
  // with TF32 products the gathered rows are only ever operands: stored rounded once
  for (int k = threadIdx.x; k < d0; k += blockDim.x) dst[k] = round ? to_tf32(src[k]) : src[k];
}

// dst[g] = transpose(src[g]) rounded to TF32: src [rows][cols] row-major, dst [cols][rows];
// src[g] at src + (by_worker ? workers[g] : g) * src_stride, dst[g] at dst + g * dst_stride.
// 32 x 32 tiles through shared memory.  The tensor-core products read both operands
// K-major, so the weight gradients read the minibatch panels X and D transposed (the batch
// as K); the hidden activations' transposes come from the forward products' epilogue.
struct TransposeArgs {
  const float* src;
  long long src_stride;
  float* dst;
  long long dst_stride;
  int rows, cols;
  int by_worker;
  int workers[kMaxGroups];
};

__global__ void __launch_bounds__(256) transpose_round_kernel(const __grid_constant__ TransposeArgs t) {
  gem::pdl_entry();
  __shared__ float tile[32][33];
  const int g = blockIdx.z, c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int rows = t.rows, cols = t.cols;
  const float* s = t.src + (t.by_worker ? (long long)t.workers[g] : (long long)g) * t.src_stride;
  float* d = t.dst + g * t.dst_stride;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int i = ty; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + tx;
    tile[i][tx] = (r < rows && c < cols) ? to_tf32(s[(long long)r * cols + c]) : 0.f;
  }
  __syncthreads();
  for (int i = ty; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + tx;
    if (r < rows && c < cols) d[(long long)c * rows + r] = tile[tx][i];
  }
}

// Softmax cross-entropy over C classes for the b rows of each slot: the mean loss, and the
// gradient of the mean with respect to the logits, (softmax - onehot) / b.
__global__ void softmax_xent_kernel(const float* logits, float* delta, long long slot_stride,
                                   int b, int C, const int32_t* labels,
                                   const int32_t* batch_rows, float* losses) {
  gem::pdl_entry();
  __shared__ float row_loss[kMaxBatch];
  const int g = blockIdx.x;
  const float* z = logits + g * slot_stride;
  float* d = delta + g * slot_stride;
  for (int r = threadIdx.x; r < b; r += blockDim.x) {
    const float* zr = z + (long long)r * C;
    int y = labels[batch_rows[(long long)g * b + r]];
    const bool bad_label = y < 0 || y >= C;  // reported as a NaN loss and gradient
    if (bad_label) y = 0;
    float zmax = zr[0];
    for (int c = 1; c < C; ++c) zmax = fmaxf(zmax, zr[c]);
    float e[kMaxClasses];
    float sum = 0.f;
    for (int c = 0; c < C; ++c) {
      e[c] = expf(zr[c] - zmax);
      sum += e[c];
    }
    const float inv_b = 1.0f / float(b);
    const float poison = bad_label ? __int_as_float(0x7fc00000) : 0.f;
    for (int c = 0; c < C; ++c)
      d[(long long)r * C + c] = (e[c] / sum - (c == y ? 1.f : 0.f)) * inv_b + poison;
    row_loss[r] = (logf(sum) + zmax) - zr[y] + poison;
  }
  __syncthreads();
  if (losses && threadIdx.x == 0) {
    float s = 0.f;
    for (int r = 0; r < b; ++r) s += row_loss[r];
    losses[g] = s / float(b);
  }
}

struct BiasGradArgs {
  int n_layers, b;
  long long row_loss_off;           // with losses: the row losses of the fused loss kernel
  float* losses;                    // [groups] minibatch losses, or null
  long long grad_off[kMaxLayers];   // offset of db_l in the flat gradient
  long long delta_off[kMaxLayers];  // offset of D_{l+1} in the slot scratch
  int width[kMaxLayers];            // d_{l+1}
  int first[kMaxLayers + 1];        // prefix sums of width
};

// db_l[o] = sum over the batch of D_{l+1}[r][o], every layer in one launch.
// Block of 32 x 8 threads: lane x owns output q = 32 blockIdx.x + x; warp y sums rows
// r = y, y + 8, ... in order, and lane x of warp 0 adds the 8 warp sums in order.  When
// the logits kernel computed the loss (losses set), thread 0 of block (0, g) also adds
// group g's row losses in row order and divides by b.
__global__ void __launch_bounds__(256)
bias_grad_kernel(const __grid_constant__ BiasGradArgs a, const float* delta,
                 long long slot_stride, float* grad, long long grad_stride) {
  gem::pdl_entry();
  __shared__ float part[8][33];
  const int g = blockIdx.y;
  const int x = threadIdx.x & 31, y = threadIdx.x >> 5;
  const int q = blockIdx.x * 32 + x;
  float s = 0.f;
  int l = 0, o = 0;
  if (q < a.first[a.n_layers]) {
    while (q >= a.first[l + 1]) ++l;
    o = q - a.first[l];
    const float* D = delta + g * slot_stride + a.delta_off[l];
    for (int r = y; r < a.b; r += 8) s += D[(long long)r * a.width[l] + o];
  }
  part[y][x] = s;
  __syncthreads();
  if (y == 0 && q < a.first[a.n_layers]) {
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) t += part[w][x];
    grad[g * grad_stride + a.grad_off[l] + o] = t;
  }
  if (a.losses && blockIdx.x == 0 && threadIdx.x == 0) {   // the minibatch loss, rows in order
    const float* rl = delta + g * slot_stride + a.row_loss_off;
    float t = 0.f;
    for (int r = 0; r < a.b; ++r) t += rl[r];
    a.losses[g] = t / float(a.b);
  }
}

template <int TBM, bool AK, bool BK_, int EPI>
void launch_tile(const GemmArgs& a, int groups, bool tf32, cudaStream_t st) {
  dim3 grid((a.N + BN - 1) / BN, (a.M + TBM - 1) / TBM, groups);
  if (tf32)
    gem::launch_pdl(gemm_grouped_kernel<TBM, AK, BK_, EPI, true>, grid, 2 * TBM, 0, st, a);
  else
    gem::launch_pdl(gemm_grouped_kernel<TBM, AK, BK_, EPI, false>, grid, 2 * TBM, 0, st, a);
}

bool operand_16b(const Operand& o) {
  return (reinterpret_cast<uintptr_t>(o.base) & 15u) == 0 && o.ld % 4 == 0 && o.group_stride % 4 == 0;
}

template <int TBN, bool AK, bool BK_, int EPI>
void launch_mma(const GemmArgs& a, int groups, cudaStream_t st) {
  dim3 grid((a.N + TBN - 1) / TBN, (a.M + kMmaBM - 1) / kMmaBM, groups);
  if (operand_16b(a.A) && operand_16b(a.B)) {
    constexpr int bytes = kPipeStages * 4 *
                          (pipe_tile_floats(kMmaBM, AK) + pipe_tile_floats(TBN, BK_));
    static bool configured[64] = {};   // one attribute call per instantiation and device
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64 || !configured[dev]) {
      if (cudaFuncSetAttribute(gemm_mma_pipe_kernel<TBN, AK, BK_, EPI>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
        return;   // the error is reported by the caller's cudaGetLastError
      if (dev >= 0 && dev < 64) configured[dev] = true;
    }
    gem::launch_pdl(gemm_mma_pipe_kernel<TBN, AK, BK_, EPI>, grid, 256, bytes, st, a);
  } else {
    gem::launch_pdl(gemm_mma_tf32_kernel<TBN, AK, BK_, EPI>, grid, 256, 0, st, a);
  }
}

// TF32 products run on the tensor cores (mma.sync), fp32 products on the CUDA cores.  The
// large tile (128 x 128 on the tensor cores, 128 x 64 on the CUDA cores) when the launch
// fills the GPU with at least two blocks per SM; otherwise the half-size tile and, when a
// split-K workspace is given and K is long, up to kMaxSplit splits of K whose partial sums a
// second kernel adds in a fixed order.
template <bool AK, bool BK_, int EPI>
cudaError_t launch_gemm(const GemmArgs& a_in, int groups, bool tf32, cudaStream_t st,
                        bool* on_tc = nullptr) {
  GemmArgs a = a_in;
  if (on_tc) *on_tc = false;
  a.ksplit = 1;
  a.kchunk = a.K;
  // Products with fewer than 32 rows or a K below 32 (the last layer's weight and input
  // gradients) would leave a 128-row tensor-core tile mostly empty or its pipeline idle:
  // they run on the CUDA cores, with the same TF32 operand rounding.
  const bool tc = tf32 && a.M >= 32 && a.K >= 32;
  if (tc && a.a_extent > 0 && a.b_extent > 0 && a.c_extent > 0) {
    // the 5th-generation tensor cores (tcgen05, accumulator in tensor memory), for products
    // whose layout, epilogue and alignment its kernel takes; the others stay on mma.sync
    gem::tc::Args t;
    std::memset(&t, 0, sizeof(t));
    t.M = a.M;
    t.N = a.N;
    t.K = a.K;
    t.A = gem::tc::Operand{a.A.base, a.A.group_stride, a.A.ld, a.a_extent, a.A.by_worker, a.a_rounded};
    t.B = gem::tc::Operand{a.B.base, a.B.group_stride, a.B.ld, a.b_extent, a.B.by_worker, a.b_rounded};
    t.C = a.C;
    t.c_group_stride = a.c_group_stride;
    t.ldc = a.ldc;
    t.c_extent = a.c_extent;
    t.round_c = a.round_c;
    t.ct = a.ct;
    t.ct_group_stride = a.ct_group_stride;
    t.ldct = a.ldct;
    t.ct_extent = a.ct_extent;
    t.bias = a.bias;
    t.bias_group_stride = a.bias_group_stride;
    t.bias_extent = a.bias_extent;
    t.mask = a.mask;
    t.mask_group_stride = a.mask_group_stride;
    t.ldmask = a.ldmask;
    t.mask_extent = a.mask_extent;
    t.status = a.status;
    for (int g = 0; g < groups && g < kMaxGroups; ++g) t.workers[g] = a.workers[g];
    if (gem::tc::supported(t, AK, BK_, EPI, groups)) {
      if (on_tc) *on_tc = true;
      return gem::tc::launch(t, groups, AK, BK_, EPI, st);
    }
  }
  const long long mt = (a.M + 127) / 128, nt64 = (a.N + 63) / 64, nt128 = (a.N + 127) / 128;
  const long long big = (tc ? nt128 : nt64) * mt * groups;
  if (big >= (tc ? GEM_TF32_BIG_TILE_BLOCKS : GEM_SIMT_BIG_TILE_BLOCKS) * kSmCountHint) {
    if (tc)
      launch_mma<128, AK, BK_, EPI>(a, groups, st);
    else
      launch_tile<128, AK, BK_, EPI>(a, groups, tf32, st);
    return cudaGetLastError();
  }
  const long long small = tc ? nt64 * mt * groups : nt64 * ((a.M + 63) / 64) * groups;
  int split = 1;
  const long long mn = (long long)a.M * a.N * groups;
  const int min_chunk = tc ? GEM_TF32_MIN_CHUNK : GEM_SIMT_MIN_CHUNK;   // the tensor cores get through K faster
  if (a.ws && a.M <= 128)
    while (split < kMaxSplit && small * split < 4 * kSmCountHint && a.K / (2 * split) >= min_chunk &&
           mn * 2 * split <= a.ws_floats)
      split *= 2;
  if (split > 1) {
    a.ksplit = split;
    a.kchunk = ((a.K + split - 1) / split + BK - 1) / BK * BK;
  }
  if (tc)
    launch_mma<64, AK, BK_, EPI>(a, groups * split, st);
  else
    launch_tile<64, AK, BK_, EPI>(a, groups * split, tf32, st);
  if (split > 1) {
    // float4 columns when every row of every array starts on a 16-byte boundary
    auto al = [](const void* ptr, long long stride) {
      return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0 && stride % 4 == 0;
    };
    const bool vec = a.N % 4 == 0 && al(a.C, a.c_group_stride) && a.ldc % 4 == 0 &&
                     (!(EPI == kBias || EPI == kBiasRelu) || al(a.bias, a.bias_group_stride)) &&
                     (EPI != kMask || (al(a.mask, a.mask_group_stride) && a.ldmask % 4 == 0));
    const int V = vec ? 4 : 1;
    dim3 grid(unsigned((a.N + 256 * V - 1) / (256 * V)), unsigned(a.M * groups));
    if (vec)
      gem::launch_pdl(splitk_reduce_kernel<EPI, 4>, grid, 256, 0, st, a);
    else
      gem::launch_pdl(splitk_reduce_kernel<EPI, 1>, grid, 256, 0, st, a);
  }
  return cudaGetLastError();
}

}  // namespace mlp
}  // namespace gem

using namespace gem::mlp;




namespace {

long long round32(long long x) { return (x + 31) / 32 * 32; }

int cuda_rc(cudaError_t e) { return e == cudaSuccess ? GEM_OK : GEM_ECUDA; }

}  // namespace

namespace gem {
namespace mlp {

int mlp_chunk(gem_mlp* M, const int32_t* workers, int G, const int32_t* batch_rows,
              float* grads, long long grad_stride, float* losses) {
  gem_t* h = M->gem;
  cudaStream_t st = h->stream;
  const bool tf32 = M->precision == GEM_MLP_TF32;
  const int L = M->L, b = M->batch;
  const long long S = M->slot_stride;
  float* scr = M->scratch;
  auto act = [&](int l) -> float* { return l == 0 ? scr + M->off_x : scr + M->off_act[l]; };

  int rc = GEM_OK;
  if (!M->external_input) {
    gem::launch_pdl(gather_rows_kernel, dim3(b, G), 256, 0, st, M->X, M->dims[0], batch_rows, b,
                                                   scr + M->off_x, S, tf32 ? 1 : 0);
    if ((rc = cuda_rc(cudaGetLastError()))) return rc;
    M->launches++;
  }

  GemmArgs a;
  std::memset(&a, 0, sizeof(a));
  for (int g = 0; g < G; ++g) a.workers[g] = workers[g];
  a.ws = M->ws;
  a.ws_floats = M->ws_floats;
  a.status = M->tc_status;
  const long long wstride = (long long)h->stride;
  // floats addressable from p when it lies in the scratch or in the snapshots (0 otherwise)
  const float* snap_end = h->s + (long long)h->n * wstride;
  auto ext = [&](const float* p) -> long long {
    if (!p) return 0;
    if (M->scratch_end && p >= M->scratch && p < M->scratch_end) return M->scratch_end - p;
    if (p >= h->s && p < snap_end) return snap_end - p;
    return 0;
  };
  // the operands, bias and mask of a product in the scratch or the snapshots, its output
  // in the scratch or in the gradient rows (the region the product writes)
  auto set_extents = [&](GemmArgs& x, int groups) {
    x.a_extent = ext(x.A.base);
    x.b_extent = ext(x.B.base);
    x.bias_extent = ext(x.bias);
    x.mask_extent = ext(x.mask);
    x.c_extent = ext(x.C);
    if (x.c_extent == 0)
      x.c_extent = (long long)(groups - 1) * x.c_group_stride + (long long)(x.M - 1) * x.ldc + x.N;
  };

  // Which activations hold TF32 values already (tensor-core products then read them without
  // rounding again): the gathered rows (rounded by the gather) and activations stored
  // rounded by a tensor-core forward product.
  bool act_rnd[kMaxLayers + 1] = {};
  act_rnd[0] = tf32 && !M->external_input;
  // Weight gradients dW_l = D_{l+1}^T A_l that run on the tensor cores read the minibatch
  // panels K-major (K = the batch): TF32-rounded transposes A_l^T and D_{l+1}^T.  A hidden
  // activation's transpose comes from the epilogue of the tensor-core product that makes it;
  // X^T and the deltas' transposes from transpose_round_kernel on the side stream, next to
  // the main stream's chain.
  auto t_dw = [&](int l) {
    return M->has_t && l + 1 < L && M->dims[l + 1] >= 32 && b >= 32 && b % 4 == 0;
  };
  TransposeArgs ta;
  std::memset(&ta, 0, sizeof(ta));
  for (int g = 0; g < G; ++g) ta.workers[g] = workers[g];
  auto transpose = [&](cudaStream_t s, const float* src, long long src_stride, bool by_worker,
                       float* dst, int rows, int cols) -> int {
    ta.src = src;
    ta.src_stride = src_stride;
    ta.by_worker = by_worker ? 1 : 0;
    ta.dst = dst;
    ta.dst_stride = S;
    ta.rows = rows;
    ta.cols = cols;
    gem::launch_pdl(transpose_round_kernel, dim3((cols + 31) / 32, (rows + 31) / 32, G), 256, 0, s, ta);
    M->launches++;
    return cuda_rc(cudaGetLastError());
  };
  const bool two_streams = M->side != nullptr;
  cudaStream_t wst = two_streams ? M->side : st;
  if (t_dw(0)) {   // X^T on the side stream, after the gather
    if (two_streams) {
      if ((rc = cuda_rc(cudaEventRecord(M->ev_x, st)))) return rc;
      if ((rc = cuda_rc(cudaStreamWaitEvent(wst, M->ev_x, 0)))) return rc;
    }
    if ((rc = transpose(wst, scr + M->off_x, S, false, scr + M->off_actT[0], b, M->dims[0]))) return rc;
  }

  // forward
  bool fused_loss = false;   // the logits kernel also produced the loss gradient
  for (int l = 0; l < L; ++l) {
    const int din = M->dims[l], dout = M->dims[l + 1];
    a.M = b; a.N = dout; a.K = din;
    a.A = Operand{act(l), S, din, 0};
    a.B = Operand{h->s + M->w_off[l], wstride, din, 1};
    a.bias = h->s + M->b_off[l];
    a.bias_group_stride = wstride;
    const bool last = l == L - 1;
    a.C = last ? scr + M->off_logits : act(l + 1);
    a.c_group_stride = S;
    a.ldc = dout;
    cudaError_t e;
    XentArgs xa;
    xa.labels = M->labels;
    xa.batch_rows = batch_rows;
    xa.delta = scr + M->off_delta[L];
    xa.row_loss = scr + M->off_row_loss;
    xa.group_stride = S;
    xa.b = b;
    if (last && dout <= kMaxClasses &&
        (tf32 ? launch_small_n<true>(a, G, st, &e, &xa) : launch_small_n<false>(a, G, st, &e, &xa))) {
      // the logits: few outputs per row, the worker's weights held in shared memory, and
      // the loss with its gradient in the same kernel
      fused_loss = true;
    } else {
      set_extents(a, G);
      a.a_rounded = act_rnd[l] ? 1 : 0;
      a.b_rounded = 0;
      a.round_c = (!last && tf32) ? 1 : 0;   // hidden activations: only ever operands and masks
      const bool want_t = !last && t_dw(l + 1);
      if (want_t) {
        a.ct = scr + M->off_actT[l + 1];
        a.ct_group_stride = S;
        a.ldct = b;
        a.ct_extent = ext(a.ct);
      }
      bool on_tc = false;
      e = last ? launch_gemm<true, true, kBias>(a, G, tf32, st, &on_tc)
               : launch_gemm<true, true, kBiasRelu>(a, G, tf32, st, &on_tc);
      if (!last) act_rnd[l + 1] = on_tc && a.round_c;
      a.round_c = 0;
      a.ct = nullptr;
      if ((rc = cuda_rc(e))) return rc;
      M->launches++;
      if (want_t && !on_tc &&
          (rc = transpose(st, act(l + 1), S, false, scr + M->off_actT[l + 1], b, dout)))
        return rc;
      continue;
    }
    if ((rc = cuda_rc(e))) return rc;
    M->launches++;
  }
  if (!fused_loss) {
    gem::launch_pdl(softmax_xent_kernel, G, 128, 0, st, scr + M->off_logits, scr + M->off_delta[L], S,
                    b, M->dims[L], M->labels, batch_rows, losses);
    if ((rc = cuda_rc(cudaGetLastError()))) return rc;
    M->launches++;
  }

  // backward.  The weight-gradient products go to the side stream when there is one: each
  // waits for its delta D_{l+1} (event recorded on the main stream) and runs next to the
  // input-gradient chain; they use no split-K workspace, which belongs to the main stream.
  for (int l = L - 1; l >= 0; --l) {
    const int din = M->dims[l], dout = M->dims[l + 1];
    if (two_streams) {
      if ((rc = cuda_rc(cudaEventRecord(M->ev_delta[l + 1], st)))) return rc;
      if ((rc = cuda_rc(cudaStreamWaitEvent(wst, M->ev_delta[l + 1], 0)))) return rc;
    }
    // dW_l = D_{l+1}^T A_l: (m = o, k = r) from D [b x dout], (k = r, n = j) from A [b x din],
    // or from the transposes D^T [dout x b] and A^T [din x b], both K-major and TF32
    GemmArgs w = a;
    w.M = dout; w.N = din; w.K = b;
    w.round_c = 0;
    w.C = grads + M->w_off[l];
    w.c_group_stride = grad_stride;
    w.ldc = din;
    if (two_streams) w.ws = nullptr;
    w.bias = nullptr;
    w.mask = nullptr;
    cudaError_t ew;
    if (t_dw(l)) {
      // D_{l+1}^T, on the weight-gradient stream (the input-gradient chain goes on)
      if ((rc = transpose(wst, scr + M->off_delta[l + 1], S, false, scr + M->off_deltaT[l + 1], b, dout)))
        return rc;
      w.A = Operand{scr + M->off_deltaT[l + 1], S, b, 0};
      w.B = Operand{scr + M->off_actT[l], S, b, 0};
      w.a_rounded = 1;
      w.b_rounded = 1;
      set_extents(w, G);
      ew = launch_gemm<true, true, kStore>(w, G, tf32, wst);
    } else {
      w.A = Operand{scr + M->off_delta[l + 1], S, dout, 0};
      w.B = Operand{act(l), S, din, 0};
      w.a_rounded = 0;
      w.b_rounded = 0;
      set_extents(w, G);
      ew = launch_gemm<false, false, kStore>(w, G, tf32, wst);
    }
    if ((rc = cuda_rc(ew))) return rc;
    M->launches++;
    if (l == 0) {
      if (!M->input_grad) break;
      // D_0 = D_1 W_0, the gradient with respect to the input rows (no activation here)
      a.M = b; a.N = din; a.K = dout;
      a.A = Operand{scr + M->off_delta[1], S, dout, 0};
      a.B = Operand{h->s + M->w_off[0], wstride, din, 1};
      a.C = scr + M->off_delta[0];
      a.c_group_stride = S;
      a.ldc = din;
      a.bias = nullptr;
      a.mask = nullptr;
      set_extents(a, G);
      if ((rc = cuda_rc(launch_gemm<true, false, kStore>(a, G, tf32, st)))) return rc;
      M->launches++;
      break;
    }
    // D_l = (D_{l+1} W_l) * [A_l > 0]: (m = r, k = o) from D, (k = o, n = j) from W_l [dout x din]
    a.M = b; a.N = din; a.K = dout;
    a.A = Operand{scr + M->off_delta[l + 1], S, dout, 0};
    a.C = scr + M->off_delta[l];
    a.c_group_stride = S;
    a.ldc = din;
    a.mask = act(l);
    a.mask_group_stride = S;
    a.ldmask = din;
    a.B = Operand{h->s + M->w_off[l], wstride, din, 1};
    a.bias = nullptr;
    a.a_rounded = 0;
    a.b_rounded = 0;
    a.round_c = 0;
    set_extents(a, G);
    if ((rc = cuda_rc(launch_gemm<true, false, kMask>(a, G, tf32, st)))) return rc;
    M->launches++;
  }
  BiasGradArgs ba;
  std::memset(&ba, 0, sizeof(ba));
  ba.n_layers = L;
  ba.b = b;
  ba.row_loss_off = M->off_row_loss;
  ba.losses = fused_loss ? losses : nullptr;
  ba.first[0] = 0;
  for (int l = 0; l < L; ++l) {
    ba.grad_off[l] = M->b_off[l];
    ba.delta_off[l] = M->off_delta[l + 1];
    ba.width[l] = M->dims[l + 1];
    ba.first[l + 1] = ba.first[l] + M->dims[l + 1];
  }
  gem::launch_pdl(bias_grad_kernel, dim3((ba.first[L] + 31) / 32, G), 256, 0, st, ba, scr, S, grads,
                                                                      grad_stride);
  if ((rc = cuda_rc(cudaGetLastError()))) return rc;
  M->launches++;
  if (two_streams) {   // the gradients are complete once the side stream is
    if ((rc = cuda_rc(cudaEventRecord(M->ev_side, wst)))) return rc;
    if ((rc = cuda_rc(cudaStreamWaitEvent(st, M->ev_side, 0)))) return rc;
  }
  return GEM_OK;
}

int mlp_build(gem_t* g, int n_layers, const int32_t* dims, int batch, int precision,
              long long param_base, bool external_input, bool input_grad, bool own_grads,
              gem_mlp** out) {
  *out = nullptr;
  gem_mlp* M = new (std::nothrow) gem_mlp();
  if (!M) return GEM_ENOMEM;
  M->gem = g;
  M->L = n_layers;
  M->batch = batch;
  M->precision = precision;
  M->param_base = param_base;
  M->external_input = external_input;
  M->input_grad = input_grad;
  long long P = param_base;
  for (int l = 0; l <= n_layers; ++l) M->dims[l] = dims[l];
  for (int l = 0; l < n_layers; ++l) {
    M->w_off[l] = P;
    M->b_off[l] = P + (long long)dims[l + 1] * dims[l];
    P = M->b_off[l] + dims[l + 1];
  }
  long long off = 0;
  M->off_x = off;
  off += round32((long long)batch * dims[0]);
  for (int l = 1; l < n_layers; ++l) {
    M->off_act[l] = off;
    off += round32((long long)batch * dims[l]);
  }
  M->off_logits = off;
  off += round32((long long)batch * dims[n_layers]);
  for (int l = input_grad ? 0 : 1; l <= n_layers; ++l) {
    M->off_delta[l] = off;
    off += round32((long long)batch * dims[l]);
  }
  M->off_row_loss = off;
  off += round32(batch);
  if (precision == GEM_MLP_TF32 && !external_input) {
    M->has_t = true;
    for (int l = 0; l + 1 < n_layers; ++l) {   // A_l^T for the weight gradients dW_l, l < L - 1
      M->off_actT[l] = off;
      off += round32((long long)batch * dims[l]);
    }
    for (int l = 1; l < n_layers; ++l) {       // D_l^T, l = 1 .. L - 1
      M->off_deltaT[l] = off;
      off += round32((long long)batch * dims[l]);
    }
  }
  M->slot_stride = off;
  M->slots = g->n < kMaxGroups ? g->n : kMaxGroups;
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(g->device);
  cudaError_t e = cudaMalloc(&M->scratch, sizeof(float) * size_t(M->slot_stride) * M->slots);
  if (e == cudaSuccess) M->scratch_end = M->scratch + M->slot_stride * M->slots;
  if (e == cudaSuccess && precision == GEM_MLP_TF32) {
    e = cudaMalloc(&M->tc_status, sizeof(unsigned));
    if (e == cudaSuccess) e = cudaMemset(M->tc_status, 0, sizeof(unsigned));
  }
  if (e == cudaSuccess && own_grads) e = cudaMalloc(&M->grads, sizeof(float) * g->stride * size_t(g->n));
  if (e == cudaSuccess && batch <= 128) {
    // split-K workspace: kMaxSplit partial products of at most batch x widest layer per slot
    int widest = 0;
    for (int l = input_grad ? 0 : 1; l <= n_layers; ++l) widest = dims[l] > widest ? dims[l] : widest;
    M->ws_floats = (long long)kMaxSplit * 128 * widest * M->slots;
    e = cudaMalloc(&M->ws, sizeof(float) * size_t(M->ws_floats));
  }
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&M->side, cudaStreamNonBlocking);
  for (int l = 0; l <= n_layers && e == cudaSuccess; ++l)
    e = cudaEventCreateWithFlags(&M->ev_delta[l], cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&M->ev_side, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&M->ev_x, cudaEventDisableTiming);
  cudaSetDevice(dev_prev);
  if (e != cudaSuccess) {
    cudaGetLastError();
    mlp_free(M);
    return GEM_ENOMEM;
  }
  *out = M;
  return GEM_OK;
}

void mlp_free(gem_mlp* M) {
  if (!M) return;
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(M->gem->device);
  cudaStreamSynchronize(M->gem->stream);
  if (M->side) cudaStreamSynchronize(M->side);
  for (int l = 0; l <= kMaxLayers; ++l)
    if (M->ev_delta[l]) cudaEventDestroy(M->ev_delta[l]);
  if (M->ev_side) cudaEventDestroy(M->ev_side);
  if (M->ev_x) cudaEventDestroy(M->ev_x);
  if (M->side) cudaStreamDestroy(M->side);
  cudaFree(M->scratch);
  cudaFree(M->tc_status);
  cudaFree(M->grads);
  cudaFree(M->ws);
  cudaFree(M->pi_rows);
  cudaFree(M->rows_dev);
  cudaGetLastError();
  cudaSetDevice(dev_prev);
  delete M;
}

}  // namespace mlp
}  // namespace gem

namespace {

// Check minibatch rows on the host and copy them to the device (stream-ordered).
int upload_rows(gem_mlp* M, const int32_t* rows_host, long long count) {
  for (long long i = 0; i < count; ++i)
    if (rows_host[i] < 0 || rows_host[i] >= M->rows) return GEM_EINVAL;
  if ((size_t)count > M->rows_cap) {
    cudaFree(M->rows_dev);  // synchronises with work still reading the old buffer
    M->rows_dev = nullptr;
    M->rows_cap = 0;
    if (cudaMalloc(&M->rows_dev, sizeof(int32_t) * size_t(count)) != cudaSuccess) {
      cudaGetLastError();
      return GEM_ENOMEM;
    }
    M->rows_cap = size_t(count);
  }
  return cuda_rc(cudaMemcpyAsync(M->rows_dev, rows_host, sizeof(int32_t) * size_t(count),
                                 cudaMemcpyHostToDevice, M->gem->stream));
}

}  // namespace

extern "C" {

int gem_mlp_create(gem_t* g, int n_layers, const int32_t* dims, int batch, int precision,
                   gem_mlp_t** out) {
  if (!out) return GEM_EINVAL;
  *out = nullptr;
  if (!g || !dims || n_layers < 1 || n_layers > kMaxLayers || batch < 1 || batch > kMaxBatch)
    return GEM_EINVAL;
  if (precision != GEM_MLP_FP32 && precision != GEM_MLP_TF32) return GEM_EINVAL;
  if (g->broken) return GEM_ESTATE;
  long long P = 0;
  for (int l = 0; l <= n_layers; ++l)
    if (dims[l] < 1) return GEM_EINVAL;
  if (dims[n_layers] > kMaxClasses) return GEM_EINVAL;
  for (int l = 0; l < n_layers; ++l) P += (long long)dims[l + 1] * dims[l] + dims[l + 1];
  if ((size_t)P != g->P) return GEM_EINVAL;
  return mlp_build(g, n_layers, dims, batch, precision, 0, false, false, true, out);
}

void gem_mlp_destroy(gem_mlp_t* M) { mlp_free(M); }

int gem_mlp_set_data(gem_mlp_t* M, const float* X, const int32_t* labels, int64_t rows) {
  if (!M || !X || !labels || rows < 1) return GEM_EINVAL;
  M->X = X;
  M->labels = labels;
  M->rows = rows;
  return GEM_OK;
}

uint64_t gem_mlp_launch_count(const gem_mlp_t* M) { return M ? M->launches : 0; }

int gem_mlp_status(gem_mlp_t* M) {
  if (!M) return GEM_EINVAL;
  gem_t* h = M->gem;
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(h->device);
  cudaError_t e = cudaStreamSynchronize(h->stream);
  if (e == cudaSuccess && M->side) e = cudaStreamSynchronize(M->side);
  unsigned tc = 0;   // a tensor-core product that gave up a wait or skipped an access
  if (e == cudaSuccess && M->tc_status)
    e = cudaMemcpy(&tc, M->tc_status, sizeof(unsigned), cudaMemcpyDeviceToHost);
  cudaSetDevice(dev_prev);
  if (e != cudaSuccess || tc != 0) {
    h->broken = true;
    return GEM_ECUDA;
  }
  return GEM_OK;
}

int gem_mlp_grad(gem_mlp_t* M, const int32_t* workers, int L, const int32_t* batch_rows,
                 float* const* grads, float* losses) {
  if (!M || L < 0 || (L > 0 && (!workers || !batch_rows || !grads))) return GEM_EINVAL;
  if (!M->X) return GEM_EINVAL;
  gem_t* h = M->gem;
  if (h->broken) return GEM_ESTATE;
  for (int i = 0; i < L; ++i) {
    if (workers[i] < 0 || workers[i] >= h->n || !grads[i]) return GEM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(grads[i]) & 15u) != 0) return GEM_EINVAL;
  }
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(h->device);
  int rc = upload_rows(M, batch_rows, (long long)L * M->batch);
  for (int c0 = 0; c0 < L && rc == GEM_OK; c0 += M->slots) {
    const int G = (L - c0) < M->slots ? (L - c0) : M->slots;
    rc = mlp_chunk(M, workers + c0, G, M->rows_dev + (long long)c0 * M->batch, M->grads,
                   (long long)h->stride, losses ? losses + c0 : nullptr);
    for (int g = 0; g < G && rc == GEM_OK; ++g)
      rc = cuda_rc(cudaMemcpyAsync(grads[c0 + g], M->grads + (long long)g * h->stride,
                                   h->P * sizeof(float), cudaMemcpyDeviceToDevice, h->stream));
  }
  if (rc == GEM_ECUDA) h->broken = true;
  cudaSetDevice(dev_prev);
  return rc;
}

}  // extern "C"

namespace {

// gem_mlp_run, with per-tensor factor medians when pi_lo is not null.
int mlp_run(gem_mlp_t* M, const int32_t* order, int T, const int32_t* batch_rows,
            float* losses, float* pi_lo, float* pi_hi) {
  if (!M || T < 0 || (T > 0 && (!order || !batch_rows))) return GEM_EINVAL;
  if (!M->X) return GEM_EINVAL;
  gem_t* h = M->gem;
  if (h->broken) return GEM_ESTATE;
  if (T == 0) return GEM_OK;
  const bool want_pi = pi_lo != nullptr;
  int64_t tensors[2 * kMaxLayers + 1];   // offsets of the tensors in the flat layout
  const int nseg = 2 * M->L;
  if (want_pi) {
    if (!pi_hi) return GEM_EINVAL;
    tensors[0] = 0;
    for (int l = 0; l < M->L; ++l) {
      tensors[2 * l + 1] = M->b_off[l];                     // end of W_l
      tensors[2 * l + 2] = M->b_off[l] + M->dims[l + 1];    // end of b_l
    }
  }
  std::vector<int32_t> seg(size_t(T) + 1);
  const int S = gem_plan_segments(order, T, h->n, seg.data());
  if (S < 0) return GEM_EINVAL;
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(h->device);
  int rc = upload_rows(M, batch_rows, (long long)T * M->batch);
  if (rc == GEM_OK && want_pi && !M->pi_rows) {
    if (cudaMalloc(&M->pi_rows, sizeof(float) * h->stride * size_t(h->n)) != cudaSuccess) {
      cudaGetLastError();
      M->pi_rows = nullptr;
      rc = GEM_ENOMEM;
    }
  }
  std::vector<const float*> gptr(size_t(T) > 0 ? size_t(T) : 1);
  std::vector<float*> pptr(want_pi ? size_t(T) : 1, nullptr);
  for (int i = 0; i < S && rc == GEM_OK; ++i) {
    const int a = seg[i], e = seg[i + 1];
    for (int c0 = a; c0 < e && rc == GEM_OK; c0 += M->slots) {
      const int G = (e - c0) < M->slots ? (e - c0) : M->slots;
      rc = mlp_chunk(M, order + c0, G, M->rows_dev + (long long)c0 * M->batch,
                     M->grads + (long long)(c0 - a) * h->stride, (long long)h->stride,
                     losses ? losses + c0 : nullptr);
    }
    if (rc == GEM_OK) {
      for (int k = a; k < e; ++k) {
        gptr[size_t(k)] = M->grads + (long long)(k - a) * h->stride;
        if (want_pi) pptr[size_t(k)] = M->pi_rows + (long long)(k - a) * h->stride;
      }
      if (!want_pi) {
        rc = cuda_rc(gem::commit_ordered(h, order + a, gptr.data() + a, e - a));
      } else {
        // commits with their factors recorded and counted, then the per-tensor medians
        const cudaError_t ce = gem::commit_pi_median_ordered(
            h, order + a, gptr.data() + a, e - a, pptr.data() + a, tensors, nseg,
            pi_lo + (long long)a * nseg, pi_hi + (long long)a * nseg);
        rc = ce == cudaErrorMemoryAllocation ? GEM_ENOMEM : cuda_rc(ce);
      }
    }
  }
  if (rc == GEM_ECUDA) h->broken = true;
  cudaSetDevice(dev_prev);
  return rc;
}

}  // namespace

extern "C" {

int gem_mlp_run(gem_mlp_t* M, const int32_t* order, int T, const int32_t* batch_rows,
                float* losses) {
  return mlp_run(M, order, T, batch_rows, losses, nullptr, nullptr);
}

int gem_mlp_run_pi(gem_mlp_t* M, const int32_t* order, int T, const int32_t* batch_rows,
                   float* losses, float* pi_lo, float* pi_hi) {
  if (!pi_lo || !pi_hi) return GEM_EINVAL;
  return mlp_run(M, order, T, batch_rows, losses, pi_lo, pi_hi);
}

}  // extern "C"

// ---------------------------------------------------------------------------------------
// Gradient without allocation (gem_mlp_grad_static).  Its scratch is this file-scope device
// array: every GPU that loads the library holds it until the process exits.  Host code
// cannot pass the symbol itself to a kernel (on the host it names a stand-in object, not
// device memory), so its device address is looked up once per device and context.
namespace {

constexpr long long kStaticScratchFloats = 1ll << 20;  // 4 MiB
__device__ __align__(256) float g_static_scratch[kStaticScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_static_mutex;
struct StaticAddress {
  CUcontext ctx;  // the context the address was looked up in
  float* addr;
};
StaticAddress g_static_addr[kMaxDevices] = {};

// The driver's current context, through the runtime's entry-point query (the library does
// not link the driver library itself, so it loads on machines without a GPU driver).
CUcontext current_context() {
  using GetCurrent = CUresult (*)(CUcontext*);
  static GetCurrent fn = nullptr;
  static bool looked = false;
  if (!looked) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<GetCurrent>(p);
    cudaGetLastError();
    looked = true;
  }
  CUcontext ctx = nullptr;
  if (!fn || fn(&ctx) != CUDA_SUCCESS) return nullptr;
  return ctx;
}

// Device address of g_static_scratch on the current device.  Looked up on the first call
// in a context, and again when the current context is another one (after a reset of the
// device's primary context, for instance).  Called with g_static_mutex held.
int static_scratch(int device, float** out) {
  if (device < 0 || device >= kMaxDevices) return GEM_EINVAL;
  StaticAddress& e = g_static_addr[device];
  CUcontext ctx = current_context();
  if (!e.addr || !ctx || e.ctx != ctx) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess || !ptr) {
      cudaGetLastError();
      return GEM_ECUDA;
    }
    // the lookup makes the device's primary context current if none was
    e.ctx = current_context();
    e.addr = static_cast<float*>(ptr);
  }
  *out = e.addr;
  return GEM_OK;
}

// The minibatch rows of one call, passed by value in the argument block and stored in the
// static array where the gradient kernels read them (no copy from pageable host memory).
struct StaticRows {
  int32_t row[kMaxBatch];
  int count;
};

__global__ void static_rows_kernel(const __grid_constant__ StaticRows a, int32_t* dst) {
  for (int i = threadIdx.x; i < a.count; i += blockDim.x) dst[i] = a.row[i];
}

}  // namespace

extern "C" int gem_mlp_grad_static(int n_layers, const int32_t* dims, int batch, int precision,
                                   const float* theta, const float* X, const int32_t* labels,
                                   int64_t rows, const int32_t* batch_rows, float* grad,
                                   float* loss, void* stream) {
  if (!dims || n_layers < 1 || n_layers > kMaxLayers || batch < 1 || batch > kMaxBatch)
    return GEM_EINVAL;
  if (precision != GEM_MLP_FP32 && precision != GEM_MLP_TF32) return GEM_EINVAL;
  if (!theta || !X || !labels || rows < 1 || !batch_rows || !grad) return GEM_EINVAL;
  if ((reinterpret_cast<uintptr_t>(grad) & 15u) != 0) return GEM_EINVAL;
  for (int l = 0; l <= n_layers; ++l)
    if (dims[l] < 1) return GEM_EINVAL;
  if (dims[n_layers] > kMaxClasses) return GEM_EINVAL;
  for (int i = 0; i < batch; ++i)
    if (batch_rows[i] < 0 || batch_rows[i] >= rows) return GEM_EINVAL;

  // descriptors on the stack: the snapshot is `theta`, one worker, one slot
  gem_ctx h{};
  gem_mlp M{};
  M.gem = &h;
  M.L = n_layers;
  M.batch = batch;
  M.precision = precision;
  M.X = X;
  M.labels = labels;
  M.rows = rows;
  long long P = 0;
  for (int l = 0; l <= n_layers; ++l) M.dims[l] = dims[l];
  for (int l = 0; l < n_layers; ++l) {
    M.w_off[l] = P;
    M.b_off[l] = P + (long long)dims[l + 1] * dims[l];
    P = M.b_off[l] + dims[l + 1];
  }
  long long off = 0;
  M.off_x = off;
  off += round32((long long)batch * dims[0]);
  for (int l = 1; l < n_layers; ++l) {
    M.off_act[l] = off;
    off += round32((long long)batch * dims[l]);
  }
  M.off_logits = off;
  off += round32((long long)batch * dims[n_layers]);
  for (int l = 1; l <= n_layers; ++l) {
    M.off_delta[l] = off;
    off += round32((long long)batch * dims[l]);
  }
  M.off_row_loss = off;
  off += round32(batch);
  M.slot_stride = off;
  M.slots = 1;
  const long long rows_floats = round32(batch);  // minibatch rows stored after the slot
  if (off + rows_floats > kStaticScratchFloats) return GEM_EINVAL;  // beyond the static array

  int device = 0;
  if (cudaGetDevice(&device) != cudaSuccess) {
    cudaGetLastError();
    return GEM_ECUDA;
  }
  float* scratch = nullptr;
  std::lock_guard<std::mutex> lock(g_static_mutex);
  int rc = static_scratch(device, &scratch);
  if (rc) return rc;
  h.device = device;
  h.P = size_t(P);
  h.stride = size_t(P);
  h.n = 1;
  h.s = const_cast<float*>(theta);
  h.stream = static_cast<cudaStream_t>(stream);
  M.scratch = scratch;
  int32_t* rows_dev = reinterpret_cast<int32_t*>(scratch + off);
  // an ordinary launch: it starts after all earlier work on the stream, including the
  // kernels of a previous call that still read the rows it overwrites
  StaticRows ra;
  std::memcpy(ra.row, batch_rows, sizeof(int32_t) * size_t(batch));
  ra.count = batch;
  static_rows_kernel<<<1, 256, 0, h.stream>>>(ra, rows_dev);
  if (cudaGetLastError() != cudaSuccess) return GEM_ECUDA;
  const int32_t worker = 0;
  rc = mlp_chunk(&M, &worker, 1, rows_dev, grad, 0, loss);
  M.gem = nullptr;
  return rc;
}
