// The MNIST convolutional network of Appendix A as the workers' model (include/gem_cnn.h).
//
// A segment of G distinct workers is processed together, each worker's layers reading
// its snapshot s_w:
//   conv1_pool_kernel      conv1 + bias, 2 x 2 max-pool, ReLU
//   conv2_pool_kernel      conv2 + bias, dropout scale, max-pool, ReLU -> the head's input
//                          (both keep, per pooled output, the position of the window's
//                          first maximum as one byte, for the backward routing)
//   dense head             fc1 -> fc2 -> fc3, softmax cross-entropy and the backward pass
//                          of the MLP engine, which also returns the gradient with respect
//                          to the features
//   pool2_back_kernel      ReLU mask, route to the window's first maximum, dropout scale
//   conv2_back_kernel      gradient with respect to conv1's pooled output, ReLU mask,
//                          route through pool1
//   conv2_wpart_kernel,    per-sample partial sums of the convolution weight and bias
//   conv1_wpart_kernel     gradients
//   conv_finish_kernel     sums of the partials over the minibatch, in sample order
// Every value is summed in a fixed order, so the gradients do not depend on timing.  The
// per-sample kernels stage a sample's maps and the worker's weights in shared memory; a
// shape whose staging exceeds 160 KB is refused.
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/gem_cnn.h"
#include "../../include/gem_sim.h"
#include "gem_internal.h"
#include "mlp_internal.h"
#include "pdl.h"

struct gem_cnn;

namespace {

using gem::mlp::kMaxGroups;

constexpr int kK = 5;  // kernel side
constexpr int kThreads = 256;
constexpr long long kMaxSampleSmem = 160 * 1024;   // per-sample staging, bytes

struct Shape {
  int H, c1, c2, f1, f2, C;
  int H1, P1, H2, P2, F;
  long long w1, b1, w2, b2, head, P;
};

bool make_shape(const int32_t* s, Shape& n) {
  if (!s) return false;
  n.H = s[0];
  n.c1 = s[1];
  n.c2 = s[2];
  n.f1 = s[3];
  n.f2 = s[4];
  n.C = s[5];
  if (n.H < kK || n.H > 1024 || n.c1 < 1 || n.c2 < 1 || n.f1 < 1 || n.f2 < 1 || n.C < 2 ||
      n.C > gem::mlp::kMaxClasses || n.c1 > 256 || n.c2 > 256)
    return false;
  n.H1 = n.H - (kK - 1);
  if (n.H1 % 2) return false;
  n.P1 = n.H1 / 2;
  n.H2 = n.P1 - (kK - 1);
  if (n.H2 < 2 || n.H2 % 2) return false;
  n.P2 = n.H2 / 2;
  n.F = n.c2 * n.P2 * n.P2;
  n.w1 = 0;
  n.b1 = n.w1 + (long long)n.c1 * kK * kK;
  n.w2 = n.b1 + n.c1;
  n.b2 = n.w2 + (long long)n.c2 * n.c1 * kK * kK;
  n.head = n.b2 + n.c2;
  n.P = n.head + (long long)n.f1 * n.F + n.f1 + (long long)n.f2 * n.f1 + n.f2 +
        (long long)n.C * n.f2 + n.C;
  return true;
}

long long round32(long long x) { return (x + 31) / 32 * 32; }

int cuda_rc(cudaError_t e) { return e == cudaSuccess ? GEM_OK : GEM_ECUDA; }

struct ConvArgs {
  int H, c1, c2, H1, P1, H2, P2, F, b, G;
  const float* X;              // [rows][H * H]
  const int32_t* rows;         // [G][b] minibatch rows
  const float* snap;           // GEM snapshots s, [n][snap_stride]
  long long snap_stride;
  long long w1, b1, w2, b2;    // parameter offsets
  const float* drop;           // [G][b][c2] dropout scales
  float* scr;                  // conv scratch, slot g at scr + g * S
  long long S;
  long long o_k1, o_a1, o_k2, o_dz2, o_dz1, o_p1, o_p2;   // o_k*: byte codes (offsets in floats)
  float* head;                 // dense head scratch, slot g at head + g * head_S
  long long head_S, head_x, head_dx;   // offsets of its input rows and input gradient
  float* grads;                // gradient of group g at grads + g * grad_stride
  long long grad_stride;
  int workers[kMaxGroups];
};

// Index of the first maximum of a 2 x 2 window (row-major), and its value in *mx.
__device__ __forceinline__ int first_max4(const float (&v)[4], float* mx) {
  int best = 0;
  float bv = v[0];
#pragma unroll
  for (int q = 1; q < 4; ++q)
    if (v[q] > bv) {
      best = q;
      bv = v[q];
    }
  *mx = bv;
  return best;
}

// The per-sample kernels below run one block per (slot g, sample i) (blockIdx.x = g b + i):
// the block first copies that sample's maps and the worker's weights into shared memory
// with asynchronous copies (every thread's copies in flight at once, so the block waits
// for about one memory latency rather than one per element), then its threads compute the
// sample's outputs from there.  Each output is summed in the same order as in the
// oracle's loops.
__device__ __forceinline__ void cp_async4(float* dst, const float* src) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(float* dst, const float* src) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
}

// Start copying n floats from global src to shared dst: 16-byte copies when both ends are
// 16-byte aligned, 4-byte copies for the rest.
__device__ __forceinline__ void stage(float* dst, const float* src, int n) {
  int head = 0;
  if (((reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(src)) & 15u) == 0) {
    const int n4 = n >> 2;
    for (int q = threadIdx.x; q < n4; q += blockDim.x) cp_async16(dst + 4 * q, src + 4 * q);
    head = n4 << 2;
  }
  for (int q = head + threadIdx.x; q < n; q += blockDim.x) cp_async4(dst + q, src + q);
}

// Wait for this thread's copies, then for the whole block's.
__device__ __forceinline__ void stage_wait() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
  __syncthreads();
}

// conv1 + bias, 2 x 2 max-pool, ReLU: thread per pooled output (co, py, px), the 6 x 6
// input patch of its window and the channel's 25 weights in registers.  HC: the input side
// when known at compile time (the paper's network: 28), 0 reads it from the arguments.
template <int HC>
__global__ void __launch_bounds__(kThreads) conv1_pool_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  extern __shared__ float sm[];
  const long long gi = blockIdx.x;
  const int g = int(gi / a.b), i = int(gi % a.b);
  const int H = HC ? HC : a.H, H1 = H - (kK - 1), P1 = H1 / 2;
  const float* th = a.snap + (long long)a.workers[g] * a.snap_stride;
  float* xs = sm;                                   // [H * H]
  float* ws = xs + H * H;                           // [c1][25]
  float* bs = ws + a.c1 * kK * kK;                  // [c1]
  stage(xs, a.X + (long long)a.rows[gi] * H * H, H * H);
  stage(ws, th + a.w1, a.c1 * kK * kK);
  stage(bs, th + a.b1, a.c1);
  stage_wait();
  uint8_t* k1s = reinterpret_cast<uint8_t*>(a.scr + g * a.S + a.o_k1) + (long long)i * a.c1 * P1 * P1;
  float* a1s = a.scr + g * a.S + a.o_a1 + (long long)i * a.c1 * P1 * P1;
  for (int q = threadIdx.x; q < a.c1 * P1 * P1; q += blockDim.x) {
    const int px = q % P1, py = q / P1 % P1, co = q / (P1 * P1);
    float x[kK + 1][kK + 1], w[kK * kK];
#pragma unroll
    for (int r = 0; r <= kK; ++r)
#pragma unroll
      for (int c = 0; c <= kK; ++c) x[r][c] = xs[(2 * py + r) * H + 2 * px + c];
#pragma unroll
    for (int k = 0; k < kK * kK; ++k) w[k] = ws[co * kK * kK + k];
    float v[4];
#pragma unroll
    for (int d = 0; d < 4; ++d) {
      float acc = bs[co];
#pragma unroll
      for (int ky = 0; ky < kK; ++ky)
#pragma unroll
        for (int kx = 0; kx < kK; ++kx) acc = fmaf(w[ky * kK + kx], x[(d >> 1) + ky][(d & 1) + kx], acc);
      v[d] = acc;
    }
    float m;
    k1s[q] = uint8_t(first_max4(v, &m));
    a1s[q] = m > 0.f ? m : 0.f;
  }
}

// conv2 + bias, dropout scale, 2 x 2 max-pool, ReLU -> the head's features: thread per
// pooled output (co, py, px), per input channel the 6 x 6 patch of its window and the 25
// weights in registers.  P1C: conv1's pooled side when known at compile time (12), 0 reads
// it from the arguments.
constexpr int kPool2Threads = 320;
template <int P1C>
__global__ void __launch_bounds__(kPool2Threads) conv2_pool_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  extern __shared__ float sm[];
  const long long gi = blockIdx.x;
  const int g = int(gi / a.b), i = int(gi % a.b);
  const int P1 = P1C ? P1C : a.P1, H2 = P1 - (kK - 1), P2 = H2 / 2;
  const float* th = a.snap + (long long)a.workers[g] * a.snap_stride;
  const int n_a1 = a.c1 * P1 * P1, n_w = a.c2 * a.c1 * kK * kK;
  float* a1s = sm;                                  // [c1][P1][P1]
  float* ws = a1s + n_a1;                           // [c2][c1][25]
  float* bs = ws + n_w;                             // [c2]
  stage(a1s, a.scr + g * a.S + a.o_a1 + (long long)i * n_a1, n_a1);
  stage(ws, th + a.w2, n_w);
  stage(bs, th + a.b2, a.c2);
  stage_wait();
  for (int q = threadIdx.x; q < a.c2 * P2 * P2; q += blockDim.x) {
    const int px = q % P2, py = q / P2 % P2, co = q / (P2 * P2);
    const float s = a.drop[gi * a.c2 + co];
    float v[4];
#pragma unroll
    for (int d = 0; d < 4; ++d) v[d] = bs[co];
    for (int ci = 0; ci < a.c1; ++ci) {
      const float* in = a1s + ci * P1 * P1;
      const float* wc = ws + (co * a.c1 + ci) * kK * kK;
      float x[kK + 1][kK + 1], w[kK * kK];
#pragma unroll
      for (int r = 0; r <= kK; ++r)
#pragma unroll
        for (int c = 0; c <= kK; ++c) x[r][c] = in[(2 * py + r) * P1 + 2 * px + c];
#pragma unroll
      for (int k = 0; k < kK * kK; ++k) w[k] = wc[k];
#pragma unroll
      for (int ky = 0; ky < kK; ++ky)
#pragma unroll
        for (int kx = 0; kx < kK; ++kx)
#pragma unroll
          for (int d = 0; d < 4; ++d) v[d] = fmaf(w[ky * kK + kx], x[(d >> 1) + ky][(d & 1) + kx], v[d]);
    }
#pragma unroll
    for (int d = 0; d < 4; ++d) v[d] = v[d] * s;   // dropout: the channel's scale
    float m;
    reinterpret_cast<uint8_t*>(a.scr + g * a.S + a.o_k2)[(long long)i * a.c2 * P2 * P2 + q] =
        uint8_t(first_max4(v, &m));
    a.head[g * a.head_S + a.head_x + (long long)i * a.F + q] = m > 0.f ? m : 0.f;
  }
}

// Gradient into conv2's (pre-dropout) output: the feature gradient through the ReLU, to
// the window's first maximum, times the channel's dropout scale; zeros elsewhere.
__global__ void __launch_bounds__(kThreads) pool2_back_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  const long long total = (long long)a.G * a.b * a.c2 * a.P2 * a.P2;
  const long long q = blockIdx.x * (long long)kThreads + threadIdx.x;
  if (q >= total) return;
  const int px = int(q % a.P2), py = int(q / a.P2 % a.P2);
  const int co = int(q / ((long long)a.P2 * a.P2) % a.c2);
  const long long gi = q / ((long long)a.P2 * a.P2 * a.c2);
  const int g = int(gi / a.b), i = int(gi % a.b);
  const long long f = (long long)i * a.F + (co * a.P2 + py) * a.P2 + px;
  const float feat = a.head[g * a.head_S + a.head_x + f];
  const float dfeat = a.head[g * a.head_S + a.head_dx + f];
  const float s = a.drop[gi * a.c2 + co];
  const long long base = g * a.S + ((long long)i * a.c2 + co) * a.H2 * a.H2;
  float* dz2 = a.scr + a.o_dz2 + base;
  const int am = reinterpret_cast<const uint8_t*>(a.scr + g * a.S + a.o_k2)
      [((long long)i * a.c2 + co) * a.P2 * a.P2 + py * a.P2 + px];
  const float gval = feat > 0.f ? dfeat * s : 0.f;
#pragma unroll
  for (int d = 0; d < 4; ++d) dz2[(2 * py + (d >> 1)) * a.H2 + 2 * px + (d & 1)] = d == am ? gval : 0.f;
}

// Gradient with respect to conv1's pooled outputs (sum over the conv2 outputs that read
// each, channels then kernel rows then columns), the ReLU mask, and the route through
// pool1 into conv1's output gradient.  A thread takes kBackRow consecutive outputs of one
// row (ci, py): the stretch of a dz2 row that a kernel row reads is loaded once into
// registers and serves all of them.  dz2 is staged with a row pitch of H2 + 1 floats,
// which spreads the rows that one warp reads over distinct banks.
constexpr int kBackRow = 12;
constexpr int kBackThreads = 128;
// H2C, P1C: conv2's output side and conv1's pooled side when known at compile time (the
// paper's network: 8 and 12), which folds the column bounds; 0 reads them from the
// arguments.  Threads take channels fastest, so the lanes of a warp share a few output
// rows: they read the same dz2 row stretch (a shared-memory broadcast) and skip the same
// kernel rows.
template <int H2C, int P1C>
__global__ void __launch_bounds__(kBackThreads) conv2_back_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  extern __shared__ float sm[];
  const long long gi = blockIdx.x;
  const int g = int(gi / a.b), i = int(gi % a.b);
  const float* th = a.snap + (long long)a.workers[g] * a.snap_stride;
  const int H2 = H2C ? H2C : a.H2, P1 = P1C ? P1C : a.P1, pitch = H2 + 1;
  const int n_dz2 = a.c2 * H2 * H2, n_w = a.c2 * a.c1 * kK * kK, n_a1 = a.c1 * P1 * P1;
  float* dzs = sm;                                  // [c2][H2][pitch]
  float* ws = dzs + a.c2 * H2 * pitch;              // [c2][c1][25]
  float* a1s = ws + n_w;                            // [c1][P1][P1]
  const float* dz_src = a.scr + g * a.S + a.o_dz2 + (long long)i * n_dz2;
  for (int q = threadIdx.x; q < n_dz2; q += blockDim.x) cp_async4(dzs + q / H2 * pitch + q % H2, dz_src + q);
  stage(ws, th + a.w2, n_w);
  stage(a1s, a.scr + g * a.S + a.o_a1 + (long long)i * n_a1, n_a1);
  stage_wait();
  const int H1 = 2 * P1;
  const uint8_t* k1s = reinterpret_cast<const uint8_t*>(a.scr + g * a.S + a.o_k1) + (long long)i * a.c1 * P1 * P1;
  float* dz1s = a.scr + g * a.S + a.o_dz1 + (long long)i * a.c1 * H1 * H1;
  const int nxb = (P1 + kBackRow - 1) / kBackRow;
  for (int q = threadIdx.x; q < a.c1 * P1 * nxb; q += blockDim.x) {
    const int ci = q % a.c1, rest = q / a.c1;
    const int xb = rest % nxb, py = rest / nxb;
    const int px0 = xb * kBackRow;
    // column t of the register stretch is dz2 column px0 - 4 + t
    bool col_ok[kBackRow + kK - 1];
#pragma unroll
    for (int t = 0; t < kBackRow + kK - 1; ++t) col_ok[t] = px0 - (kK - 1) + t >= 0 && px0 - (kK - 1) + t < H2;
    float acc[kBackRow];
#pragma unroll
    for (int j = 0; j < kBackRow; ++j) acc[j] = 0.f;
    for (int co = 0; co < a.c2; ++co) {
      const float* wc = ws + (co * a.c1 + ci) * kK * kK;
      const float* dc = dzs + co * H2 * pitch;
#pragma unroll
      for (int ky = 0; ky < kK; ++ky) {
        const int y = py - ky;
        if (y < 0 || y >= H2) continue;
        const float* drow = dc + y * pitch + px0 - (kK - 1);
        float d[kBackRow + kK - 1];
#pragma unroll
        for (int t = 0; t < kBackRow + kK - 1; ++t) d[t] = col_ok[t] ? drow[t] : 0.f;
        float w[kK];
#pragma unroll
        for (int kx = 0; kx < kK; ++kx) w[kx] = wc[ky * kK + kx];
#pragma unroll
        for (int j = 0; j < kBackRow; ++j)
#pragma unroll
          for (int kx = 0; kx < kK; ++kx)
            if (col_ok[j - kx + kK - 1]) acc[j] = fmaf(d[j - kx + kK - 1], w[kx], acc[j]);
      }
    }
    float* dz1 = dz1s + ci * H1 * H1;
#pragma unroll
    for (int j = 0; j < kBackRow; ++j) {
      const int px = px0 + j;
      if (px >= P1) break;
      const float dv = a1s[(ci * P1 + py) * P1 + px] > 0.f ? acc[j] : 0.f;
      const int am = k1s[(ci * P1 + py) * P1 + px];
#pragma unroll
      for (int d = 0; d < 4; ++d) dz1[(2 * py + (d >> 1)) * H1 + 2 * px + (d & 1)] = d == am ? dv : 0.f;
    }
  }
}

// Per-sample partial sums of conv2's weight and bias gradients, each over the output rows
// then columns.  A thread takes the kK weights (co, ci, ky, 0..kK-1) of one kernel row and
// slides a window of kK input values along each input row (one new load per column); the
// last c2 work items are the biases.
// H2C, P1C as in conv2_back_kernel.
template <int H2C, int P1C>
__global__ void __launch_bounds__(kThreads) conv2_wpart_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  extern __shared__ float sm[];
  const long long gi = blockIdx.x;
  const int g = int(gi / a.b), i = int(gi % a.b);
  const int H2 = H2C ? H2C : a.H2, P1 = P1C ? P1C : a.P1;
  const int n_dz2 = a.c2 * H2 * H2, n_a1 = a.c1 * P1 * P1;
  float* dzs = sm;                                  // [c2][H2][H2]
  float* a1s = dzs + n_dz2;                         // [c1][P1][P1]
  stage(dzs, a.scr + g * a.S + a.o_dz2 + (long long)i * n_dz2, n_dz2);
  stage(a1s, a.scr + g * a.S + a.o_a1 + (long long)i * n_a1, n_a1);
  stage_wait();
  const int per = a.c1 * kK * kK + 1;
  const int n_rows = a.c2 * a.c1 * kK;
  float* part = a.scr + g * a.S + a.o_p2 + (long long)i * a.c2 * per;
  for (int q = threadIdx.x; q < n_rows + a.c2; q += blockDim.x) {
    if (q >= n_rows) {
      const int co = q - n_rows;
      const float* dz2 = dzs + co * H2 * H2;
      float acc = 0.f;
      for (int p = 0; p < H2 * H2; ++p) acc += dz2[p];
      part[co * per + per - 1] = acc;
      continue;
    }
    const int ky = q % kK, ci = q / kK % a.c1, co = q / (kK * a.c1);
    const float* dz2 = dzs + co * H2 * H2;
    const float* in = a1s + (ci * P1 + ky) * P1;
    float acc[kK];
#pragma unroll
    for (int kx = 0; kx < kK; ++kx) acc[kx] = 0.f;
    for (int y = 0; y < H2; ++y) {
      const float* drow = dz2 + y * H2;
      const float* irow = in + y * P1;
      float win[kK];
#pragma unroll
      for (int kx = 0; kx < kK - 1; ++kx) win[kx] = irow[kx];
#pragma unroll 4
      for (int xx = 0; xx < H2; ++xx) {
        win[kK - 1] = irow[xx + kK - 1];
        const float dv = drow[xx];
#pragma unroll
        for (int kx = 0; kx < kK; ++kx) acc[kx] = fmaf(dv, win[kx], acc[kx]);
#pragma unroll
        for (int kx = 0; kx < kK - 1; ++kx) win[kx] = win[kx + 1];
      }
    }
#pragma unroll
    for (int kx = 0; kx < kK; ++kx) part[co * per + (ci * kK + ky) * kK + kx] = acc[kx];
  }
}

// Per-sample partial sums of conv1's weight and bias gradients, over the output rows then
// columns: a thread per kernel row (co, ky) with a sliding window as in conv2_wpart_kernel,
// then the c1 biases.
// H1C, HC: conv1's output side and the input side when known at compile time (the
// paper's network: 24 and 28); 0 reads them from the arguments.
constexpr int kW1Threads = 64;
template <int H1C, int HC>
__global__ void __launch_bounds__(kW1Threads) conv1_wpart_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  extern __shared__ float sm[];
  const long long gi = blockIdx.x;
  const int g = int(gi / a.b), i = int(gi % a.b);
  const int H1 = H1C ? H1C : a.H1, H = HC ? HC : a.H;
  const int n_dz1 = a.c1 * H1 * H1;
  float* dzs = sm;                                  // [c1][H1][H1]
  float* xs = dzs + n_dz1;                          // [H][H]
  stage(dzs, a.scr + g * a.S + a.o_dz1 + (long long)i * n_dz1, n_dz1);
  stage(xs, a.X + (long long)a.rows[gi] * H * H, H * H);
  stage_wait();
  constexpr int per = kK * kK + 1;
  const int n_rows = a.c1 * kK;
  float* part = a.scr + g * a.S + a.o_p1 + (long long)i * a.c1 * per;
  for (int q = threadIdx.x; q < n_rows + a.c1; q += blockDim.x) {
    if (q >= n_rows) {
      const int co = q - n_rows;
      const float* dz1 = dzs + co * H1 * H1;
      float acc = 0.f;
      for (int p = 0; p < H1 * H1; ++p) acc += dz1[p];
      part[co * per + per - 1] = acc;
      continue;
    }
    const int ky = q % kK, co = q / kK;
    const float* dz1 = dzs + co * H1 * H1;
    float acc[kK];
#pragma unroll
    for (int kx = 0; kx < kK; ++kx) acc[kx] = 0.f;
    for (int y = 0; y < H1; ++y) {
      const float* drow = dz1 + y * H1;
      const float* irow = xs + (y + ky) * H;
      float win[kK];
#pragma unroll
      for (int kx = 0; kx < kK - 1; ++kx) win[kx] = irow[kx];
#pragma unroll 4
      for (int xx = 0; xx < H1; ++xx) {
        win[kK - 1] = irow[xx + kK - 1];
        const float dv = drow[xx];
#pragma unroll
        for (int kx = 0; kx < kK; ++kx) acc[kx] = fmaf(dv, win[kx], acc[kx]);
#pragma unroll
        for (int kx = 0; kx < kK - 1; ++kx) win[kx] = win[kx + 1];
      }
    }
#pragma unroll
    for (int kx = 0; kx < kK; ++kx) part[co * per + ky * kK + kx] = acc[kx];
  }
}

// Convolution gradients: the partials summed over the minibatch in sample order.
__global__ void __launch_bounds__(kThreads) conv_finish_kernel(const __grid_constant__ ConvArgs a) {
  gem::pdl_entry();
  const int per1 = kK * kK + 1, per2 = a.c1 * kK * kK + 1;
  const long long n1 = (long long)a.c1 * per1, n2 = (long long)a.c2 * per2;
  const long long total = (long long)a.G * (n1 + n2);
  const long long q = blockIdx.x * (long long)kThreads + threadIdx.x;
  if (q >= total) return;
  const int g = int(q / (n1 + n2));
  const long long e = q % (n1 + n2);
  float* grad = a.grads + g * a.grad_stride;
  const float* slot = a.scr + g * a.S;
  float acc = 0.f;
  if (e < n1) {
    const int co = int(e / per1), k = int(e % per1);
    for (int i = 0; i < a.b; ++i) acc += slot[a.o_p1 + ((long long)i * a.c1 + co) * per1 + k];
    grad[k < per1 - 1 ? a.w1 + co * (per1 - 1) + k : a.b1 + co] = acc;
  } else {
    const long long e2 = e - n1;
    const int co = int(e2 / per2), k = int(e2 % per2);
    for (int i = 0; i < a.b; ++i) acc += slot[a.o_p2 + ((long long)i * a.c2 + co) * per2 + k];
    grad[k < per2 - 1 ? a.w2 + (long long)co * (per2 - 1) + k : a.b2 + co] = acc;
  }
}

unsigned blocks_for(long long n) { return unsigned((n + kThreads - 1) / kThreads); }

}  // namespace

struct gem_cnn {
  gem_t* gem = nullptr;
  Shape sh{};
  int batch = 0;
  gem_mlp* head = nullptr;   // fc1 -> fc2 -> fc3 and the loss, external input
  const float* X = nullptr;
  const int32_t* labels = nullptr;
  int64_t rows = 0;
  long long o_k1 = 0, o_a1 = 0, o_k2 = 0, o_dz2 = 0, o_dz1 = 0, o_p1 = 0, o_p2 = 0;
  long long slot_stride = 0;
  int slots = 0;
  float* scratch = nullptr;
  float* grads = nullptr;        // [n][gem stride]
  int32_t* rows_dev = nullptr;   // minibatch rows uploaded from the host
  size_t rows_cap = 0;
  float* pi_rows = nullptr;      // [n][gem stride] scaling factors of a segment's commits
  int smem[5] = {};              // dynamic shared memory of the per-sample kernels (bytes)
  uint64_t launches = 0;
};

namespace {

// Forward and backward of groups [0, G) of one chunk (workers, rows [G][b] and dropout
// scales [G][b][c2] on the device), gradient of group g at grads + g * grad_stride.
int cnn_chunk(gem_cnn* N, const int32_t* workers, int G, const int32_t* rows_dev,
              const float* drop, float* grads, long long grad_stride, float* losses) {
  gem_t* h = N->gem;
  cudaStream_t st = h->stream;
  const Shape& s = N->sh;
  ConvArgs a;
  std::memset(&a, 0, sizeof(a));
  a.H = s.H; a.c1 = s.c1; a.c2 = s.c2; a.H1 = s.H1; a.P1 = s.P1; a.H2 = s.H2; a.P2 = s.P2;
  a.F = s.F; a.b = N->batch; a.G = G;
  a.X = N->X;
  a.rows = rows_dev;
  a.snap = h->s;
  a.snap_stride = (long long)h->stride;
  a.w1 = s.w1; a.b1 = s.b1; a.w2 = s.w2; a.b2 = s.b2;
  a.drop = drop;
  a.scr = N->scratch;
  a.S = N->slot_stride;
  a.o_k1 = N->o_k1; a.o_a1 = N->o_a1; a.o_k2 = N->o_k2; a.o_dz2 = N->o_dz2; a.o_dz1 = N->o_dz1;
  a.o_p1 = N->o_p1; a.o_p2 = N->o_p2;
  a.head = N->head->scratch;
  a.head_S = N->head->slot_stride;
  a.head_x = N->head->off_x;
  a.head_dx = N->head->off_delta[0];
  a.grads = grads;
  a.grad_stride = grad_stride;
  for (int g = 0; g < G; ++g) a.workers[g] = workers[g];
  const long long b = N->batch;
  const long long n_pool2 = G * b * s.c2 * s.P2 * s.P2;
  int rc;
  const unsigned samples = unsigned(G * b);
  if (s.H == 28) {
    gem::launch_pdl(conv1_pool_kernel<28>, samples, kThreads, N->smem[0], st, a);
    gem::launch_pdl(conv2_pool_kernel<12>, samples, kPool2Threads, N->smem[1], st, a);
  } else {
    gem::launch_pdl(conv1_pool_kernel<0>, samples, kThreads, N->smem[0], st, a);
    gem::launch_pdl(conv2_pool_kernel<0>, samples, kPool2Threads, N->smem[1], st, a);
  }
  if ((rc = cuda_rc(cudaGetLastError()))) return rc;
  N->launches += 2;
  // the dense head: forward, loss, backward, and the feature gradient
  if ((rc = gem::mlp::mlp_chunk(N->head, workers, G, rows_dev, grads, grad_stride, losses))) return rc;
  gem::launch_pdl(pool2_back_kernel, blocks_for(n_pool2), kThreads, 0, st, a);
  if (s.H == 28) {   // the paper's map sizes: loop bounds known at compile time
    gem::launch_pdl(conv2_back_kernel<8, 12>, samples, kBackThreads, N->smem[2], st, a);
    gem::launch_pdl(conv2_wpart_kernel<8, 12>, samples, kThreads, N->smem[3], st, a);
    gem::launch_pdl(conv1_wpart_kernel<24, 28>, samples, kW1Threads, N->smem[4], st, a);
  } else {
    gem::launch_pdl(conv2_back_kernel<0, 0>, samples, kBackThreads, N->smem[2], st, a);
    gem::launch_pdl(conv2_wpart_kernel<0, 0>, samples, kThreads, N->smem[3], st, a);
    gem::launch_pdl(conv1_wpart_kernel<0, 0>, samples, kW1Threads, N->smem[4], st, a);
  }
  gem::launch_pdl(conv_finish_kernel, blocks_for(G * ((long long)s.c1 * (kK * kK + 1) +
                                       (long long)s.c2 * (s.c1 * kK * kK + 1))), kThreads, 0, st, a);
  if ((rc = cuda_rc(cudaGetLastError()))) return rc;
  N->launches += 5;
  return GEM_OK;
}

// Check minibatch rows on the host and copy them to the device (stream-ordered).
int upload_rows(gem_cnn* N, const int32_t* rows_host, long long count) {
  for (long long i = 0; i < count; ++i)
    if (rows_host[i] < 0 || rows_host[i] >= N->rows) return GEM_EINVAL;
  if ((size_t)count > N->rows_cap) {
    cudaFree(N->rows_dev);   // synchronises with work still reading the old buffer
    N->rows_dev = nullptr;
    N->rows_cap = 0;
    if (cudaMalloc(&N->rows_dev, sizeof(int32_t) * size_t(count)) != cudaSuccess) {
      cudaGetLastError();
      return GEM_ENOMEM;
    }
    N->rows_cap = size_t(count);
  }
  return cuda_rc(cudaMemcpyAsync(N->rows_dev, rows_host, sizeof(int32_t) * size_t(count),
                                 cudaMemcpyHostToDevice, N->gem->stream));
}

}  // namespace

extern "C" {

int64_t gem_cnn_param_count(const int32_t* shape) {
  Shape s;
  return make_shape(shape, s) ? s.P : -1;
}

int gem_cnn_create(gem_t* g, const int32_t* shape, int batch, gem_cnn_t** out) {
  if (!out) return GEM_EINVAL;
  *out = nullptr;
  Shape s;
  if (!g || !make_shape(shape, s) || batch < 1 || batch > gem::mlp::kMaxBatch) return GEM_EINVAL;
  if (g->broken) return GEM_ESTATE;
  if ((size_t)s.P != g->P) return GEM_EINVAL;
  gem_cnn* N = new (std::nothrow) gem_cnn();
  if (!N) return GEM_ENOMEM;
  N->gem = g;
  N->sh = s;
  N->batch = batch;
  const int32_t dims[4] = {s.F, s.f1, s.f2, s.C};
  int rc = gem::mlp::mlp_build(g, 3, dims, batch, GEM_MLP_FP32, s.head, true, true, false, &N->head);
  if (rc) {
    delete N;
    return rc;
  }
  const long long b = batch;
  long long off = 0;
  auto take = [&](long long n) {
    const long long o = off;
    off += round32(n);
    return o;
  };
  N->o_k1 = take((b * s.c1 * s.P1 * s.P1 + 3) / 4);   // one byte per pooled output
  N->o_a1 = take(b * s.c1 * s.P1 * s.P1);
  N->o_k2 = take((b * s.c2 * s.P2 * s.P2 + 3) / 4);
  N->o_dz2 = take(b * s.c2 * s.H2 * s.H2);
  N->o_dz1 = take(b * s.c1 * s.H1 * s.H1);
  N->o_p1 = take(b * s.c1 * (kK * kK + 1));
  N->o_p2 = take(b * s.c2 * (s.c1 * kK * kK + 1));
  N->slot_stride = off;
  N->slots = N->head->slots;
  {
    const long long f = sizeof(float);
    const long long need[5] = {
        f * (s.H * s.H + s.c1 * kK * kK + s.c1),                                    // conv1_pool
        f * (s.c1 * s.P1 * s.P1 + (long long)s.c2 * s.c1 * kK * kK + s.c2),        // conv2_pool
        f * (s.c2 * s.H2 * (s.H2 + 1) + (long long)s.c2 * s.c1 * kK * kK + s.c1 * s.P1 * s.P1),  // conv2_back
        f * (s.c2 * s.H2 * s.H2 + s.c1 * s.P1 * s.P1),                              // conv2_wpart
        f * (s.c1 * s.H1 * s.H1 + s.H * s.H)};                                      // conv1_wpart
    // per kernel, the generic instantiation and the one for the paper's map sizes
    const void* fn[5][2] = {{(const void*)conv1_pool_kernel<0>, (const void*)conv1_pool_kernel<28>},
                            {(const void*)conv2_pool_kernel<0>, (const void*)conv2_pool_kernel<12>},
                            {(const void*)conv2_back_kernel<0, 0>, (const void*)conv2_back_kernel<8, 12>},
                            {(const void*)conv2_wpart_kernel<0, 0>, (const void*)conv2_wpart_kernel<8, 12>},
                            {(const void*)conv1_wpart_kernel<0, 0>, (const void*)conv1_wpart_kernel<24, 28>}};
    for (int k = 0; k < 5; ++k) {
      if (need[k] > kMaxSampleSmem) {   // a sample's maps and weights must fit on chip
        gem::mlp::mlp_free(N->head);
        delete N;
        return GEM_EINVAL;
      }
      N->smem[k] = int(need[k]);
      bool ok = true;
      for (int v = 0; v < 2 && need[k] > 48 * 1024; ++v)
        if (fn[k][v] && cudaFuncSetAttribute(fn[k][v], cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             int(need[k])) != cudaSuccess)
          ok = false;
      if (!ok) {
        cudaGetLastError();
        gem::mlp::mlp_free(N->head);
        delete N;
        return GEM_ECUDA;
      }
    }
  }
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(g->device);
  cudaError_t e = cudaMalloc(&N->scratch, sizeof(float) * size_t(N->slot_stride) * N->slots);
  if (e == cudaSuccess) e = cudaMalloc(&N->grads, sizeof(float) * g->stride * size_t(g->n));
  cudaSetDevice(dev_prev);
  if (e != cudaSuccess) {
    cudaGetLastError();
    cudaFree(N->scratch);
    cudaFree(N->grads);
    gem::mlp::mlp_free(N->head);
    delete N;
    return GEM_ENOMEM;
  }
  *out = N;
  return GEM_OK;
}

void gem_cnn_destroy(gem_cnn_t* N) {
  if (!N) return;
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(N->gem->device);
  cudaStreamSynchronize(N->gem->stream);
  cudaFree(N->scratch);
  cudaFree(N->grads);
  cudaFree(N->rows_dev);
  cudaFree(N->pi_rows);
  cudaGetLastError();
  cudaSetDevice(dev_prev);
  gem::mlp::mlp_free(N->head);
  delete N;
}

int gem_cnn_set_data(gem_cnn_t* N, const float* X, const int32_t* labels, int64_t rows) {
  if (!N || !X || !labels || rows < 1) return GEM_EINVAL;
  N->X = X;
  N->labels = labels;
  N->rows = rows;
  N->head->labels = labels;
  N->head->rows = rows;
  return GEM_OK;
}

int gem_cnn_status(gem_cnn_t* N) {
  if (!N) return GEM_EINVAL;
  return gem_sync(N->gem);
}

uint64_t gem_cnn_launch_count(const gem_cnn_t* N) {
  return N ? N->launches + N->head->launches : 0;
}

int gem_cnn_grad(gem_cnn_t* N, const int32_t* workers, int L, const int32_t* batch_rows,
                 const float* drop, float* const* grads, float* losses) {
  if (!N || L < 0 || (L > 0 && (!workers || !batch_rows || !grads || !drop))) return GEM_EINVAL;
  if (!N->X) return GEM_EINVAL;
  gem_t* h = N->gem;
  if (h->broken) return GEM_ESTATE;
  for (int i = 0; i < L; ++i) {
    if (workers[i] < 0 || workers[i] >= h->n || !grads[i]) return GEM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(grads[i]) & 15u) != 0) return GEM_EINVAL;
  }
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(h->device);
  int rc = upload_rows(N, batch_rows, (long long)L * N->batch);
  const long long db = (long long)N->batch * N->sh.c2;
  for (int c0 = 0; c0 < L && rc == GEM_OK; c0 += N->slots) {
    const int G = (L - c0) < N->slots ? (L - c0) : N->slots;
    rc = cnn_chunk(N, workers + c0, G, N->rows_dev + (long long)c0 * N->batch, drop + c0 * db,
                   N->grads, (long long)h->stride, losses ? losses + c0 : nullptr);
    for (int g = 0; g < G && rc == GEM_OK; ++g)
      rc = cuda_rc(cudaMemcpyAsync(grads[c0 + g], N->grads + (long long)g * h->stride,
                                   h->P * sizeof(float), cudaMemcpyDeviceToDevice, h->stream));
  }
  if (rc == GEM_ECUDA) h->broken = true;
  cudaSetDevice(dev_prev);
  return rc;
}

}  // extern "C"

namespace {

// gem_cnn_run, with per-tensor factor medians when pi_lo is not null.
int cnn_run(gem_cnn_t* N, const int32_t* order, int T, const int32_t* batch_rows,
            const float* drop, float* losses, float* pi_lo, float* pi_hi) {
  if (!N || T < 0 || (T > 0 && (!order || !batch_rows || !drop))) return GEM_EINVAL;
  if (!N->X) return GEM_EINVAL;
  gem_t* h = N->gem;
  if (h->broken) return GEM_ESTATE;
  if (T == 0) return GEM_OK;
  const bool want_pi = pi_lo != nullptr;
  if (want_pi && !pi_hi) return GEM_EINVAL;
  constexpr int kTensors = 10;
  int64_t tensors[kTensors + 1];
  {
    const Shape& sh = N->sh;
    const int64_t head = sh.head;
    const int64_t t[kTensors + 1] = {0, sh.b1, sh.w2, sh.b2, head, head + (int64_t)sh.f1 * sh.F,
                                     head + (int64_t)sh.f1 * sh.F + sh.f1,
                                     head + (int64_t)sh.f1 * sh.F + sh.f1 + (int64_t)sh.f2 * sh.f1,
                                     head + (int64_t)sh.f1 * sh.F + sh.f1 + (int64_t)sh.f2 * sh.f1 + sh.f2,
                                     sh.P - sh.C, sh.P};
    for (int i = 0; i <= kTensors; ++i) tensors[i] = t[i];
  }
  std::vector<int32_t> seg(size_t(T) + 1);
  const int S = gem_plan_segments(order, T, h->n, seg.data());
  if (S < 0) return GEM_EINVAL;
  int dev_prev = 0;
  cudaGetDevice(&dev_prev);
  cudaSetDevice(h->device);
  int rc = upload_rows(N, batch_rows, (long long)T * N->batch);
  if (rc == GEM_OK && want_pi && !N->pi_rows) {
    if (cudaMalloc(&N->pi_rows, sizeof(float) * h->stride * size_t(h->n)) != cudaSuccess) {
      cudaGetLastError();
      N->pi_rows = nullptr;
      rc = GEM_ENOMEM;
    }
  }
  std::vector<const float*> gptr(static_cast<size_t>(T));
  std::vector<float*> pptr(want_pi ? static_cast<size_t>(T) : 1, nullptr);
  const long long db = (long long)N->batch * N->sh.c2;
  for (int i = 0; i < S && rc == GEM_OK; ++i) {
    const int a = seg[i], e = seg[i + 1];
    for (int c0 = a; c0 < e && rc == GEM_OK; c0 += N->slots) {
      const int G = (e - c0) < N->slots ? (e - c0) : N->slots;
      rc = cnn_chunk(N, order + c0, G, N->rows_dev + (long long)c0 * N->batch, drop + c0 * db,
                     N->grads + (long long)(c0 - a) * h->stride, (long long)h->stride,
                     losses ? losses + c0 : nullptr);
    }
    if (rc == GEM_OK) {
      for (int k = a; k < e; ++k) {
        gptr[size_t(k)] = N->grads + (long long)(k - a) * h->stride;
        if (want_pi) pptr[size_t(k)] = N->pi_rows + (long long)(k - a) * h->stride;
      }
      if (!want_pi) {
        rc = cuda_rc(gem::commit_ordered(h, order + a, gptr.data() + a, e - a));
      } else {
        // commits with their factors recorded and counted, then the per-tensor medians
        const cudaError_t ce = gem::commit_pi_median_ordered(
            h, order + a, gptr.data() + a, e - a, pptr.data() + a, tensors, kTensors,
            pi_lo + (long long)a * kTensors, pi_hi + (long long)a * kTensors);
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

int gem_cnn_run(gem_cnn_t* N, const int32_t* order, int T, const int32_t* batch_rows,
                const float* drop, float* losses) {
  return cnn_run(N, order, T, batch_rows, drop, losses, nullptr, nullptr);
}

int gem_cnn_run_pi(gem_cnn_t* N, const int32_t* order, int T, const int32_t* batch_rows,
                   const float* drop, float* losses, float* pi_lo, float* pi_hi) {
  if (!pi_lo || !pi_hi) return GEM_EINVAL;
  return cnn_run(N, order, T, batch_rows, drop, losses, pi_lo, pi_hi);
}

}  // extern "C"
