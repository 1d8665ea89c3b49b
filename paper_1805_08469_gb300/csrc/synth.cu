// Device twin of the seeded input generators (include/gem_synth.h).  Inputs only: no
// GEM arithmetic lives here.  Integer operations, exact int->float conversions and single
// IEEE fp32 operations (the __f*_rn intrinsics, never contracted) make each value
// bit-identical to the host generator module.
#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/gem_synth.h"

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kStreamTheta0 = 1, kStreamGradZ = 2, kStreamGradT = 3, kStreamMask = 4,
                   kStreamDataX = 6, kStreamTeacher = 7, kStreamXavier = 8, kStreamDropout = 10,
                   kStreamCnnInit = 11, kStreamCnnTemplate = 12, kStreamCnnLabel = 13;
constexpr uint64_t kHeavyThresholdU24 = 1677722;  // ceil(0.1 * 2^24)

__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__host__ __device__ __forceinline__ uint64_t stream_key(uint64_t seed, uint64_t stream) {
  return mix64(seed * kGamma + stream);
}

__device__ __forceinline__ uint64_t draw(uint64_t key, uint64_t c) {
  return mix64(key + kGamma * (c + 1));
}

__device__ __forceinline__ int32_t normal_int(uint64_t key, uint64_t c) {
  const uint64_t c4 = c * 4;
  int64_t acc = 0;
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const uint64_t h = draw(key, c4 + r);
    acc += int64_t(((h >> 4) & 0xFFFFF) + ((h >> 24) & 0xFFFFF) + ((h >> 44) & 0xFFFFF));
  }
  return int32_t(acc - (int64_t(6) << 20));
}

__device__ __forceinline__ float normal(uint64_t key, uint64_t c) {
  return __fmul_rn(__int2float_rn(normal_int(key, c)), 0x1p-20f);
}

__device__ __forceinline__ float student_t3(uint64_t key, uint64_t c) {
  const uint64_t c4 = c * 4;
  const float z0 = normal(key, c4), z1 = normal(key, c4 + 1), z2 = normal(key, c4 + 2),
              z3 = normal(key, c4 + 3);
  float q = __fadd_rn(__fadd_rn(__fmul_rn(z1, z1), __fmul_rn(z2, z2)), __fmul_rn(z3, z3));
  q = __fdiv_rn(q, 3.0f);
  if (q == 0.0f) return 0.0f;
  return __fdiv_rn(z0, __fsqrt_rn(q));
}

unsigned grid_for(size_t n, unsigned threads) {
  size_t g = (n + threads - 1) / threads;
  if (g > 152u * 64u) g = 152u * 64u;  // grid-stride beyond this
  return unsigned(g < 1 ? 1 : g);
}

__global__ void theta0_kernel(uint64_t key, size_t P, float* out) {
  for (size_t j = blockIdx.x * size_t(blockDim.x) + threadIdx.x; j < P;
       j += size_t(gridDim.x) * blockDim.x)
    out[j] = __fmul_rn(0.05f, normal(key, j));
}

__global__ void heavytail_kernel(uint64_t kz, uint64_t kt, uint64_t kmask, uint64_t row0,
                                 int rows, size_t P, size_t ld, float* out) {
  const size_t total = size_t(rows) * P;
  for (size_t q = blockIdx.x * size_t(blockDim.x) + threadIdx.x; q < total;
       q += size_t(gridDim.x) * blockDim.x) {
    const size_t r = q / P, j = q - r * P;
    const uint64_t c = ((row0 + r) << 32) | uint64_t(j);
    const bool heavy = (draw(kmask, j) >> 40) < kHeavyThresholdU24;
    const float v = heavy ? student_t3(kt, c) : normal(kz, c);
    out[r * ld + j] = __fmul_rn(0.01f, v);
  }
}

__global__ void loguniform_kernel(uint64_t kz, uint64_t t, size_t P, const float* sigma,
                                  float* out) {
  for (size_t j = blockIdx.x * size_t(blockDim.x) + threadIdx.x; j < P;
       j += size_t(gridDim.x) * blockDim.x)
    out[j] = __fmul_rn(sigma[j], normal(kz, (t << 32) | uint64_t(j)));
}

__global__ void data_kernel(uint64_t kx, uint64_t kteach, int rows, int d_in, int classes,
                            float* X, int32_t* labels) {
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += gridDim.x * blockDim.x) {
    int64_t score[16];
    for (int c = 0; c < classes; ++c) score[c] = 0;
    for (int k = 0; k < d_in; ++k) {
      const uint64_t cx = uint64_t(r) * uint64_t(d_in) + uint64_t(k);
      const int32_t a = normal_int(kx, cx);
      X[size_t(r) * d_in + k] = __fmul_rn(__int2float_rn(a), 0x1p-20f);
      for (int c = 0; c < classes; ++c)
        score[c] += int64_t(a) * int64_t(normal_int(kteach, uint64_t(k) * classes + c));
    }
    int best = 0;
    for (int c = 1; c < classes; ++c)
      if (score[c] > score[best]) best = c;
    labels[r] = best;
  }
}

__global__ void xavier_kernel(uint64_t key, size_t count, int fan_in, float a, float* W) {
  for (size_t q = blockIdx.x * size_t(blockDim.x) + threadIdx.x; q < count;
       q += size_t(gridDim.x) * blockDim.x) {
    const float u = __fmul_rn(__uint2float_rn(unsigned(draw(key, q) >> 40)), 0x1p-24f);
    W[q] = __fmul_rn(a, __fsub_rn(__fmul_rn(2.0f, u), 1.0f));
  }
}

// Channel dropout scales: 0 where the 24-bit uniform of counter first + q is below p,
// else keep.
__global__ void dropout_kernel(uint64_t key, uint64_t first, size_t count, float p, float keep,
                               float* out) {
  for (size_t q = blockIdx.x * size_t(blockDim.x) + threadIdx.x; q < count;
       q += size_t(gridDim.x) * blockDim.x) {
    const float u = __fmul_rn(__uint2float_rn(unsigned(draw(key, first + q) >> 40)), 0x1p-24f);
    out[q] = u < p ? 0.0f : keep;
  }
}

// MNIST-shaped stand-in for the network: one thread block per row; label from the
// multiply-shift of a 32-bit draw, pixel = +-0.5 template cell of its class + normal noise.
__global__ void cnn_data_kernel(uint64_t kx, uint64_t kt, uint64_t ky, int rows, int H,
                                int classes, float* X, int32_t* labels) {
  const int cells = (H + 3) / 4;
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    const uint64_t h = draw(ky, uint64_t(r)) >> 32;
    const int y = int((h * uint64_t(classes)) >> 32);
    if (threadIdx.x == 0) labels[r] = y;
    for (int p = threadIdx.x; p < H * H; p += blockDim.x) {
      const int cell = ((y * cells) + (p / H) / 4) * cells + (p % H) / 4;
      const float t = (draw(kt, uint64_t(cell)) >> 63) ? -0.5f : 0.5f;
      X[size_t(r) * H * H + p] = __fadd_rn(t, normal(kx, uint64_t(r) * uint64_t(H * H) + p));
    }
  }
}

int launched() { return cudaGetLastError() == cudaSuccess ? 0 : -3; }

}  // namespace

extern "C" {

int gem_synth_theta0(uint64_t seed, size_t P, float* theta0, void* stream) {
  if (!theta0) return -1;
  if (P == 0) return 0;
  theta0_kernel<<<grid_for(P, 256), 256, 0, cudaStream_t(stream)>>>(
      stream_key(seed, kStreamTheta0), P, theta0);
  return launched();
}

int gem_synth_grad_heavytail(uint64_t seed, uint64_t first_row, int rows, size_t P, size_t ld,
                             float* out, void* stream) {
  if (!out || rows < 0 || ld < P || P > 0xFFFFFFFFull) return -1;
  if (rows == 0 || P == 0) return 0;
  heavytail_kernel<<<grid_for(size_t(rows) * P, 256), 256, 0, cudaStream_t(stream)>>>(
      stream_key(seed, kStreamGradZ), stream_key(seed, kStreamGradT),
      stream_key(seed, kStreamMask), first_row, rows, P, ld, out);
  return launched();
}

int gem_synth_grad_loguniform(uint64_t seed, uint64_t t, size_t P, const float* sigma,
                              float* out, void* stream) {
  if (!out || !sigma || P > 0xFFFFFFFFull) return -1;
  if (P == 0) return 0;
  loguniform_kernel<<<grid_for(P, 256), 256, 0, cudaStream_t(stream)>>>(
      stream_key(seed, kStreamGradZ), t, P, sigma, out);
  return launched();
}

int gem_synth_data(uint64_t seed, int rows, int d_in, int classes, float* X, int32_t* labels,
                   void* stream) {
  if (!X || !labels || rows < 0 || d_in < 1 || classes < 1 || classes > 16) return -1;
  if (rows == 0) return 0;
  data_kernel<<<grid_for(size_t(rows), 128), 128, 0, cudaStream_t(stream)>>>(
      stream_key(seed, kStreamDataX), stream_key(seed, kStreamTeacher), rows, d_in, classes,
      X, labels);
  return launched();
}

int gem_synth_xavier(uint64_t seed, const int32_t* dims, int n_layers, float* theta,
                     void* stream) {
  if (!dims || !theta || n_layers < 1) return -1;
  size_t off = 0;
  for (int l = 0; l < n_layers; ++l) {
    const int fi = dims[l], fo = dims[l + 1];
    if (fi < 1 || fo < 1) return -1;
    const size_t count = size_t(fo) * size_t(fi);
    const float a = float(sqrt(6.0 / double(fi + fo)));
    xavier_kernel<<<grid_for(count, 256), 256, 0, cudaStream_t(stream)>>>(
        stream_key(seed, kStreamXavier + 256ull * uint64_t(l)), count, fi, a, theta + off);
    if (cudaMemsetAsync(theta + off + count, 0, size_t(fo) * sizeof(float),
                        cudaStream_t(stream)) != cudaSuccess)
      return -3;
    off += count + size_t(fo);
  }
  return launched();
}

int gem_synth_cnn_theta0(uint64_t seed, const int32_t* shape, float* theta, void* stream) {
  if (!shape || !theta) return -1;
  const int H = shape[0], c1 = shape[1], c2 = shape[2], f1 = shape[3], f2 = shape[4],
            C = shape[5];
  if (H < 5 || c1 < 1 || c2 < 1 || f1 < 1 || f2 < 1 || C < 2 || (H - 4) % 2) return -1;
  const int h2 = (H - 4) / 2 - 4;
  if (h2 < 2 || h2 % 2) return -1;
  const long long feat = (long long)c2 * (h2 / 2) * (h2 / 2);
  const long long count[10] = {c1 * 25LL, c1, (long long)c2 * c1 * 25, c2, f1 * feat, f1,
                               (long long)f2 * f1, f2, (long long)C * f2, C};
  const long long fan_in[10] = {25, 25, c1 * 25LL, c1 * 25LL, feat, feat, f1, f1, f2, f2};
  size_t off = 0;
  for (int t = 0; t < 10; ++t) {
    const float bound = float(1.0 / sqrt(double(fan_in[t])));
    xavier_kernel<<<grid_for(size_t(count[t]), 256), 256, 0, cudaStream_t(stream)>>>(
        stream_key(seed, kStreamCnnInit + 256ull * uint64_t(t)), size_t(count[t]), 0, bound,
        theta + off);
    off += size_t(count[t]);
  }
  return launched();
}

int gem_synth_cnn_data(uint64_t seed, int rows, int H, int classes, float* X, int32_t* labels,
                       void* stream) {
  if (!X || !labels || rows < 0 || H < 1 || classes < 1) return -1;
  if (rows == 0) return 0;
  cnn_data_kernel<<<grid_for(size_t(rows), 1), 256, 0, cudaStream_t(stream)>>>(
      stream_key(seed, kStreamDataX), stream_key(seed, kStreamCnnTemplate),
      stream_key(seed, kStreamCnnLabel), rows, H, classes, X, labels);
  return launched();
}

int gem_synth_dropout(uint64_t seed, uint64_t t0, int T, int b, int channels, float p,
                      float* out, void* stream) {
  if (!out || T < 0 || b < 1 || channels < 1 || !(p >= 0.0f && p < 1.0f)) return -1;
  const size_t count = size_t(T) * size_t(b) * size_t(channels);
  if (count == 0) return 0;
  const float keep = float(1.0 / (1.0 - double(p)));
  dropout_kernel<<<grid_for(count, 256), 256, 0, cudaStream_t(stream)>>>(
      stream_key(seed, kStreamDropout), t0 * uint64_t(b) * uint64_t(channels), count, p, keep,
      out);
  return launched();
}

}  // extern "C"
