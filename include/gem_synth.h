/* gem_synth.h -- seeded synthetic inputs on the device (not part of GEM itself).
 *
 * Device generators for the synthetic workloads that exercise the GEM commit path:
 * initial parameters, gradient pools, an MNIST-shaped data set with teacher labels and
 * Xavier-initialised MLP parameters.  Each value is a pure function of
 * (seed, stream, counter) built on SplitMix64 (Steele, Lea & Flood, OOPSLA 2014), and
 * follows the definitions of the host generator module paper_1805_08469_gb300/synth.py
 * bit for bit:
 *   key(seed, stream) = mix64(seed * GAMMA + stream)
 *   draw(key, c)      = mix64(key + GAMMA * (c + 1))
 *   normal(key, c)    = (sum of twelve 20-bit fields of draws 4c..4c+3 - 6 * 2^20) * 2^-20
 *   student_t3(key,c) = z0 / sqrt(((z1 z1 + z2 z2) + z3 z3) / 3), z_r = normal(key, 4c + r)
 * The paper prints no data of its own here: these stand in for its MNIST / ImageNet
 * workloads (experiments section) with the shapes the benchmarks use.
 *
 * All calls are asynchronous on `stream` (a cudaStream_t, NULL = legacy default stream),
 * write only their output buffers, and return 0, or -1 on an invalid argument, or -3
 * if the launch failed.
 */
#ifndef GEM_SYNTH_H
#define GEM_SYNTH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* theta0[j] = 0.05 * normal(key(seed, 1), j), j < P. */
int gem_synth_theta0(uint64_t seed, size_t P, float* theta0, void* stream);

/* Rows first_row .. first_row + rows - 1 of the heavy-tailed gradient pool, row r at
 * out + (r - first_row) * ld: g[r][j] = 0.01 * (student_t3(key(seed, 3), (r << 32) | j)
 * on the fixed 10% mask draw(key(seed, 4), j) >> 40 < 1677722, else
 * normal(key(seed, 2), (r << 32) | j)).  Requires ld >= P. */
int gem_synth_grad_heavytail(uint64_t seed, uint64_t first_row, int rows, size_t P,
                             size_t ld, float* out, void* stream);

/* Gradient of commit t: g[j] = sigma[j] * normal(key(seed, 2), (t << 32) | j). */
int gem_synth_grad_loguniform(uint64_t seed, uint64_t t, size_t P, const float* sigma,
                              float* out, void* stream);

/* Synthetic inputs X [rows][d_in], X[r][k] = normal(key(seed, 6), r d_in + k), and labels
 * [rows] = argmax_c sum_k X[r][k] T[k][c] with T[k][c] = normal(key(seed, 7), k C + c),
 * evaluated exactly on the integer numerators (ties to the lowest class).  classes <= 16. */
int gem_synth_data(uint64_t seed, int rows, int d_in, int classes, float* X, int32_t* labels,
                   void* stream);

/* Xavier-uniform MLP parameters in the flat layout [W_1 (out x in), b_1, W_2, b_2, ...]:
 * W_l = a_l (2u - 1), a_l = sqrt(6 / (in + out)), u = (draw(key(seed, 8 + 256 l), o in + i)
 * >> 40) 2^-24; biases 0.  dims has n_layers + 1 entries. */
int gem_synth_xavier(uint64_t seed, const int32_t* dims, int n_layers, float* theta,
                     void* stream);

/* Parameters of the MNIST convolutional network (gem_cnn.h) with shape {H, c1, c2, f1, f2,
 * C}, PyTorch's default initialisation: tensor t of the flat layout (conv1.W, conv1.b,
 * conv2.W, conv2.b, fc1.W, fc1.b, fc2.W, fc2.b, fc3.W, fc3.b) holds bound_t (2u - 1),
 * bound_t = 1 / sqrt(fan_in_t) rounded to fp32, u = (draw(key(seed, 11 + 256 t), q) >> 40)
 * 2^-24. */
int gem_synth_cnn_theta0(uint64_t seed, const int32_t* shape, float* theta, void* stream);

/* Training set of the network with spatial class structure: labels [rows], y_r =
 * ((draw(key(seed, 13), r) >> 32) classes) >> 32; X [rows][H * H], pixel p of row r =
 * template(y_r, p) + normal(key(seed, 6), r H H + p), template +-0.5 constant on cells of
 * 4 x 4 pixels, the sign of cell (c, row, col) the top bit of draw(key(seed, 12),
 * (c cells + row) cells + col), cells = ceil(H / 4).  Exact in fp32. */
int gem_synth_cnn_data(uint64_t seed, int rows, int H, int classes, float* X, int32_t* labels,
                       void* stream);

/* Channel-dropout scales of commits t0 .. t0 + T - 1: out [T][b][channels], entry
 * ((t - t0) b + i) channels + c is 0 when (draw(key(seed, 10), (t b + i) channels + c) >> 40)
 * 2^-24 < p, else 1 / (1 - p) rounded to fp32.  0 <= p < 1. */
int gem_synth_dropout(uint64_t seed, uint64_t t0, int T, int b, int channels, float p,
                      float* out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* GEM_SYNTH_H */
