"""Seeded synthetic inputs for GEM workloads (host side, numpy).

This module only *draws numbers*: parameter initialisations, synthetic gradients, an
MNIST-shaped synthetic data set with teacher labels, and per-commit minibatch indices.
It holds none of GEM's arithmetic (no update, moment, energy or scaling factor), so both
the CUDA path (through its device twin of these generators) and the oracle may consume
what it produces.

Every value is a pure function of (seed, stream, counter), built on the SplitMix64
generator of Steele, Lea and Flood ("Fast splittable pseudorandom number generators",
OOPSLA 2014): the c-th output (0-based) of the stream whose state starts at `key` is
``mix64(key + GAMMA * (c + 1))``.  Floating-point values are formed with integer
operations, exact int->float conversions and single IEEE fp32 operations, so a device
implementation that follows the same definitions produces the same bits.

Definitions (shared by the device twin in ``csrc/synth.cu``):

* ``key(seed, stream) = mix64(seed * GAMMA + stream)``
* ``normal(key, c)``: Irwin-Hall sum of twelve 20-bit uniforms taken from the draws at
  counters 4c..4c+3 (bits 4..23, 24..43, 44..63 of each), recentred by 6 * 2**20 and
  scaled by 2**-20.  The result is exact in fp32, mean 0 and variance 1 (up to the 20-bit
  discretisation); its support is [-6, 6).
* ``student_t3(key, c) = z0 / sqrt(((z1*z1 + z2*z2) + z3*z3) / 3)`` with
  ``z_r = normal(key, 4c + r)``; fp32, one rounding per operation; 0 when the
  denominator is 0.
* ``u24(h) = (h >> 40) * 2**-24`` and ``u53(h) = (h >> 11) * 2**-53``.
"""
from __future__ import annotations

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

# stream identifiers (one independent stream per kind of input)
STREAM_THETA0 = 1
STREAM_GRAD_Z = 2
STREAM_GRAD_T = 3
STREAM_GRAD_MASK = 4
STREAM_SIGMA = 5
STREAM_DATA_X = 6
STREAM_TEACHER = 7
STREAM_XAVIER = 8  # + 256 * layer
STREAM_BATCH = 9
STREAM_DROPOUT = 10
STREAM_CNN_INIT = 11  # + 256 * tensor
STREAM_CNN_TEMPLATE = 12
STREAM_CNN_LABEL = 13

# workload constants
THETA0_SCALE = np.float32(0.05)
FLAT_GRAD_SCALE = np.float32(0.01)          # std 0.01, i.e. variance 1e-4
HEAVY_TAIL_THRESHOLD_U24 = 1677722          # ceil(0.1 * 2**24): 10% of coordinates
DATA_ROWS = 60000                           # MNIST-shaped training-set stand-in
TWO_POW_M20 = np.float32(2.0 ** -20)

_U64 = np.uint64


def mix64(z):
    """SplitMix64 output function applied elementwise (uint64 in, uint64 out)."""
    z = np.asarray(z, dtype=_U64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> _U64(30))) * _U64(_M1)
        z = (z ^ (z >> _U64(27))) * _U64(_M2)
    return z ^ (z >> _U64(31))


def splitmix64_sequence(state: int, count: int) -> list[int]:
    """The first `count` outputs of the classic sequential SplitMix64 seeded with `state`."""
    out = []
    for _ in range(count):
        state = (state + GAMMA) & MASK64
        out.append(int(mix64(_U64(state))))
    return out


def key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        return mix64(_U64(seed & MASK64) * _U64(GAMMA) + _U64(stream))


def draw(k, counter):
    """counter-th output of the stream with initial state k (vectorised over counter)."""
    c = np.asarray(counter, dtype=_U64)
    with np.errstate(over="ignore"):
        return mix64(_U64(k) + _U64(GAMMA) * (c + _U64(1)))


def u24(h):
    return ((np.asarray(h, dtype=_U64) >> _U64(40)).astype(np.float32)
            * np.float32(2.0 ** -24))


def u53(h):
    return (np.asarray(h, dtype=_U64) >> _U64(11)).astype(np.float64) * (2.0 ** -53)


def normal_int(k, counter):
    """Integer part a of normal(k, c) = a * 2**-20 (int64), vectorised over counter."""
    c4 = np.asarray(counter, dtype=_U64) * _U64(4)
    acc = np.zeros(c4.shape, dtype=np.int64)
    f = _U64(0xFFFFF)
    for r in range(4):
        h = draw(k, c4 + _U64(r))
        acc += (((h >> _U64(4)) & f) + ((h >> _U64(24)) & f) + ((h >> _U64(44)) & f)).astype(np.int64)
    return acc - np.int64(6 << 20)


def normal(k, counter):
    """Irwin-Hall N(0,1) stand-in, exact fp32 (vectorised over counter)."""
    return normal_int(k, counter).astype(np.float32) * TWO_POW_M20


def student_t3(k, counter):
    """Student-t with 3 degrees of freedom from four normals, fp32 one rounding per op."""
    c4 = np.asarray(counter, dtype=_U64) * _U64(4)
    z0 = normal(k, c4)
    z1 = normal(k, c4 + _U64(1))
    z2 = normal(k, c4 + _U64(2))
    z3 = normal(k, c4 + _U64(3))
    q = (z1 * z1 + z2 * z2) + z3 * z3
    q = q / np.float32(3.0)
    den = np.sqrt(q)
    with np.errstate(divide="ignore", invalid="ignore"):
        t = z0 / den
    return np.where(q == np.float32(0.0), np.float32(0.0), t).astype(np.float32)


def _cols(j):
    return np.asarray(j, dtype=_U64)


# ---------------------------------------------------------------- flat workloads

def theta0_flat(seed: int, j) -> np.ndarray:
    """Initial central variable of the flat workloads: 0.05 * normal, fp32."""
    return (THETA0_SCALE * normal(key(seed, STREAM_THETA0), _cols(j))).astype(np.float32)


def sigma_loguniform(seed: int, j) -> np.ndarray:
    """Per-coordinate gradient scale sigma_j = 10**(-4 + 3u), log-uniform in [1e-4, 1e-1].

    Computed in float64 on the host and rounded to fp32; the device receives this array.
    """
    u = u53(draw(key(seed, STREAM_SIGMA), _cols(j)))
    return np.power(10.0, -4.0 + 3.0 * u).astype(np.float32)


def grad_loguniform(seed: int, t: int, j, sigma: np.ndarray) -> np.ndarray:
    """Gradient of commit t at coordinates j: sigma_j * normal, fp32 (one rounding)."""
    c = (_U64(t) << _U64(32)) | _cols(j)
    return (sigma * normal(key(seed, STREAM_GRAD_Z), c)).astype(np.float32)


def heavy_mask(seed: int, j) -> np.ndarray:
    """Fixed 10% coordinate mask of the heavy-tailed gradient workload."""
    h = draw(key(seed, STREAM_GRAD_MASK), _cols(j))
    return (h >> _U64(40)) < _U64(HEAVY_TAIL_THRESHOLD_U24)


def grad_heavytail(seed: int, i: int, j) -> np.ndarray:
    """Pool gradient i at coordinates j: 0.01 * (normal, or Student-t(3) on the mask)."""
    j = _cols(j)
    c = (_U64(i) << _U64(32)) | j
    mask = heavy_mask(seed, j)
    v = np.empty(j.shape, dtype=np.float32)
    v[~mask] = normal(key(seed, STREAM_GRAD_Z), c[~mask])
    v[mask] = student_t3(key(seed, STREAM_GRAD_T), c[mask])
    return (FLAT_GRAD_SCALE * v).astype(np.float32)


# ---------------------------------------------------------------- MLP workloads

def mlp_param_count(dims) -> int:
    return sum(dims[l + 1] * dims[l] + dims[l + 1] for l in range(len(dims) - 1))


def mlp_layout(dims):
    """Flat parameter layout [W1 (out x in, row-major), b1, W2, b2, ...]: list of
    (w_offset, b_offset, out, in)."""
    off = 0
    lay = []
    for l in range(len(dims) - 1):
        fi, fo = dims[l], dims[l + 1]
        lay.append((off, off + fo * fi, fo, fi))
        off += fo * fi + fo
    return lay


def xavier_theta0(seed: int, dims) -> np.ndarray:
    """Xavier-uniform weights a * (2u - 1), a = sqrt(6 / (fan_in + fan_out)); biases 0."""
    theta = np.zeros(mlp_param_count(dims), dtype=np.float32)
    for l, (wo, _bo, fo, fi) in enumerate(mlp_layout(dims)):
        a = np.float32(np.sqrt(6.0 / (fi + fo)))
        u = u24(draw(key(seed, STREAM_XAVIER + 256 * l), np.arange(fo * fi, dtype=np.uint64)))
        theta[wo:wo + fo * fi] = a * (np.float32(2.0) * u - np.float32(1.0))
    return theta


def data_rows_int(seed: int, rows, d_in: int) -> np.ndarray:
    """Integer numerators a of the synthetic inputs x = a * 2**-20, shape [len(rows), d_in]."""
    rows = np.asarray(rows, dtype=np.uint64)
    c = rows[:, None] * _U64(d_in) + np.arange(d_in, dtype=np.uint64)[None, :]
    return normal_int(key(seed, STREAM_DATA_X), c)


def data_rows(seed: int, rows, d_in: int) -> np.ndarray:
    """Synthetic N(0,1) inputs x for the given training-set rows, fp32 [len(rows), d_in]."""
    return data_rows_int(seed, rows, d_in).astype(np.float32) * TWO_POW_M20


def teacher_int(seed: int, d_in: int, classes: int) -> np.ndarray:
    c = np.arange(d_in * classes, dtype=np.uint64)
    return normal_int(key(seed, STREAM_TEACHER), c).reshape(d_in, classes)


def teacher_labels(seed: int, rows, d_in: int, classes: int) -> np.ndarray:
    """Labels argmax_c x . T[:, c] of a fixed random linear teacher, ties to the lowest c.

    x and T are both integers times 2**-20, so the dot products are evaluated exactly in
    int64 and the argmax is independent of summation order.
    """
    xa = data_rows_int(seed, rows, d_in)
    ta = teacher_int(seed, d_in, classes)
    scores = xa @ ta                       # exact: |sum| < 784 * 2**46 < 2**63
    return np.argmax(scores, axis=1).astype(np.int32)


def batch_indices(seed: int, worker: int, k: int, b: int, n_rows: int = DATA_ROWS) -> np.ndarray:
    """Rows of worker `worker`'s k-th minibatch: b draws with replacement (uint32 multiply-shift)."""
    i = np.arange(b, dtype=np.uint64)
    c = (_U64(worker) << _U64(40)) | (_U64(k) << _U64(16)) | i
    h = draw(key(seed, STREAM_BATCH), c) >> _U64(32)
    return ((h * _U64(n_rows)) >> _U64(32)).astype(np.int32)


def schedule_batches(seed: int, order, b: int, n_rows: int = DATA_ROWS) -> np.ndarray:
    """Minibatch rows for every commit of a schedule: commit t by worker w uses w's k-th
    batch, k = number of earlier commits by w.  Shape [T, b] int32."""
    order = np.asarray(order)
    seen: dict[int, int] = {}
    out = np.empty((len(order), b), dtype=np.int32)
    for t, w in enumerate(order.tolist()):
        k = seen.get(w, 0)
        seen[w] = k + 1
        out[t] = batch_indices(seed, w, k, b, n_rows)
    return out


# ------------------------------------------------------------- the MNIST network

# The convolutional network of the MNIST experiments (Appendix A): 28 x 28 inputs, conv 5x5
# to 10 channels, conv 5x5 to 20 channels, fully connected 320 -> 128 -> 64 -> 10.
CNN_MNIST = (28, 10, 20, 128, 64, 10)


def cnn_layout(shape):
    """[(name, offset, count, fan_in)] of the flat parameter vector: conv1.W, conv1.b,
    conv2.W, conv2.b, fc1.W, fc1.b, fc2.W, fc2.b, fc3.W, fc3.b."""
    H, c1, c2, f1, f2, C = shape
    p2 = ((H - 4) // 2 - 4) // 2
    feat = c2 * p2 * p2
    tensors = [("conv1.W", c1 * 25, 25), ("conv1.b", c1, 25),
               ("conv2.W", c2 * c1 * 25, c1 * 25), ("conv2.b", c2, c1 * 25),
               ("fc1.W", f1 * feat, feat), ("fc1.b", f1, feat),
               ("fc2.W", f2 * f1, f1), ("fc2.b", f2, f1),
               ("fc3.W", C * f2, f2), ("fc3.b", C, f2)]
    out, off = [], 0
    for name, count, fan_in in tensors:
        out.append((name, off, count, fan_in))
        off += count
    return out


def cnn_param_count(shape) -> int:
    name, off, count, _f = cnn_layout(shape)[-1]
    return off + count


def cnn_init_bound(fan_in: int) -> np.float32:
    return np.float32(1.0 / np.sqrt(float(fan_in)))


def cnn_theta0(seed: int, shape) -> np.ndarray:
    """PyTorch's default initialisation of the network: every weight and bias uniform in
    [-1/sqrt(fan_in), 1/sqrt(fan_in)), as bound * (2u - 1) with a 24-bit u, fp32."""
    theta = np.empty(cnn_param_count(shape), dtype=np.float32)
    for t, (_name, off, count, fan_in) in enumerate(cnn_layout(shape)):
        u = u24(draw(key(seed, STREAM_CNN_INIT + 256 * t), np.arange(count, dtype=np.uint64)))
        theta[off:off + count] = cnn_init_bound(fan_in) * (np.float32(2.0) * u - np.float32(1.0))
    return theta


def dropout_scales(seed: int, t0: int, T: int, b: int, channels: int, p: float = 0.5) -> np.ndarray:
    """Channel dropout of commits t0 .. t0 + T - 1: scale [T, b, channels] is 0 where the
    24-bit uniform of counter ((t b + i) channels + c) is below p, else 1 / (1 - p) (fp32)."""
    c = ((np.arange(t0, t0 + T, dtype=np.uint64)[:, None, None] * _U64(b)
          + np.arange(b, dtype=np.uint64)[None, :, None]) * _U64(channels)
         + np.arange(channels, dtype=np.uint64)[None, None, :])
    u = u24(draw(key(seed, STREAM_DROPOUT), c))
    keep = np.float32(1.0 / (1.0 - p))
    return np.where(u < np.float32(p), np.float32(0.0), keep).astype(np.float32)


CNN_TEMPLATE_BLOCK = 4       # template cells of 4 x 4 pixels
CNN_TEMPLATE_AMPLITUDE = 0.5


def cnn_labels(seed: int, rows, classes: int = 10) -> np.ndarray:
    """Uniform class of each training row (multiply-shift of a 32-bit draw)."""
    h = draw(key(seed, STREAM_CNN_LABEL), np.asarray(rows, dtype=np.uint64)) >> _U64(32)
    return ((h * _U64(classes)) >> _U64(32)).astype(np.int32)


def cnn_templates(seed: int, H: int = 28, classes: int = 10) -> np.ndarray:
    """Class templates [classes, H * H]: +-0.5 on cells of 4 x 4 pixels, the sign of cell
    (c, row, col) from the top bit of draw(key(seed, 12), (c * cells + row) * cells + col)."""
    cells = (H + CNN_TEMPLATE_BLOCK - 1) // CNN_TEMPLATE_BLOCK
    idx = np.arange(classes * cells * cells, dtype=np.uint64)
    sign = np.where((draw(key(seed, STREAM_CNN_TEMPLATE), idx) >> _U64(63)) == 1, -1.0, 1.0)
    sign = sign.reshape(classes, cells, cells).astype(np.float32)
    py = np.arange(H) // CNN_TEMPLATE_BLOCK
    t = sign[:, py[:, None], py[None, :]] * np.float32(CNN_TEMPLATE_AMPLITUDE)
    return t.reshape(classes, H * H).astype(np.float32)


def cnn_data_rows(seed: int, rows, H: int = 28, classes: int = 10):
    """MNIST-shaped stand-in with spatial class structure: image = template of its class +
    N(0, 1) pixel noise (the noise of data_rows), exact in fp32.  Returns (X [len, H*H],
    labels [len])."""
    y = cnn_labels(seed, rows, classes)
    X = cnn_templates(seed, H, classes)[y] + data_rows(seed, rows, H * H)
    return X.astype(np.float32), y
