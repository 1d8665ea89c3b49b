"""Binding of the device input generators (include/gem_synth.h): the same inputs as the
host module ``synth``, produced on the GPU where they are too large to draw on the host
(a 10 GB gradient pool, a 60,000 x 784 data set)."""
from __future__ import annotations

import ctypes as C

from ._lib import lib


def _stream(stream) -> C.c_void_p:
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream if isinstance(stream, int) else int(stream.cuda_stream))


def _check(rc: int, where: str):
    if rc != 0:
        raise RuntimeError(f"{where} failed ({rc})")


def theta0_flat(seed: int, out, stream=None):
    _check(lib().gem_synth_theta0(seed, out.numel(), C.c_void_p(out.data_ptr()), _stream(stream)),
           "gem_synth_theta0")
    return out


def grad_heavytail(seed: int, first_row: int, out, P: int, stream=None):
    """Rows first_row.. of the heavy-tailed pool into out [rows, ld] (ld >= P)."""
    rows, ld = out.shape
    _check(lib().gem_synth_grad_heavytail(seed, first_row, rows, P, ld, C.c_void_p(out.data_ptr()),
                                          _stream(stream)), "gem_synth_grad_heavytail")
    return out


def grad_loguniform(seed: int, t: int, sigma, out, stream=None):
    _check(lib().gem_synth_grad_loguniform(seed, t, out.numel(), C.c_void_p(sigma.data_ptr()),
                                           C.c_void_p(out.data_ptr()), _stream(stream)),
           "gem_synth_grad_loguniform")
    return out


def data(seed: int, X, labels, classes: int, stream=None):
    rows, d_in = X.shape
    _check(lib().gem_synth_data(seed, rows, d_in, classes, C.c_void_p(X.data_ptr()),
                                C.c_void_p(labels.data_ptr()), _stream(stream)), "gem_synth_data")
    return X, labels


def xavier(seed: int, dims, theta, stream=None):
    d = (C.c_int32 * len(dims))(*dims)
    _check(lib().gem_synth_xavier(seed, d, len(dims) - 1, C.c_void_p(theta.data_ptr()),
                                  _stream(stream)), "gem_synth_xavier")
    return theta


def cnn_theta0(seed: int, shape, theta, stream=None):
    sh = (C.c_int32 * 6)(*shape)
    _check(lib().gem_synth_cnn_theta0(seed, sh, C.c_void_p(theta.data_ptr()), _stream(stream)),
           "gem_synth_cnn_theta0")
    return theta


def dropout(seed: int, t0: int, out, p: float = 0.5, stream=None):
    """out: float32 CUDA tensor [T, b, channels]."""
    T, b, ch = out.shape
    _check(lib().gem_synth_dropout(seed, t0, T, b, ch, p, C.c_void_p(out.data_ptr()),
                                   _stream(stream)), "gem_synth_dropout")
    return out


def cnn_data(seed: int, X, labels, classes: int = 10, stream=None):
    """X: float32 CUDA tensor [rows, H * H]; labels: int32 CUDA tensor [rows]."""
    rows, HH = X.shape
    H = int(round(HH ** 0.5))
    _check(lib().gem_synth_cnn_data(seed, rows, H, classes, C.c_void_p(X.data_ptr()),
                                    C.c_void_p(labels.data_ptr()), _stream(stream)), "gem_synth_cnn_data")
    return X, labels
