"""Python binding of the convolutional-network ABI (include/gem_cnn.h).

Argument marshalling only: the network's forward and backward passes and the commits run
in the CUDA library.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from ._lib import check, lib

# The network of the paper's MNIST experiments: {H, c1, c2, f1, f2, C}.
CNN_MNIST = (28, 10, 20, 128, 64, 10)


def _shape(shape):
    return (C.c_int32 * 6)(*[int(x) for x in shape])


def _p(a: np.ndarray):
    return a.ctypes.data_as(C.c_void_p)


def _opt_ptr(t):
    return C.c_void_p(0 if t is None else t.data_ptr())


def gem_cnn_param_count(shape) -> int:
    return int(lib().gem_cnn_param_count(_shape(shape)))


def gem_cnn_create(h: int, shape, batch: int) -> int:
    out = C.c_void_p()
    check(lib().gem_cnn_create(C.c_void_p(h), _shape(shape), int(batch), C.byref(out)), "gem_cnn_create")
    return int(out.value)


def gem_cnn_set_data(net: int, X, labels) -> None:
    check(lib().gem_cnn_set_data(C.c_void_p(net), C.c_void_p(X.data_ptr()),
                                 C.c_void_p(labels.data_ptr()), int(X.shape[0])), "gem_cnn_set_data")


def gem_cnn_grad(net: int, workers, batch_rows, drop, grads, losses=None) -> None:
    """workers [L]; batch_rows host int array [L, b]; drop CUDA tensor [L, b, c2];
    grads: L float32 CUDA tensors of P values."""
    w = np.ascontiguousarray(workers, dtype=np.int32)
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    if r.shape[0] != w.shape[0] or len(grads) != w.shape[0]:
        raise ValueError("workers, batch_rows and grads differ in length")
    g = (C.c_void_p * max(len(grads), 1))(*[x.data_ptr() for x in grads])
    check(lib().gem_cnn_grad(C.c_void_p(net), _p(w), len(w), _p(r), C.c_void_p(drop.data_ptr()), g,
                             _opt_ptr(losses)), "gem_cnn_grad")


def gem_cnn_run(net: int, order, batch_rows, drop, losses=None) -> None:
    """order [T]; batch_rows host int array [T, b]; drop CUDA tensor [T, b, c2]."""
    o = np.ascontiguousarray(order, dtype=np.int32)
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    if r.shape[0] != o.shape[0]:
        raise ValueError("batch_rows must have one row per commit")
    check(lib().gem_cnn_run(C.c_void_p(net), _p(o), len(o), _p(r), C.c_void_p(drop.data_ptr()),
                            _opt_ptr(losses)), "gem_cnn_run")


def gem_cnn_run_pi(net: int, order, batch_rows, drop, pi_lo, pi_hi, losses=None) -> None:
    """gem_cnn_run with each commit's per-tensor factor medians in pi_lo, pi_hi (float32
    CUDA tensors [T, 10])."""
    o = np.ascontiguousarray(order, dtype=np.int32)
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    if r.shape[0] != o.shape[0]:
        raise ValueError("batch_rows must have one row per commit")
    check(lib().gem_cnn_run_pi(C.c_void_p(net), _p(o), len(o), _p(r), C.c_void_p(drop.data_ptr()),
                               _opt_ptr(losses), _opt_ptr(pi_lo), _opt_ptr(pi_hi)), "gem_cnn_run_pi")


def gem_cnn_status(net: int) -> None:
    check(lib().gem_cnn_status(C.c_void_p(net)), "gem_cnn_status")


def gem_cnn_launch_count(net: int) -> int:
    return int(lib().gem_cnn_launch_count(C.c_void_p(net)))


def gem_cnn_destroy(net: int) -> None:
    lib().gem_cnn_destroy(C.c_void_p(net))
