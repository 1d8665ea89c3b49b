"""Binding of the simulator calls (include/gem_sim.h): seeded commit schedules and the
segment planner.  Argument marshalling only."""
from __future__ import annotations

import ctypes as C

import numpy as np

from ._lib import lib


def _p(a):
    return a.ctypes.data_as(C.c_void_p)


def gem_schedule_uniform(seed: int, n: int, T: int):
    order = np.empty(T, np.int32)
    tau = np.empty(T, np.int32)
    if lib().gem_schedule_uniform(seed, n, T, _p(order), _p(tau)) != 0:
        raise ValueError("gem_schedule_uniform: invalid argument")
    return order, tau


def gem_schedule_queue(seed: int, n: int, T: int, rate: float = 1.0):
    order = np.empty(T, np.int32)
    tau = np.empty(T, np.int32)
    if lib().gem_schedule_queue(seed, n, T, rate, _p(order), _p(tau)) != 0:
        raise ValueError("gem_schedule_queue: invalid argument")
    return order, tau


def gem_plan_segments(order, n: int) -> np.ndarray:
    order = np.ascontiguousarray(order, dtype=np.int32)
    T = order.shape[0]
    seg = np.empty(T + 1, np.int32)
    S = lib().gem_plan_segments(_p(order), T, n, _p(seg))
    if S < 0:
        raise ValueError("gem_plan_segments: invalid argument")
    return seg[:S + 1].copy()


GEM_MLP_FP32 = 0
GEM_MLP_TF32 = 1


def gem_mlp_create(gem_handle: int, dims, batch: int, precision: int = GEM_MLP_FP32) -> int:
    from ._lib import check
    d = (C.c_int32 * len(dims))(*[int(x) for x in dims])
    h = C.c_void_p()
    check(lib().gem_mlp_create(C.c_void_p(gem_handle), len(dims) - 1, d, batch, precision,
                               C.byref(h)), "gem_mlp_create")
    return int(h.value)


def gem_mlp_destroy(h: int) -> None:
    lib().gem_mlp_destroy(C.c_void_p(h))


def gem_mlp_set_data(h: int, X, labels) -> None:
    """X: float32 CUDA tensor [rows, d0]; labels: int32 CUDA tensor [rows] (borrowed)."""
    from ._lib import check
    check(lib().gem_mlp_set_data(C.c_void_p(h), C.c_void_p(X.data_ptr()),
                                 C.c_void_p(labels.data_ptr()), X.shape[0]), "gem_mlp_set_data")


def _opt_ptr(t):
    return C.c_void_p(0 if t is None else t.data_ptr())


def gem_mlp_grad(h: int, workers, batch_rows, grads, losses=None) -> None:
    """workers [L] ints; batch_rows host int array [L, b]; grads: L float32 CUDA tensors."""
    from ._lib import check
    w = np.ascontiguousarray(workers, dtype=np.int32)
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    g = (C.c_void_p * len(grads))(*[x.data_ptr() for x in grads])
    check(lib().gem_mlp_grad(C.c_void_p(h), _p(w), len(w), _p(r), g, _opt_ptr(losses)), "gem_mlp_grad")


def gem_mlp_run(h: int, order, batch_rows, losses=None) -> None:
    """order [T] ints; batch_rows host int array [T, b]; losses: float32 CUDA tensor [T] or None."""
    from ._lib import check
    o = np.ascontiguousarray(order, dtype=np.int32)
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    if r.shape[0] != o.shape[0]:
        raise ValueError("batch_rows must have one row per commit")
    check(lib().gem_mlp_run(C.c_void_p(h), _p(o), len(o), _p(r), _opt_ptr(losses)), "gem_mlp_run")


def gem_mlp_run_pi(h: int, order, batch_rows, pi_lo, pi_hi, losses=None) -> None:
    """gem_mlp_run that also writes each commit's per-tensor factor medians to pi_lo and
    pi_hi (float32 CUDA tensors [T, 2 * n_layers])."""
    from ._lib import check
    o = np.ascontiguousarray(order, dtype=np.int32)
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    if r.shape[0] != o.shape[0]:
        raise ValueError("batch_rows must have one row per commit")
    check(lib().gem_mlp_run_pi(C.c_void_p(h), _p(o), len(o), _p(r), _opt_ptr(losses),
                               _opt_ptr(pi_lo), _opt_ptr(pi_hi)), "gem_mlp_run_pi")


def gem_mlp_status(h: int) -> None:
    """Waits for the MLP's work; raises if device work failed."""
    from ._lib import check
    check(lib().gem_mlp_status(C.c_void_p(h)), "gem_mlp_status")


def gem_mlp_launch_count(h: int) -> int:
    return int(lib().gem_mlp_launch_count(C.c_void_p(h)))


def gem_mlp_grad_static(dims, batch: int, precision: int, theta, X, labels, batch_rows, grad,
                        loss=None, stream=None) -> None:
    """Gradient without any allocation (include/gem_sim.h): theta [P], X [rows, d0], labels
    [rows], grad [P] (and loss [1]) are CUDA tensors; batch_rows a host int array [batch]."""
    from ._lib import check
    d = (C.c_int32 * len(dims))(*[int(x) for x in dims])
    r = np.ascontiguousarray(batch_rows, dtype=np.int32)
    if r.shape != (batch,):
        raise ValueError("batch_rows must hold `batch` row indices")
    st = 0 if stream is None else (stream if isinstance(stream, int) else int(stream.cuda_stream))
    check(lib().gem_mlp_grad_static(len(dims) - 1, d, batch, precision, C.c_void_p(theta.data_ptr()),
                                    C.c_void_p(X.data_ptr()), C.c_void_p(labels.data_ptr()), X.shape[0],
                                    _p(r), C.c_void_p(grad.data_ptr()), _opt_ptr(loss), C.c_void_p(st)),
          "gem_mlp_grad_static")
