"""ctypes wrapper of the oracle library (test infrastructure, not part of the product)."""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

from ._build import build_oracle

MODE_GEM = 0
MODE_DOWNPOUR = 1
MODE_ADAPTIVE = 2
MODE_KAPPA_SQRT = 3
MODE_KAPPA_LINEAR = 4
MODE_MOMENTUM = 5

_lib = None


def lib():
    global _lib
    if _lib is None:
        # ORACLE_LIBRARY: a library built from altered oracle sources, for the tests that
        # check that a planted mistake makes the oracle's pins fail
        _lib = C.CDLL(os.environ.get("ORACLE_LIBRARY") or str(build_oracle()))
        p = C.c_void_p
        i64, i32, f64 = C.c_int64, C.c_int, C.c_double
        run_args = [i64, i32, i32, p, p, p, i64, p, p, p, p, i64, f64, f64, f64, i32, f64,
                    i32, p, i32, p]
        for name in ("oracle_gem_run_f32", "oracle_gem_run_f64"):
            fn = getattr(_lib, name)
            fn.argtypes = run_args
            fn.restype = C.c_int
        for name in ("oracle_gem_run_pi_f32", "oracle_gem_run_pi_f64"):
            fn = getattr(_lib, name)
            fn.argtypes = run_args[:17] + [p]
            fn.restype = C.c_int
        _lib.oracle_splitmix64_raw.argtypes = [C.c_uint64, C.c_uint64]
        _lib.oracle_splitmix64_raw.restype = C.c_uint64
        _lib.oracle_splitmix64_draw.argtypes = [C.c_uint64, C.c_uint64, C.c_uint64]
        _lib.oracle_splitmix64_draw.restype = C.c_uint64
        _lib.oracle_schedule_uniform.argtypes = [C.c_uint64, i32, i32, p, p]
        _lib.oracle_schedule_uniform.restype = C.c_int
        _lib.oracle_schedule_queue.argtypes = [C.c_uint64, i32, i32, f64, p, p]
        _lib.oracle_schedule_queue.restype = C.c_int
        _lib.oracle_tf32_rna.argtypes = [C.c_float]
        _lib.oracle_tf32_rna.restype = C.c_float
        _lib.oracle_set_commit_threads.argtypes = [i32]
        _lib.oracle_set_commit_threads.restype = C.c_int
        _lib.oracle_threads.argtypes = []
        _lib.oracle_threads.restype = C.c_int
        _lib.oracle_mlp_loss_grad_f64.argtypes = [i32, p, p, p, p, i32, p, i32]
        _lib.oracle_mlp_loss_grad_f64.restype = C.c_double
        _lib.oracle_mlp_sim_run.argtypes = [i32, p, i32, i32, p, p, p, i64, p, p, i32, p, p,
                                            p, i64, f64, f64, f64, i32, f64, i32, i32, p, p, p]
        _lib.oracle_mlp_sim_run.restype = C.c_int
        _lib.oracle_mlp_sim_run_pi.argtypes = _lib.oracle_mlp_sim_run.argtypes + [p]
        _lib.oracle_mlp_sim_run_pi.restype = C.c_int
        _lib.oracle_cnn_param_count.argtypes = [p]
        _lib.oracle_cnn_param_count.restype = i64
        _lib.oracle_cnn_loss_grad_f64.argtypes = [p, p, p, p, p, i32, p, p]
        _lib.oracle_cnn_loss_grad_f64.restype = f64
        _lib.oracle_cnn_sim_run.argtypes = [p, i32, i32, p, p, p, i64, p, p, i32, p, p, p, p, i64,
                                            f64, f64, f64, i32, f64, i32, p, p, p]
        _lib.oracle_cnn_sim_run.restype = C.c_int
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _need(a, dtype, name):
    if not (isinstance(a, np.ndarray) and a.dtype == dtype and a.flags.c_contiguous):
        raise TypeError(f"{name} must be a C-contiguous {np.dtype(dtype).name} array")
    return a


def gem_run(theta, m, s, grads, order, *, eta, mu, eps, grad_index=None, tau=None,
            mode=MODE_GEM, kappa=1.0, precommit_snapshot=False, record_cols=None,
            record_pi=False):
    """Apply len(order) commits in place (fp32 or fp64 state, chosen by theta's dtype).

    theta [P]; m, s [n, P]; grads [R, P] (row grad_index[t], or row t); returns the
    [T, len(record_cols)] trajectory of theta at record_cols when asked for, or with
    record_pi the [T, P] scaling factors pi that the commits applied.
    """
    if record_pi and record_cols is not None:
        raise ValueError("record_pi and record_cols are separate runs")
    dt = theta.dtype
    if dt not in (np.float32, np.float64):
        raise TypeError("theta must be float32 or float64")
    fn = lib().oracle_gem_run_f32 if dt == np.float32 else lib().oracle_gem_run_f64
    _need(theta, dt, "theta"), _need(m, dt, "m"), _need(s, dt, "s"), _need(grads, dt, "grads")
    P = theta.shape[0]
    n = m.shape[0]
    if m.shape != (n, P) or s.shape != (n, P) or grads.ndim != 2 or grads.shape[1] != P:
        raise ValueError("shape mismatch")
    order = np.ascontiguousarray(order, dtype=np.int32)
    T = order.shape[0]
    gi = None if grad_index is None else np.ascontiguousarray(grad_index, dtype=np.int32)
    rows = grads.shape[0]
    if (gi is None and rows < T) or (gi is not None and (gi.min(initial=0) < 0 or gi.max(initial=0) >= rows)):
        raise ValueError("gradient rows out of range")
    tau_a = None if tau is None else np.ascontiguousarray(tau, dtype=np.int32)
    rec = None
    rc_cols = None
    nrec = 0
    if record_cols is not None:
        rc_cols = np.ascontiguousarray(record_cols, dtype=np.int64)
        nrec = rc_cols.shape[0]
        rec = np.empty((T, nrec), dtype=dt)
    if record_pi:
        fn = lib().oracle_gem_run_pi_f32 if dt == np.float32 else lib().oracle_gem_run_pi_f64
        pi = np.empty((T, P), dtype=dt)
        rc = fn(P, n, T, _ptr(order), _ptr(tau_a), _ptr(grads), P, _ptr(gi), _ptr(theta), _ptr(m),
                _ptr(s), P, eta, mu, eps, mode, kappa, int(precommit_snapshot), _ptr(pi))
        if rc:
            raise ValueError(f"oracle_gem_run_pi failed ({rc})")
        return pi
    rc = fn(P, n, T, _ptr(order), _ptr(tau_a), _ptr(grads), P, _ptr(gi), _ptr(theta), _ptr(m),
            _ptr(s), P, eta, mu, eps, mode, kappa, int(precommit_snapshot), _ptr(rc_cols), nrec,
            _ptr(rec))
    if rc:
        raise ValueError(f"oracle_gem_run failed ({rc})")
    return rec


def pi_median(pi, seg):
    """Per-segment lower and upper medians of the scaling factors of one commit (the median
    per-parameter pi of the experiments section, per tensor when the segments are the
    tensors of the flat layout).

    pi [P]; seg [nseg + 1] increasing offsets into pi.  Segment i is pi[seg[i]:seg[i+1]]
    with N elements, sorted ascending; its lower median is element (N - 1) // 2 and its
    upper median element N // 2 (equal for odd N; numpy's median is their mean).  Empty
    segments give NaN.  Returns two float arrays [nseg] in pi's dtype.
    """
    seg = np.asarray(seg, dtype=np.int64)
    lo = np.full(len(seg) - 1, np.nan, dtype=pi.dtype)
    hi = np.full(len(seg) - 1, np.nan, dtype=pi.dtype)
    for i in range(len(seg) - 1):
        x = np.sort(pi[seg[i]:seg[i + 1]])
        N = x.shape[0]
        if N:
            lo[i] = x[(N - 1) // 2]
            hi[i] = x[N // 2]
    return lo, hi


def splitmix64_raw(state: int, counter: int) -> int:
    return int(lib().oracle_splitmix64_raw(state, counter))


def splitmix64_draw(seed: int, stream: int, counter: int) -> int:
    return int(lib().oracle_splitmix64_draw(seed, stream, counter))


def schedule_uniform(seed: int, n: int, T: int):
    order = np.empty(T, dtype=np.int32)
    tau = np.empty(T, dtype=np.int32)
    if lib().oracle_schedule_uniform(seed, n, T, _ptr(order), _ptr(tau)):
        raise ValueError("invalid schedule arguments")
    return order, tau


def schedule_queue(seed: int, n: int, T: int, rate: float = 1.0):
    order = np.empty(T, dtype=np.int32)
    tau = np.empty(T, dtype=np.int32)
    if lib().oracle_schedule_queue(seed, n, T, rate, _ptr(order), _ptr(tau)):
        raise ValueError("invalid schedule arguments")
    return order, tau


def tf32_rna(x: float) -> float:
    return float(lib().oracle_tf32_rna(x))


def threads() -> int:
    return int(lib().oracle_threads())


def set_commit_threads(threads: int) -> int:
    """Threads that split the coordinates of each commit of gem_run (1 by default).  The
    result does not depend on it: every coordinate is updated independently.  Returns the
    previous value."""
    return int(lib().oracle_set_commit_threads(int(threads)))


def mlp_loss_grad(dims, theta, X, y, *, tf32=False):
    """Mean softmax cross-entropy and its gradient (double). theta [P], X [b, d0], y [b]."""
    dims_a = np.ascontiguousarray(dims, dtype=np.int32)
    theta = np.ascontiguousarray(theta, dtype=np.float64)
    X = np.ascontiguousarray(X, dtype=np.float64)
    y = np.ascontiguousarray(y, dtype=np.int32)
    grad = np.empty_like(theta)
    loss = lib().oracle_mlp_loss_grad_f64(len(dims) - 1, _ptr(dims_a), _ptr(theta), _ptr(X),
                                          _ptr(y), X.shape[0], _ptr(grad), int(tf32))
    return float(loss), grad


def mlp_sim_run(dims, theta, m, s, order, X, labels, batch_rows, *, eta, mu, eps, tau=None,
                mode=MODE_GEM, kappa=1.0, tf32=False, record_at=(), want_losses=False,
                record_pi=False):
    """End-to-end GEM on the MLP; fp32 state updated in place.  X [rows, d0] holds the
    rows that batch_rows [T, b] index.  Returns (records [len(record_at), P], losses), and
    with record_pi a third item, the scaling factors [T, P] of every commit."""
    dims_a = np.ascontiguousarray(dims, dtype=np.int32)
    for a, nm in ((theta, "theta"), (m, "m"), (s, "s")):
        _need(a, np.float32, nm)
    P = theta.shape[0]
    n = m.shape[0]
    order = np.ascontiguousarray(order, dtype=np.int32)
    T = order.shape[0]
    X = np.ascontiguousarray(X, dtype=np.float32)
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    batch_rows = np.ascontiguousarray(batch_rows, dtype=np.int32)
    b = batch_rows.shape[1]
    rec_at = np.ascontiguousarray(sorted(record_at), dtype=np.int32)
    rec = np.empty((len(rec_at), P), dtype=np.float32)
    losses = np.empty(T, dtype=np.float64) if want_losses else None
    tau_a = None if tau is None else np.ascontiguousarray(tau, dtype=np.int32)
    pi = np.empty((T, P), dtype=np.float32) if record_pi else None
    rc = lib().oracle_mlp_sim_run_pi(len(dims) - 1, _ptr(dims_a), n, T, _ptr(order), _ptr(tau_a),
                                     _ptr(X), X.shape[0], _ptr(labels), _ptr(batch_rows), b,
                                     _ptr(theta), _ptr(m), _ptr(s), P, eta, mu, eps, mode, kappa,
                                     int(tf32), len(rec_at), _ptr(rec_at), _ptr(rec), _ptr(losses),
                                     _ptr(pi))
    if rc:
        raise ValueError(f"oracle_mlp_sim_run failed ({rc})")
    return (rec, losses, pi) if record_pi else (rec, losses)


# The MNIST convolutional network of Appendix A: shape = (H, c1, c2, f1, f2, C).
CNN_MNIST = (28, 10, 20, 128, 64, 10)


def cnn_param_count(shape) -> int:
    sh = np.ascontiguousarray(shape, dtype=np.int32)
    P = int(lib().oracle_cnn_param_count(_ptr(sh)))
    if P < 0:
        raise ValueError(f"invalid network shape {tuple(shape)}")
    return P


def cnn_loss_grad(shape, theta, X, y, drop, *, want_logits=False):
    """Mean loss, gradient [P] (double) and optionally logits [b, C] of the network at
    theta for the samples X [b, H*H], labels y [b] and dropout scales drop [b, c2]."""
    sh = np.ascontiguousarray(shape, dtype=np.int32)
    theta = np.ascontiguousarray(theta, dtype=np.float64)
    X = np.ascontiguousarray(X, dtype=np.float64)
    y = np.ascontiguousarray(y, dtype=np.int32)
    drop = np.ascontiguousarray(drop, dtype=np.float64)
    b = X.shape[0]
    grad = np.empty_like(theta)
    logits = np.empty((b, shape[5]), dtype=np.float64) if want_logits else None
    loss = lib().oracle_cnn_loss_grad_f64(_ptr(sh), _ptr(theta), _ptr(X), _ptr(y), _ptr(drop), b,
                                          _ptr(grad), _ptr(logits))
    if np.isnan(loss):
        raise ValueError("invalid shape or label")
    return (float(loss), grad, logits) if want_logits else (float(loss), grad)


def cnn_sim_run(shape, theta, m, s, order, X, labels, batch_rows, drop, *, eta, mu, eps,
                tau=None, mode=MODE_GEM, kappa=1.0, record_at=(), want_losses=False):
    """End-to-end GEM on the CNN; fp32 state updated in place.  X [rows, H*H] holds the
    rows that batch_rows [T, b] index; drop [T, b, c2] the dropout scales of each commit.
    Returns (records [len(record_at), P], losses)."""
    sh = np.ascontiguousarray(shape, dtype=np.int32)
    for a, nm in ((theta, "theta"), (m, "m"), (s, "s")):
        _need(a, np.float32, nm)
    P = theta.shape[0]
    n = m.shape[0]
    order = np.ascontiguousarray(order, dtype=np.int32)
    T = order.shape[0]
    X = np.ascontiguousarray(X, dtype=np.float32)
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    batch_rows = np.ascontiguousarray(batch_rows, dtype=np.int32)
    drop = np.ascontiguousarray(drop, dtype=np.float32)
    b = batch_rows.shape[1]
    rec_at = np.ascontiguousarray(sorted(record_at), dtype=np.int32)
    rec = np.empty((len(rec_at), P), dtype=np.float32)
    losses = np.empty(T, dtype=np.float64) if want_losses else None
    tau_a = None if tau is None else np.ascontiguousarray(tau, dtype=np.int32)
    rc = lib().oracle_cnn_sim_run(_ptr(sh), n, T, _ptr(order), _ptr(tau_a), _ptr(X), X.shape[0],
                                  _ptr(labels), _ptr(batch_rows), b, _ptr(drop), _ptr(theta),
                                  _ptr(m), _ptr(s), P, eta, mu, eps, mode, kappa, len(rec_at),
                                  _ptr(rec_at), _ptr(rec), _ptr(losses))
    if rc:
        raise ValueError(f"oracle_cnn_sim_run failed ({rc})")
    return rec, losses
