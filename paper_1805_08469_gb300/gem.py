"""Python binding of the GEM commit ABI (include/gem.h).

Argument marshalling only: each function has the name of the C entry point it calls and
forwards raw pointers, sizes and the stream.  Every step of a commit runs in the CUDA
library; there is no CPU path.  Loading fails loudly when ``libgem.so`` is missing.
"""
from __future__ import annotations

import ctypes as C
from typing import Sequence

from ._lib import check, lib

GEM_OK = 0
GEM_EINVAL = -1
GEM_ENOMEM = -2
GEM_ECUDA = -3
GEM_ESTATE = -4

GEM_MODE_GEM = 0
GEM_MODE_DOWNPOUR = 1
GEM_MODE_ADAPTIVE = 2
GEM_MODE_KAPPA_SQRT = 3
GEM_MODE_KAPPA_LINEAR = 4
GEM_MODE_MOMENTUM = 5


def _dev_ptr(t, what: str) -> int:
    """Address of a contiguous fp32 CUDA tensor (or an int address)."""
    if isinstance(t, int):
        return t
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{what}: expected a torch.Tensor or an int address")
    if t.dtype != torch.float32 or not t.is_contiguous():
        raise TypeError(f"{what}: expected a contiguous float32 tensor")
    return t.data_ptr()


def _stream_ptr(stream) -> int:
    if stream is None:
        return 0
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def gem_create(P: int, n: int, eta: float, mu: float, eps: float) -> int:
    h = C.c_void_p()
    check(lib().gem_create(P, n, eta, mu, eps, C.byref(h)), "gem_create")
    return int(h.value)


def gem_destroy(h: int) -> None:
    lib().gem_destroy(C.c_void_p(h))


def gem_set_stream(h: int, stream) -> None:
    check(lib().gem_set_stream(C.c_void_p(h), C.c_void_p(_stream_ptr(stream))), "gem_set_stream")


def gem_set_theta(h: int, theta0) -> None:
    import torch
    if isinstance(theta0, torch.Tensor):
        if theta0.dtype != torch.float32 or not theta0.is_contiguous():
            raise TypeError("theta0: expected a contiguous float32 tensor")
        ptr = theta0.data_ptr()
    else:
        ptr = int(theta0)
    check(lib().gem_set_theta(C.c_void_p(h), C.c_void_p(ptr)), "gem_set_theta")


def gem_pull(h: int, worker: int) -> int:
    p = C.c_void_p()
    check(lib().gem_pull(C.c_void_p(h), worker, C.byref(p)), "gem_pull")
    return int(p.value)


def gem_moment(h: int, worker: int) -> int:
    p = C.c_void_p()
    check(lib().gem_moment(C.c_void_p(h), worker, C.byref(p)), "gem_moment")
    return int(p.value)


def gem_theta(h: int) -> int:
    p = C.c_void_p()
    check(lib().gem_theta(C.c_void_p(h), C.byref(p)), "gem_theta")
    return int(p.value)


def gem_commit(h: int, worker: int, grad) -> None:
    check(lib().gem_commit(C.c_void_p(h), worker, C.c_void_p(_dev_ptr(grad, "grad"))), "gem_commit")


def _batch_arrays(order: Sequence[int], ptrs: Sequence[int]):
    K = len(order)
    if len(ptrs) != K:
        raise ValueError("order and grads differ in length")
    o = (C.c_int * K)(*[int(w) for w in order])
    g = (C.c_void_p * K)(*ptrs)
    return o, g, K


def gem_commit_batch(h: int, order: Sequence[int], grads: Sequence) -> None:
    o, g, K = _batch_arrays(order, [_dev_ptr(x, "grads[k]") for x in grads])
    check(lib().gem_commit_batch(C.c_void_p(h), o, g, K), "gem_commit_batch")


def gem_commit_batch_pi(h: int, order: Sequence[int], grads: Sequence, pi: Sequence) -> None:
    """gem_commit_batch that also writes each commit's scaling factors to pi[k] (a [P]
    float32 CUDA tensor, or None for a commit whose factors are not wanted)."""
    o, g, K = _batch_arrays(order, [_dev_ptr(x, "grads[k]") for x in grads])
    if len(pi) != K:
        raise ValueError("order and pi differ in length")
    pp = (C.c_void_p * max(K, 1))(*[None if x is None else _dev_ptr(x, "pi[k]") for x in pi])
    check(lib().gem_commit_batch_pi(C.c_void_p(h), o, g, K, pp), "gem_commit_batch_pi")


def gem_pi_median(h: int, pi: Sequence, seg: Sequence[int], lo, hi) -> None:
    """Per-segment lower / upper medians of the rows pi[k] into lo, hi [K, nseg] (float32
    CUDA tensors); seg holds nseg + 1 offsets.  Stream-ordered."""
    K = len(pi)
    rows = (C.c_void_p * max(K, 1))(*[_dev_ptr(x, "pi[k]") for x in pi])
    sg = (C.c_int64 * len(seg))(*[int(x) for x in seg])
    check(lib().gem_pi_median(C.c_void_p(h), rows, K, sg, len(seg) - 1,
                              C.c_void_p(_dev_ptr(lo, "lo")), C.c_void_p(_dev_ptr(hi, "hi"))),
          "gem_pi_median")


def gem_commit_batch_pi_median(h: int, order: Sequence[int], grads: Sequence, pi: Sequence,
                               seg: Sequence[int], lo, hi) -> None:
    """gem_commit_batch_pi with every factor recorded in pi[k] ([P] float32 CUDA tensors),
    then the per-segment lower / upper medians of those rows into lo, hi [K, nseg], with the
    factor counts taken by the commit kernel.  Stream-ordered."""
    o, g, K = _batch_arrays(order, [_dev_ptr(x, "grads[k]") for x in grads])
    if len(pi) != K:
        raise ValueError("order and pi differ in length")
    rows = (C.c_void_p * max(K, 1))(*[_dev_ptr(x, "pi[k]") for x in pi])
    sg = (C.c_int64 * len(seg))(*[int(x) for x in seg])
    check(lib().gem_commit_batch_pi_median(C.c_void_p(h), o, g, K, rows, sg, len(seg) - 1,
                                           C.c_void_p(_dev_ptr(lo, "lo")),
                                           C.c_void_p(_dev_ptr(hi, "hi"))),
          "gem_commit_batch_pi_median")


def gem_commit_batch_host(h: int, order: Sequence[int], grads: Sequence) -> None:
    ptrs = []
    for x in grads:
        if isinstance(x, int):
            ptrs.append(x)
        else:
            if x.dtype.itemsize != 4 or not x.is_contiguous() or x.is_cuda:
                raise TypeError("grads[k]: expected a contiguous float32 host tensor")
            ptrs.append(x.data_ptr())
    o, g, K = _batch_arrays(order, ptrs)
    check(lib().gem_commit_batch_host(C.c_void_p(h), o, g, K), "gem_commit_batch_host")


def gem_read_theta(h: int, out) -> None:
    if isinstance(out, int):
        ptr = out
    else:
        if out.dtype.itemsize != 4 or not out.is_contiguous():
            raise TypeError("out: expected a contiguous float32 tensor")
        ptr = out.data_ptr()
    check(lib().gem_read_theta(C.c_void_p(h), C.c_void_p(ptr)), "gem_read_theta")


def _any_ptr(x) -> int:
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if x.dtype.itemsize != 4 or not x.is_contiguous():
            raise TypeError("expected a contiguous float32 tensor")
        return x.data_ptr()
    import numpy as np
    if isinstance(x, np.ndarray):
        if x.dtype != np.float32 or not x.flags.c_contiguous:
            raise TypeError("expected a C-contiguous float32 array")
        return x.ctypes.data
    raise TypeError("expected a tensor, an array or an address")


def gem_save_state(h: int, theta=None, m=None, s=None) -> None:
    """Copies theta [P], m [n, P], s [n, P] out (host or device buffers); stream-ordered."""
    check(lib().gem_save_state(C.c_void_p(h), C.c_void_p(_any_ptr(theta)), C.c_void_p(_any_ptr(m)),
                               C.c_void_p(_any_ptr(s))), "gem_save_state")


def gem_load_state(h: int, theta=None, m=None, s=None) -> None:
    """Replaces theta [P], m [n, P], s [n, P] (host or device buffers); stream-ordered."""
    check(lib().gem_load_state(C.c_void_p(h), C.c_void_p(_any_ptr(theta)), C.c_void_p(_any_ptr(m)),
                               C.c_void_p(_any_ptr(s))), "gem_load_state")


def gem_shard_range(P: int, world: int, rank: int) -> tuple[int, int]:
    """[begin, end) of parameter shard `rank` of `world` (contiguous, 128-byte boundaries);
    host-only."""
    b, e = C.c_size_t(), C.c_size_t()
    check(lib().gem_shard_range(P, world, rank, C.byref(b), C.byref(e)), "gem_shard_range")
    return int(b.value), int(e.value)


def gem_sync(h: int) -> None:
    check(lib().gem_sync(C.c_void_p(h)), "gem_sync")


def gem_shape(h: int) -> tuple[int, int, int]:
    P = C.c_size_t()
    n = C.c_int()
    stride = C.c_size_t()
    check(lib().gem_shape(C.c_void_p(h), C.byref(P), C.byref(n), C.byref(stride)), "gem_shape")
    return int(P.value), int(n.value), int(stride.value)


def gem_launch_count(h: int) -> int:
    return int(lib().gem_launch_count(C.c_void_p(h)))


def gem_set_mode(h: int, mode: int, kappa: float = 1.0) -> None:
    check(lib().gem_set_mode(C.c_void_p(h), int(mode), float(kappa)), "gem_set_mode")


def gem_get_mode(h: int) -> tuple[int, float]:
    mode = C.c_int()
    kappa = C.c_float()
    check(lib().gem_get_mode(C.c_void_p(h), C.byref(mode), C.byref(kappa)), "gem_get_mode")
    return int(mode.value), float(kappa.value)


def gem_staleness(h: int, worker: int) -> int:
    tau = C.c_int64()
    check(lib().gem_staleness(C.c_void_p(h), int(worker), C.byref(tau)), "gem_staleness")
    return int(tau.value)


def gem_get_clock(h: int, n: int):
    """(clock, last[n]) of the handle's commit clock."""
    clock = C.c_int64()
    last = (C.c_int64 * n)()
    check(lib().gem_get_clock(C.c_void_p(h), C.byref(clock), last), "gem_get_clock")
    return int(clock.value), [int(x) for x in last]


def gem_set_clock(h: int, clock: int, last=None) -> None:
    arr = None if last is None else (C.c_int64 * len(last))(*[int(x) for x in last])
    check(lib().gem_set_clock(C.c_void_p(h), int(clock), arr), "gem_set_clock")


class _DeviceArray:
    """Exposes a borrowed device address as a CUDA array (zero-copy torch view)."""

    def __init__(self, ptr: int, count: int):
        self.__cuda_array_interface__ = {"shape": (count,), "typestr": "<f4",
                                         "data": (ptr, False), "version": 3, "strides": None}


def device_view(ptr: int, count: int):
    import torch
    return torch.as_tensor(_DeviceArray(ptr, count), device="cuda")


class Gem:
    """Owning wrapper of a GEM handle with torch views of its state."""

    def __init__(self, P: int, n: int, eta: float, mu: float, eps: float, stream=None):
        self.h = gem_create(P, n, eta, mu, eps)
        self.P, self.n, self.stride = gem_shape(self.h)
        if stream is not None:
            gem_set_stream(self.h, stream)

    def close(self):
        if self.h:
            gem_destroy(self.h)
            self.h = 0

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_stream(self, stream):
        gem_set_stream(self.h, stream)

    def set_theta(self, theta0):
        gem_set_theta(self.h, theta0)

    def commit(self, worker: int, grad):
        gem_commit(self.h, worker, grad)

    def commit_batch(self, order, grads):
        gem_commit_batch(self.h, order, grads)

    def commit_batch_host(self, order, grads):
        gem_commit_batch_host(self.h, order, grads)

    def commit_batch_pi(self, order, grads, pi):
        gem_commit_batch_pi(self.h, order, grads, pi)

    def commit_batch_pi_median(self, order, grads, pi, seg, lo, hi):
        gem_commit_batch_pi_median(self.h, order, grads, pi, seg, lo, hi)

    def pi_median(self, pi, seg, lo, hi):
        gem_pi_median(self.h, pi, seg, lo, hi)

    def sync(self):
        gem_sync(self.h)

    def theta(self):
        return device_view(gem_theta(self.h), self.P)

    def snapshot(self, worker: int):
        return device_view(gem_pull(self.h, worker), self.P)

    def moment(self, worker: int):
        return device_view(gem_moment(self.h, worker), self.P)

    def launches(self) -> int:
        return gem_launch_count(self.h)

    def set_mode(self, mode: int, kappa: float = 1.0):
        gem_set_mode(self.h, mode, kappa)

    def staleness(self, worker: int) -> int:
        return gem_staleness(self.h, worker)

    def clock(self):
        return gem_get_clock(self.h, self.n)

    def set_clock(self, clock: int, last=None):
        gem_set_clock(self.h, clock, last)
