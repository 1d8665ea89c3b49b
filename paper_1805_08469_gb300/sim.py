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
