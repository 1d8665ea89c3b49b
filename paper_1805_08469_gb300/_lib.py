"""Loader of the in-tree CUDA library ``libgem.so`` (ctypes).

There is no fallback: when the library is missing or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes as C
from pathlib import Path

LIB_PATH = Path(__file__).resolve().parent / "libgem.so"

_lib = None


class GemError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


def _declare(L):
    p, i, sz = C.c_void_p, C.c_int, C.c_size_t
    sig = {
        "gem_create": ([sz, i, C.c_float, C.c_float, C.c_float, p], i),
        "gem_destroy": ([p], None),
        "gem_set_stream": ([p, p], i),
        "gem_set_theta": ([p, p], i),
        "gem_pull": ([p, i, p], i),
        "gem_moment": ([p, i, p], i),
        "gem_theta": ([p, p], i),
        "gem_commit": ([p, i, p], i),
        "gem_commit_batch": ([p, p, p, i], i),
        "gem_commit_batch_host": ([p, p, p, i], i),
        "gem_read_theta": ([p, p], i),
        "gem_save_state": ([p, p, p, p], i),
        "gem_load_state": ([p, p, p, p], i),
        "gem_sync": ([p], i),
        "gem_shape": ([p, p, p, p], i),
        "gem_launch_count": ([p], C.c_uint64),
        "gem_set_mode": ([p, i, C.c_float], i),
        "gem_get_mode": ([p, p, p], i),
        "gem_staleness": ([p, i, p], i),
        "gem_get_clock": ([p, p, p], i),
        "gem_set_clock": ([p, C.c_int64, p], i),
        "gem_commit_batch_pi": ([p, p, p, i, p], i),
        "gem_pi_median": ([p, p, i, p, i, p, p], i),
        "gem_commit_batch_pi_median": ([p, p, p, i, p, p, i, p, p], i),
        "gem_status_string": ([i], C.c_char_p),
        "gem_shard_range": ([C.c_size_t, i, i, p, p], i),
        "gem_schedule_uniform": ([C.c_uint64, i, i, p, p], i),
        "gem_schedule_queue": ([C.c_uint64, i, i, C.c_double, p, p], i),
        "gem_plan_segments": ([p, i, i, p], i),
        "gem_mlp_create": ([p, i, p, i, i, p], i),
        "gem_mlp_set_data": ([p, p, p, C.c_int64], i),
        "gem_mlp_grad": ([p, p, i, p, p, p], i),
        "gem_mlp_run": ([p, p, i, p, p], i),
        "gem_mlp_run_pi": ([p, p, i, p, p, p, p], i),
        "gem_mlp_destroy": ([p], None),
        "gem_mlp_status": ([p], i),
        "gem_mlp_grad_static": ([i, p, i, i, p, p, p, C.c_int64, p, p, p, p], i),
        "gem_mlp_launch_count": ([p], C.c_uint64),
        "gem_cnn_param_count": ([p], C.c_int64),
        "gem_cnn_create": ([p, p, i, p], i),
        "gem_cnn_set_data": ([p, p, p, C.c_int64], i),
        "gem_cnn_grad": ([p, p, i, p, p, p, p], i),
        "gem_cnn_run": ([p, p, i, p, p, p], i),
        "gem_cnn_run_pi": ([p, p, i, p, p, p, p, p], i),
        "gem_cnn_status": ([p], i),
        "gem_cnn_launch_count": ([p], C.c_uint64),
        "gem_cnn_destroy": ([p], None),
        "gem_synth_theta0": ([C.c_uint64, sz, p, p], i),
        "gem_synth_grad_heavytail": ([C.c_uint64, C.c_uint64, i, sz, sz, p, p], i),
        "gem_synth_grad_loguniform": ([C.c_uint64, C.c_uint64, sz, p, p, p], i),
        "gem_synth_data": ([C.c_uint64, i, i, i, p, p, p], i),
        "gem_synth_xavier": ([C.c_uint64, p, i, p, p], i),
        "gem_synth_cnn_theta0": ([C.c_uint64, p, p, p], i),
        "gem_synth_dropout": ([C.c_uint64, C.c_uint64, i, i, i, C.c_float, p, p], i),
        "gem_synth_cnn_data": ([C.c_uint64, i, i, i, p, p, p], i),
    }
    for name, (args, res) in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = res
    return L


def lib():
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not LIB_PATH.exists():
            raise RuntimeError(
                f"{LIB_PATH} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()')")
        _lib = _declare(C.CDLL(str(LIB_PATH)))
    return _lib


def status_string(status: int) -> str:
    try:
        return lib().gem_status_string(status).decode()
    except Exception:
        return "unknown"


def check(status: int, where: str) -> None:
    if status != 0:
        raise GemError(status, where)
