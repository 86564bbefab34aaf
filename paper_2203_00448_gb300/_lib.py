"""ctypes loader for libmemplan.so (the C ABI declared in include/memplan.h).

Loads the in-tree library only.  There is no fallback: if the library is
missing the import of any compute entry point raises.
"""
from __future__ import annotations

import ctypes
import os

from .build import LIB_PATH

OK, EINVAL, EOVERFLOW, ECUDA, ETIMEOUT, ENOMEM, EINTERNAL = range(7)
FIT_FIRST, FIT_BEST = 0, 1

# Every symbol include/memplan.h declares.
EXPORTS = (
    "mp_live_profile",
    "mp_plan_workspace_bytes",
    "mp_plan_greedy_by_size",
    "mp_plan_greedy_by_size_static",
    "mp_plan_and_validate",
    "mp_host_path_bytes",
    "mp_plan_and_validate_host",
    "mp_validate_workspace_bytes",
    "mp_validate_plan",
    "mp_peak",
    "mp_bump_workspace_bytes",
    "mp_plan_bump",
    "mp_optimal_workspace_bytes",
    "mp_plan_optimal",
    "mp_breadth_workspace_bytes",
    "mp_plan_greedy_by_breadth",
    "mp_slab_layout",
    "mp_replay_workspace_bytes",
    "mp_replay_plan",
    "mp_status_string",
    "mp_abi_version",
)


class MpBatch(ctypes.Structure):
    """Mirror of struct mp_batch."""

    _fields_ = [
        ("n_traces", ctypes.c_int32),
        ("max_tensors", ctypes.c_int32),
        ("max_steps", ctypes.c_int32),
        ("reserved0", ctypes.c_int32),
        ("n_tensors", ctypes.c_int64),
        ("n_steps", ctypes.c_int64),
        ("trace_ptr", ctypes.c_void_p),
        ("steps", ctypes.c_void_p),
        ("profile_ptr", ctypes.c_void_p),
        ("alloc_step", ctypes.c_void_p),
        ("free_step", ctypes.c_void_p),
        ("size_bytes", ctypes.c_void_p),
    ]


class MpHostResults(ctypes.Structure):
    """Mirror of struct mp_host_results."""

    _fields_ = [(name, ctypes.c_void_p) for name in
                ("profile", "peak_lb", "offsets", "plan_peak", "verdict", "conflict", "trace_status")]


HOST_PATH_MAX_CHUNKS = 64
SLAB_ALIGN = 256  # MP_SLAB_ALIGN


class MemplanError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} returned {status_string(status)}")
        self.status = status


_lib = None


def load(path: str = LIB_PATH):
    """Loads libmemplan.so and declares the signatures; raises if it is absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2203_00448_gb300.build.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    P, BP = ctypes.c_void_p, ctypes.POINTER(MpBatch)
    i32, sz = ctypes.c_int32, ctypes.c_size_t
    lib.mp_live_profile.argtypes = [BP, P, P, P, P]
    lib.mp_live_profile.restype = i32
    lib.mp_plan_workspace_bytes.argtypes = [BP]
    lib.mp_plan_workspace_bytes.restype = sz
    lib.mp_plan_greedy_by_size.argtypes = [BP, i32, P, P, P, P, sz, P]
    lib.mp_plan_greedy_by_size.restype = i32
    lib.mp_plan_greedy_by_size_static.argtypes = [BP, i32, P, P, P, P]
    lib.mp_plan_greedy_by_size_static.restype = i32
    lib.mp_plan_and_validate.argtypes = [BP, i32, P, P, P, P, P, P, P, P, sz, P]
    lib.mp_plan_and_validate.restype = i32
    lib.mp_host_path_bytes.argtypes = [BP, i32]
    lib.mp_host_path_bytes.restype = sz
    lib.mp_plan_and_validate_host.argtypes = [BP, i32, ctypes.POINTER(MpHostResults), i32, P, sz, P, P, P]
    lib.mp_plan_and_validate_host.restype = i32
    lib.mp_validate_workspace_bytes.argtypes = [BP]
    lib.mp_validate_workspace_bytes.restype = sz
    lib.mp_validate_plan.argtypes = [BP, P, P, P, P, P, sz, P]
    lib.mp_validate_plan.restype = i32
    lib.mp_peak.argtypes = [BP, P, P, P, P]
    lib.mp_peak.restype = i32
    lib.mp_bump_workspace_bytes.argtypes = [BP]
    lib.mp_bump_workspace_bytes.restype = sz
    lib.mp_plan_bump.argtypes = [BP, P, P, P, P, sz, P]
    lib.mp_plan_bump.restype = i32
    lib.mp_optimal_workspace_bytes.argtypes = [BP]
    lib.mp_optimal_workspace_bytes.restype = sz
    lib.mp_plan_optimal.argtypes = [BP, P, P, P, P, sz, P]
    lib.mp_plan_optimal.restype = i32
    lib.mp_breadth_workspace_bytes.argtypes = [BP]
    lib.mp_breadth_workspace_bytes.restype = sz
    lib.mp_plan_greedy_by_breadth.argtypes = [BP, i32, P, P, P, P, sz, P]
    lib.mp_plan_greedy_by_breadth.restype = i32
    lib.mp_slab_layout.argtypes = [BP, P, P, P, P, P, P]
    lib.mp_slab_layout.restype = i32
    lib.mp_replay_workspace_bytes.argtypes = [BP]
    lib.mp_replay_workspace_bytes.restype = sz
    lib.mp_replay_plan.argtypes = [BP, P, P, P, ctypes.c_int64, P, P, P, P, sz, P]
    lib.mp_replay_plan.restype = i32
    lib.mp_status_string.argtypes = [i32]
    lib.mp_status_string.restype = ctypes.c_char_p
    lib.mp_abi_version.argtypes = []
    lib.mp_abi_version.restype = i32
    _lib = lib
    return lib


def status_string(status: int) -> str:
    try:
        return load().mp_status_string(int(status)).decode()
    except RuntimeError:
        return f"status {status}"
