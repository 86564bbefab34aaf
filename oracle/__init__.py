"""CPU oracle for the memory-planning path -- TEST INFRASTRUCTURE ONLY.

Plain single-threaded C (``oracle.c``) behind ctypes.  Only the tests, the
package's ``smoke()`` check and the bench's CPU-baseline leg may import this
package; the product path never does, and it shares no code with the CUDA
library.  Every function takes a ``tracegen.TraceSet`` (host numpy arrays).

Passages followed: Eq. 2.1 with its pairwise ordering constraints and the
strategy list of Sec. 2.3 (greedy_by_size, bump_allocation); Sec. 3.2 makes
greedy_by_size the default; Sec. 6 describes greedy by breadth (operators by
the sizes of their input and output tensors), read here with the operator at
step t producing the tensors allocated at t and using for the last time the
tensors freed at t + 1.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_HDR = os.path.join(_HERE, "oracle.h")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None

OK, EINVAL, EOVERFLOW = 0, 1, 2
FIT_FIRST, FIT_BEST = 0, 1


def build(force: bool = False) -> str:
    """Compile liboracle.so next to its source with gcc (no CUDA involved)."""
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= newest:
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-Wall", "-Wextra", "-o", tmp, _SRC],
                   check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Batch(ctypes.Structure):
    _fields_ = [
        ("n_traces", ctypes.c_int32),
        ("trace_ptr", ctypes.c_void_p),
        ("steps", ctypes.c_void_p),
        ("profile_ptr", ctypes.c_void_p),
        ("alloc_step", ctypes.c_void_p),
        ("free_step", ctypes.c_void_p),
        ("size_bytes", ctypes.c_void_p),
    ]


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    BP = ctypes.POINTER(_Batch)
    lib.or_live_profile.argtypes = [BP, P, P, P]
    lib.or_plan_greedy_by_size.argtypes = [BP, ctypes.c_int32, P, P, P]
    lib.or_plan_greedy_by_breadth.argtypes = [BP, ctypes.c_int32, P, P, P]
    lib.or_plan_bump.argtypes = [BP, P, P, P]
    lib.or_validate_plan.argtypes = [BP, P, P, P, P]
    lib.or_peak.argtypes = [BP, P, P, P]
    lib.or_bruteforce_opt.argtypes = [ctypes.c_int32, P, P, P, P]
    lib.or_bruteforce_opt.restype = ctypes.c_int64
    _lib = lib
    return lib


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _batch(ts, keep):
    arrs = [_c(ts.trace_ptr, np.int64), _c(ts.steps, np.int32), _c(ts.profile_ptr, np.int64),
            _c(ts.alloc_step, np.int32), _c(ts.free_step, np.int32), _c(ts.size_bytes, np.int64)]
    keep.extend(arrs)
    b = _Batch(ts.n_traces, *[a.ctypes.data for a in arrs])
    return ctypes.byref(b), b


def _out(n, dt):
    return np.zeros(max(int(n), 0), dtype=dt)


def live_profile(ts):
    """Returns (profile int64[sum T], peak_lb int64[B], status int32[B])."""
    lib, keep = _load(), []
    ref, _b = _batch(ts, keep)
    prof = _out(ts.n_steps, np.int64)
    lb = _out(ts.n_traces, np.int64)
    st = _out(ts.n_traces, np.int32)
    lib.or_live_profile(ref, prof.ctypes.data, lb.ctypes.data, st.ctypes.data)
    return prof, lb, st


def plan_greedy_by_size(ts, policy: int = FIT_FIRST):
    """Returns (offsets int64[N], plan_peak int64[B], status int32[B])."""
    lib, keep = _load(), []
    ref, _b = _batch(ts, keep)
    off = _out(ts.n_tensors, np.int64)
    peak = _out(ts.n_traces, np.int64)
    st = _out(ts.n_traces, np.int32)
    lib.or_plan_greedy_by_size(ref, int(policy), off.ctypes.data, peak.ctypes.data, st.ctypes.data)
    return off, peak, st


def plan_greedy_by_breadth(ts, policy: int = FIT_FIRST):
    """Greedy by breadth (operator at step t: outputs allocated at t, inputs last used at t): returns
    (offsets int64[N], plan_peak int64[B], status int32[B])."""
    lib, keep = _load(), []
    ref, _b = _batch(ts, keep)
    off = _out(ts.n_tensors, np.int64)
    peak = _out(ts.n_traces, np.int64)
    st = _out(ts.n_traces, np.int32)
    lib.or_plan_greedy_by_breadth(ref, int(policy), off.ctypes.data, peak.ctypes.data, st.ctypes.data)
    return off, peak, st


def plan_bump(ts):
    """bump_allocation: returns (offsets, plan_peak, status)."""
    lib, keep = _load(), []
    ref, _b = _batch(ts, keep)
    off = _out(ts.n_tensors, np.int64)
    peak = _out(ts.n_traces, np.int64)
    st = _out(ts.n_traces, np.int32)
    lib.or_plan_bump(ref, off.ctypes.data, peak.ctypes.data, st.ctypes.data)
    return off, peak, st


def validate_plan(ts, offsets):
    """Returns (verdict int32[B], conflict int32[B, 2], status int32[B])."""
    lib, keep = _load(), []
    ref, _b = _batch(ts, keep)
    off = _c(offsets, np.int64)
    verdict = _out(ts.n_traces, np.int32)
    conflict = _out(2 * ts.n_traces, np.int32)
    st = _out(ts.n_traces, np.int32)
    lib.or_validate_plan(ref, off.ctypes.data, verdict.ctypes.data, conflict.ctypes.data, st.ctypes.data)
    return verdict, conflict.reshape(-1, 2), st


def peak(ts, offsets):
    """Returns (plan_peak int64[B], status int32[B])."""
    lib, keep = _load(), []
    ref, _b = _batch(ts, keep)
    off = _c(offsets, np.int64)
    pk = _out(ts.n_traces, np.int64)
    st = _out(ts.n_traces, np.int32)
    lib.or_peak(ref, off.ctypes.data, pk.ctypes.data, st.ctypes.data)
    return pk, st


def bruteforce_opt(alloc, free, size):
    """Exact DSA optimum (Eq. 2.1) of one trace with at most 10 tensors: (total_mem, offsets)."""
    lib = _load()
    a, f, s = _c(alloc, np.int32), _c(free, np.int32), _c(size, np.int64)
    n = a.shape[0]
    if n > 10:
        raise ValueError("brute force is limited to 10 tensors")
    off = _out(n, np.int64)
    best = lib.or_bruteforce_opt(n, a.ctypes.data, f.ctypes.data, s.ctypes.data, off.ctypes.data)
    return int(best), off
