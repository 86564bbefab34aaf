"""Seeded synthetic allocation traces (input generator shared by the oracle and the CUDA path).

The paper's traces come from an instrumented allocator run over real models
(Sec. 3.1, Table 3.1); none exist here, so the workloads below are seeded
stand-ins shaped after Table 1.1, Table 3.1 and the size distributions of
Sec. 2.2.  This module holds random sampling only -- no planning arithmetic --
and is the one module both sides of the parity tests import.

A batch is a structure of arrays with CSR offsets:

* ``trace_ptr``  int64[B+1]  tensor range of trace b is [trace_ptr[b], trace_ptr[b+1])
* ``steps``      int32[B]    T_b, the number of op steps of trace b
* ``profile_ptr`` int64[B+1] exclusive prefix sum of ``steps`` (profile output CSR)
* ``alloc_step`` int32[N]    first step a tensor is live
* ``free_step``  int32[N]    first step it is no longer live (exclusive)
* ``size_bytes`` int64[N]    bytes
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tracegen.c")
_LIB_PATH = os.path.join(_HERE, "libtracegen.so")
_lib = None

# Five workloads: (name, description).  Sizes and seeds are fixed here.
CONFIG_NAMES = {
    0: "random-64x128-seed0",
    1: "resnet50-chain-374-seed1",
    2: "batched-random-4096x512x1024-seeds0-4095",
    3: "long-tail-20000x10000-seed7",
    4: "seq2seq-256x2000x4000-seeds100-355",
}


def build(force: bool = False) -> str:
    """Compile libtracegen.so next to its source (gcc, no FP contraction)."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
           "-Wall", "-Wextra", "-o", tmp, _SRC]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    i32, i64, u64, dbl = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
    lib.tg_debug_next.argtypes = [u64, i32]
    lib.tg_debug_next.restype = u64
    lib.tg_debug_exp2.argtypes = [dbl]
    lib.tg_debug_exp2.restype = dbl
    lib.tg_debug_uniform_int.argtypes = [u64, i64, i64, i32]
    lib.tg_debug_uniform_int.restype = i64
    lib.tg_random_trace.argtypes = [u64, i32, i32, dbl, i32, i32, P, P, P]
    lib.tg_random_trace.restype = None
    lib.tg_random_batch.argtypes = [u64, i32, i32, i32, dbl, i32, i32, P, P, P]
    lib.tg_random_batch.restype = None
    lib.tg_resnet_chain_trace.argtypes = [u64, P, P, P]
    lib.tg_resnet_chain_trace.restype = i32
    lib.tg_long_tail_trace.argtypes = [u64, i32, i32, i32, i32, i32, dbl, i32, i32, P, P, P, P, P]
    lib.tg_long_tail_trace.restype = None
    lib.tg_seq2seq_trace.argtypes = [u64, i32, i32, i32, dbl, P, P, P, P, P]
    lib.tg_seq2seq_trace.restype = None
    _lib = lib
    return lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


@dataclass
class TraceSet:
    """A batch of traces in host memory (numpy), structure of arrays + CSR."""

    trace_ptr: np.ndarray
    steps: np.ndarray
    profile_ptr: np.ndarray
    alloc_step: np.ndarray
    free_step: np.ndarray
    size_bytes: np.ndarray
    name: str = "custom"

    @property
    def n_traces(self) -> int:
        return int(self.steps.shape[0])

    @property
    def n_tensors(self) -> int:
        return int(self.alloc_step.shape[0])

    @property
    def n_steps(self) -> int:
        return int(self.profile_ptr[-1]) if self.profile_ptr.shape[0] else 0

    @property
    def max_tensors(self) -> int:
        return int(np.max(np.diff(self.trace_ptr))) if self.n_traces else 0

    @property
    def max_steps(self) -> int:
        return int(np.max(self.steps)) if self.n_traces else 0

    def trace(self, b: int):
        lo, hi = int(self.trace_ptr[b]), int(self.trace_ptr[b + 1])
        return (int(self.steps[b]), self.alloc_step[lo:hi], self.free_step[lo:hi], self.size_bytes[lo:hi])

    def pairs(self) -> int:
        """Number of unordered tensor pairs N_b (N_b - 1) / 2 summed over traces."""
        n = np.diff(self.trace_ptr).astype(np.int64)
        return int(np.sum(n * (n - 1) // 2))

    def select(self, traces) -> "TraceSet":
        """A new TraceSet holding only the listed traces, in the given order."""
        traces = [int(b) for b in traces]
        parts = [self.trace(b) for b in traces]
        return from_arrays([(T, a, f, s) for (T, a, f, s) in parts], name=f"{self.name}[sel{len(traces)}]")


def _csr(steps: np.ndarray, counts: np.ndarray):
    trace_ptr = np.zeros(len(counts) + 1, dtype=np.int64)
    np.cumsum(counts, out=trace_ptr[1:])
    profile_ptr = np.zeros(len(steps) + 1, dtype=np.int64)
    np.cumsum(steps.astype(np.int64), out=profile_ptr[1:])
    return trace_ptr, profile_ptr


def from_arrays(traces, name: str = "custom") -> TraceSet:
    """Build a TraceSet from a list of (T, alloc, free, size) tuples (any array-likes)."""
    steps = np.array([int(t[0]) for t in traces], dtype=np.int32)
    counts = np.array([len(t[1]) for t in traces], dtype=np.int64)
    trace_ptr, profile_ptr = _csr(steps, counts)
    cat = lambda k, dt: (np.concatenate([np.asarray(t[k], dtype=dt) for t in traces])
                         if len(traces) else np.zeros(0, dtype=dt))
    return TraceSet(trace_ptr, steps, profile_ptr, cat(1, np.int32), cat(2, np.int32), cat(3, np.int64), name)


def from_tuples(traces, name: str = "custom") -> TraceSet:
    """Build a TraceSet from a list of (T, [(alloc, free, size), ...])."""
    out = []
    for T, tensors in traces:
        arr = np.array(tensors, dtype=np.int64).reshape(-1, 3)
        out.append((T, arr[:, 0], arr[:, 1], arr[:, 2]))
    return from_arrays(out, name)


def random_batch(seed0: int, n_traces: int, n: int, T: int, p: float = 0.5, lo_e: int = 6,
                 hi_e: int = 20, name: str | None = None) -> TraceSet:
    """n_traces random traces (seeds seed0 .. seed0 + n_traces - 1), each n tensors over T steps."""
    lib = _load()
    N = n_traces * n
    a = np.empty(N, dtype=np.int32)
    f = np.empty(N, dtype=np.int32)
    s = np.empty(N, dtype=np.int64)
    if N:
        lib.tg_random_batch(seed0, n_traces, n, T, p, lo_e, hi_e, _ptr(a), _ptr(f), _ptr(s))
    steps = np.full(n_traces, T, dtype=np.int32)
    trace_ptr, profile_ptr = _csr(steps, np.full(n_traces, n, dtype=np.int64))
    return TraceSet(trace_ptr, steps, profile_ptr, a, f, s,
                    name or f"random-{n_traces}x{n}x{T}-seed{seed0}")


def resnet_chain(seed: int = 1) -> TraceSet:
    lib = _load()
    a = np.empty(374, dtype=np.int32)
    f = np.empty(374, dtype=np.int32)
    s = np.empty(374, dtype=np.int64)
    n = lib.tg_resnet_chain_trace(seed, _ptr(a), _ptr(f), _ptr(s))
    return from_arrays([(160, a[:n], f[:n], s[:n])], name=f"resnet50-chain-{n}-seed{seed}")


def long_tail(seed: int = 7, n: int = 20000, T: int = 10000, n_long: int = 1000, long_lo: int = 100,
              long_hi: int = 5000, p: float = 0.4, lo_e: int = 6, hi_e: int = 26) -> TraceSet:
    lib = _load()
    a = np.empty(n, dtype=np.int32)
    f = np.empty(n, dtype=np.int32)
    s = np.empty(n, dtype=np.int64)
    idx = np.empty(max(n, 1), dtype=np.int32)
    mark = np.empty(max(n, 1), dtype=np.uint8)
    lib.tg_long_tail_trace(seed, n, T, n_long, long_lo, long_hi, p, lo_e, hi_e, _ptr(a), _ptr(f), _ptr(s),
                           _ptr(idx), _ptr(mark))
    return from_arrays([(T, a, f, s)], name=f"long-tail-{n}x{T}-seed{seed}")


def seq2seq_batch(seed0: int = 100, n_traces: int = 256, n: int = 2000, T: int = 4000,
                  n_full: int = 40, p: float = 0.3) -> TraceSet:
    lib = _load()
    N = n_traces * n
    a = np.empty(N, dtype=np.int32)
    f = np.empty(N, dtype=np.int32)
    s = np.empty(N, dtype=np.int64)
    idx = np.empty(max(n, 1), dtype=np.int32)
    mark = np.empty(max(n, 1), dtype=np.uint8)
    for k in range(n_traces):
        lo = k * n
        lib.tg_seq2seq_trace(seed0 + k, n, T, n_full, p, _ptr(a[lo:]), _ptr(f[lo:]), _ptr(s[lo:]),
                             _ptr(idx), _ptr(mark))
    steps = np.full(n_traces, T, dtype=np.int32)
    trace_ptr, profile_ptr = _csr(steps, np.full(n_traces, n, dtype=np.int64))
    return TraceSet(trace_ptr, steps, profile_ptr, a, f, s, f"seq2seq-{n_traces}x{n}x{T}-seed{seed0}")


def config(k: int) -> TraceSet:
    """The five fixed workloads.

    0  one random trace: 64 tensors, T = 128, seed 0, sizes log-uniform 64 B .. 1 MiB
    1  ResNet-50-shaped chain: 160 ops, 374 tensors, seed 1
    2  4096 random traces of 512 tensors over T = 1024, seeds 0 .. 4095
    3  one 20,000-tensor trace over T = 10,000 with 1,000 long-lived tensors, seed 7
    4  256 seq2seq serving traces of 2,000 tensors over T = 4,000, seeds 100 .. 355
    """
    if k == 0:
        ts = random_batch(0, 1, 64, 128, 0.5, 6, 20)
    elif k == 1:
        ts = resnet_chain(1)
    elif k == 2:
        ts = random_batch(0, 4096, 512, 1024, 0.5, 6, 20)
    elif k == 3:
        ts = long_tail()
    elif k == 4:
        ts = seq2seq_batch()
    else:
        raise ValueError(f"no workload {k}")
    ts.name = CONFIG_NAMES[k]
    return ts


def random_small(seed: int, n_traces: int, n_max: int, T_max: int, size_max: int = 1 << 12):
    """Random small traces for property tests: per trace N ~ U[0, n_max], T ~ U[1, T_max],
    alloc/free uniform, sizes uniform in [1, size_max].  Uses numpy's PCG64."""
    rng = np.random.default_rng(seed)
    traces = []
    for _ in range(n_traces):
        T = int(rng.integers(1, T_max + 1))
        n = int(rng.integers(0, n_max + 1))
        a = rng.integers(0, T, size=n)
        life = rng.integers(1, T + 1, size=n)
        f = np.minimum(a + life, T)
        s = rng.integers(1, size_max + 1, size=n)
        traces.append((T, a, f, s))
    return from_arrays(traces, name=f"random-small-seed{seed}")


def digest(ts: TraceSet) -> str:
    """SHA-256 over the batch's arrays (detects generator drift across hosts)."""
    import hashlib

    h = hashlib.sha256()
    for arr in (ts.trace_ptr, ts.steps, ts.profile_ptr, ts.alloc_step, ts.free_step, ts.size_bytes):
        h.update(np.ascontiguousarray(arr).tobytes())
    return h.hexdigest()
