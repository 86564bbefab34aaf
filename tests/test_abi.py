"""The C ABI library: builds, loads, exports every declared symbol, and rejects
bad host-side arguments before touching the GPU (so these run without one)."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2203_00448_gb300 import _lib, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "memplan.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mp_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return _lib.load()


def test_header_and_binding_agree():
    assert declared_functions() == sorted(_lib.EXPORTS)


def test_every_declared_symbol_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", build.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\s(mp_\w+)$", out, flags=re.M))
    for name in declared_functions():
        assert name in exported, name
        assert getattr(lib, name) is not None
    # nothing else leaks out under the mp_ prefix
    assert exported == set(declared_functions())


def test_status_strings(lib):
    assert lib.mp_abi_version() == 2
    names = [lib.mp_status_string(k).decode() for k in range(7)]
    assert names == ["MP_OK", "MP_EINVAL", "MP_EOVERFLOW", "MP_ECUDA", "MP_ETIMEOUT", "MP_ENOMEM", "MP_EINTERNAL"]
    assert lib.mp_status_string(99).decode() == "MP_UNKNOWN"


def _batch(**kw):
    # Fake device addresses: every call below must fail its host-side checks
    # before any CUDA call could dereference them.
    b = _lib.MpBatch(4, 16, 16, 0, 40, 40, 0x1000, 0x2000, 0x3000, 0x4000, 0x5000, 0x6000)
    for k, v in kw.items():
        setattr(b, k, v)
    return b


def test_host_argument_errors(lib):
    P = 0x10000
    EINVAL, ENOMEM = _lib.EINVAL, _lib.ENOMEM
    assert lib.mp_live_profile(None, P, P, P, None) == EINVAL
    for bad in (dict(n_traces=-1), dict(reserved0=1), dict(max_steps=-2), dict(n_tensors=-1),
                dict(trace_ptr=None), dict(size_bytes=0x6004), dict(alloc_step=0x4002)):
        b = _batch(**bad)
        assert lib.mp_live_profile(ctypes.byref(b), P, P, P, None) == EINVAL, bad
        assert lib.mp_peak(ctypes.byref(b), P, P, P, None) == EINVAL, bad
    b = _batch(profile_ptr=None)
    assert lib.mp_live_profile(ctypes.byref(b), P, P, P, None) == EINVAL
    b = _batch()
    assert lib.mp_live_profile(ctypes.byref(b), None, P, P, None) == EINVAL   # profile output missing
    assert lib.mp_live_profile(ctypes.byref(b), P + 4, P, P, None) == EINVAL  # misaligned int64
    assert lib.mp_plan_greedy_by_size(ctypes.byref(b), 7, P, P, P, P, 1 << 30, None) == EINVAL  # policy
    need = lib.mp_plan_workspace_bytes(ctypes.byref(b))
    assert need > 0
    assert lib.mp_plan_greedy_by_size(ctypes.byref(b), 0, P, P, P, P, need - 1, None) == ENOMEM
    assert lib.mp_plan_greedy_by_size(ctypes.byref(b), 0, P, P, P, None, need, None) == EINVAL
    assert lib.mp_plan_greedy_by_size(ctypes.byref(b), 0, P, P, P, P + 8, need, None) == EINVAL  # alignment
    assert lib.mp_validate_plan(ctypes.byref(b), P, None, P, P, P, 1 << 30, None) == EINVAL
    assert lib.mp_validate_plan(ctypes.byref(b), P, P, P + 2, P, P, 1 << 30, None) == EINVAL


def test_workspace_sizes(lib):
    b = _batch(n_traces=0)
    assert lib.mp_plan_workspace_bytes(ctypes.byref(b)) == 0
    assert lib.mp_validate_workspace_bytes(ctypes.byref(b)) == 0
    small = _batch(n_traces=4096, max_tensors=512, max_steps=1024)
    assert lib.mp_validate_workspace_bytes(ctypes.byref(small)) == 0  # fits shared memory
    big = _batch(n_traces=1, max_tensors=20000, max_steps=10000)
    assert lib.mp_validate_workspace_bytes(ctypes.byref(big)) > 0
    assert lib.mp_plan_workspace_bytes(ctypes.byref(big)) > lib.mp_plan_workspace_bytes(ctypes.byref(_batch(n_traces=1, max_tensors=200, max_steps=100)))


def test_product_path_never_touches_the_oracle():
    pkg = os.path.join(ROOT, "paper_2203_00448_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, fn)).read()
                assert not re.search(r"\bimport\s+oracle\b|\bfrom\s+oracle\b|liboracle|oracle\.h", src), fn


def test_host_argument_errors_of_the_other_strategies(lib):
    """The entry points beyond the hot path reject bad host arguments before
    anything is enqueued (fake device addresses are never dereferenced)."""
    P = 0x10000
    EINVAL, ENOMEM = _lib.EINVAL, _lib.ENOMEM
    b = _batch()
    assert lib.mp_plan_bump(None, P, P, P, None, 0, None) == EINVAL
    assert lib.mp_plan_bump(ctypes.byref(b), None, P, P, None, 0, None) == EINVAL
    assert lib.mp_plan_bump(ctypes.byref(b), P, P + 4, P, None, 0, None) == EINVAL   # misaligned int64
    assert lib.mp_plan_greedy_by_breadth(ctypes.byref(b), 5, P, P, P, None, 0, None) == EINVAL  # policy
    assert lib.mp_plan_greedy_by_breadth(ctypes.byref(b), 0, P, None, P, None, 0, None) == EINVAL
    need = lib.mp_optimal_workspace_bytes(ctypes.byref(b))
    assert need > 0
    assert lib.mp_plan_optimal(ctypes.byref(b), P, P, P, P, need - 1, None) == ENOMEM
    assert lib.mp_plan_optimal(ctypes.byref(b), P, P, P, None, need, None) == EINVAL
    assert lib.mp_slab_layout(None, P, None, None, P, None, None) == EINVAL
    assert lib.mp_slab_layout(ctypes.byref(_batch(n_traces=-1)), P, None, None, P, None, None) == EINVAL
    assert lib.mp_slab_layout(ctypes.byref(b), None, None, None, P, None, None) == EINVAL       # no peaks
    assert lib.mp_slab_layout(ctypes.byref(b), P, P + 2, None, P, None, None) == EINVAL        # misaligned status
    assert lib.mp_slab_layout(ctypes.byref(b), P, None, None, P, P, None) == EINVAL            # addresses, no plan
    assert lib.mp_slab_layout(ctypes.byref(b), P, None, P, P, P + 4, None) == EINVAL           # misaligned addresses
    assert lib.mp_replay_plan(ctypes.byref(b), P, P, None, 64, P, P, P, None, 0, None) == EINVAL  # no slab
    assert lib.mp_replay_plan(ctypes.byref(b), P, P, P, -1, P, P, P, None, 0, None) == EINVAL     # negative size
    assert lib.mp_replay_plan(ctypes.byref(b), P, None, P, 64, P, P, P, None, 0, None) == EINVAL  # no slab bases
    big = _batch(max_tensors=20000, max_steps=10000)
    for fn in ("mp_bump_workspace_bytes", "mp_breadth_workspace_bytes", "mp_replay_workspace_bytes"):
        assert getattr(lib, fn)(ctypes.byref(_batch())) == 0  # small traces: shared memory
        assert getattr(lib, fn)(ctypes.byref(big)) > 0


def test_host_path_argument_errors(lib):
    """mp_plan_and_validate_host checks its host batch, results, chunk count
    and device buffer before any CUDA call (so this runs without a GPU)."""
    import numpy as np

    EINVAL, ENOMEM = _lib.EINVAL, _lib.ENOMEM
    tp = np.array([0, 2, 2, 5], np.int64)
    pp = np.array([0, 4, 4, 10], np.int64)
    st = np.array([4, 0, 6], np.int32)
    a = np.zeros(5, np.int32)
    f = np.ones(5, np.int32)
    s = np.full(5, 64, np.int64)

    def hb(trace_ptr=tp, profile_ptr=pp):
        return _lib.MpBatch(3, 3, 6, 0, 5, 10, trace_ptr.ctypes.data, st.ctypes.data, profile_ptr.ctypes.data,
                            a.ctypes.data, f.ctypes.data, s.ctypes.data)

    outs = [np.zeros(10, np.int64), np.zeros(3, np.int64), np.zeros(5, np.int64), np.zeros(3, np.int64),
            np.zeros(3, np.int32), np.zeros(6, np.int32), np.zeros(3, np.int32)]
    res = _lib.MpHostResults(*(o.ctypes.data for o in outs))
    good = hb()
    need = lib.mp_host_path_bytes(ctypes.byref(good), 2)
    assert need > 0
    assert lib.mp_host_path_bytes(ctypes.byref(good), 0) > 0  # the direct mode: workspace only
    assert lib.mp_host_path_bytes(ctypes.byref(good), -1) == 0
    assert lib.mp_host_path_bytes(ctypes.byref(good), _lib.HOST_PATH_MAX_CHUNKS + 1) == 0
    D = 0x100000  # a fake device address: never dereferenced by a call that fails its checks

    def call(b=good, policy=0, r=res, chunks=2, dbuf=D, dbytes=need):
        return lib.mp_plan_and_validate_host(ctypes.byref(b), policy, ctypes.byref(r) if r is not None else None,
                                             chunks, dbuf, dbytes, None, None, None)

    for bad_tp in (np.array([1, 2, 2, 5], np.int64), np.array([0, 3, 2, 5], np.int64), np.array([0, 2, 2, 4], np.int64)):
        assert call(b=hb(trace_ptr=bad_tp)) == EINVAL
        assert lib.mp_host_path_bytes(ctypes.byref(hb(trace_ptr=bad_tp)), 2) == 0
    assert call(b=hb(profile_ptr=np.array([0, 4, 4, 9], np.int64))) == EINVAL  # does not end at n_steps
    assert call(policy=7) == EINVAL
    assert call(r=None) == EINVAL
    assert call(chunks=-1) == EINVAL
    assert call(chunks=0, dbuf=None) == EINVAL
    assert call(chunks=0, dbytes=0) == ENOMEM
    assert call(dbuf=None) == EINVAL
    assert call(dbuf=D + 8) == EINVAL  # not 256-byte aligned
    assert call(dbytes=need - 1) == ENOMEM
    bad_res = _lib.MpHostResults(*(o.ctypes.data for o in outs))
    bad_res.offsets = outs[2].ctypes.data + 4  # misaligned int64 output
    assert call(r=bad_res) == EINVAL


def test_host_path_sizes_follow_the_chunking(lib):
    """The host path's device buffer holds the batch, its results and the
    planner workspace of the largest chunk: more chunks never need more, one
    chunk needs the whole batch's workspace plus the copies, no chunking (0)
    only that workspace, and an empty batch the same for any chunk count.
    Host-only computation (no GPU)."""
    import numpy as np

    B, n, T = 64, 300, 400  # 300 tensors per trace: the CTA tier's per-trace buffers are sized
    tp = np.arange(B + 1, dtype=np.int64) * n
    pp = np.arange(B + 1, dtype=np.int64) * T
    st = np.full(B, T, np.int32)
    a = np.zeros(B * n, np.int32)
    f = np.ones(B * n, np.int32)
    s = np.full(B * n, 64, np.int64)
    hb = _lib.MpBatch(B, n, T, 0, B * n, B * T, tp.ctypes.data, st.ctypes.data, pp.ctypes.data, a.ctypes.data,
                      f.ctypes.data, s.ctypes.data)
    sizes = [lib.mp_host_path_bytes(ctypes.byref(hb), k) for k in (1, 2, 4, 8, 64)]
    assert all(x > 0 for x in sizes)
    assert all(x >= y for x, y in zip(sizes, sizes[1:]))
    inputs_outputs = (B * n) * 24 + (B * T) * 8  # alloc/free/size in, offsets and profile out
    assert sizes[-1] >= inputs_outputs
    direct = lib.mp_host_path_bytes(ctypes.byref(hb), 0)  # the whole batch's workspace, no copies
    assert 0 < direct < sizes[0] and sizes[0] - direct >= inputs_outputs
    tp0 = np.zeros(1, np.int64)
    empty = _lib.MpBatch(0, 0, 0, 0, 0, 0, tp0.ctypes.data, 0, tp0.ctypes.data, 0, 0, 0)
    assert lib.mp_host_path_bytes(ctypes.byref(empty), 4) == lib.mp_host_path_bytes(ctypes.byref(empty), 1)


def test_workspace_sizes_saturate_instead_of_wrapping(lib):
    """A batch whose planner workspace does not fit in size_t gets SIZE_MAX, so
    no workspace (and not the fixed scratch of the no-allocation entry point)
    can pass the size check; nothing is launched (fake device addresses)."""
    P = 0x10000
    size_max = (1 << 64) - 1
    huge = _batch(n_traces=(1 << 31) - 1, max_tensors=(1 << 28) - 1, max_steps=(1 << 31) - 1)
    assert lib.mp_plan_workspace_bytes(ctypes.byref(huge)) == size_max
    for fn in ("mp_validate_workspace_bytes", "mp_bump_workspace_bytes", "mp_breadth_workspace_bytes",
               "mp_replay_workspace_bytes"):
        assert getattr(lib, fn)(ctypes.byref(huge)) == size_max, fn
    assert lib.mp_plan_greedy_by_size(ctypes.byref(huge), 0, P, P, P, P, 1 << 40, None) == _lib.ENOMEM
    assert lib.mp_plan_greedy_by_size_static(ctypes.byref(huge), 0, P, P, P, None) == _lib.ENOMEM
    assert lib.mp_plan_and_validate(ctypes.byref(huge), 0, None, None, P, P, P, None, P, P, 1 << 40,
                                    None) == _lib.ENOMEM
