"""The planner's bounded waits run out cleanly (MP_ETIMEOUT), on the GPU.

A test build of the library (paper_2203_00448_gb300.build.build_test_hooks:
waits bounded at about 8 ms, and the entry point mp_test_plan_hold) keeps one
tensor out of the ready queue, as if the entry announcing it never came.  Its
trace then cannot finish: the workers waiting for that entry give up after the
bound, the call returns, that trace reports MP_ETIMEOUT, the other traces of
the batch are planned exactly as the oracle plans them, and the same library
plans the same batch correctly right after (the context is still usable).
Both waiting places are covered: the ready queue of the per-trace CTA tier
(components with long-lived members), and the queues of the grid-wide planner
(batches of a few traces of more than 1,024 tensors).
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import tracegen as tg

pytestmark = pytest.mark.gpu

ETIMEOUT = 4


@pytest.fixture(scope="module")
def hooks_lib(cuda_lib):
    from paper_2203_00448_gb300 import _lib, build

    lib = ctypes.CDLL(build.build_test_hooks())
    P, BP = ctypes.c_void_p, ctypes.POINTER(_lib.MpBatch)
    lib.mp_test_plan_hold.argtypes = [BP, ctypes.c_int32, P, P, P, P, ctypes.c_size_t, ctypes.c_int32,
                                      ctypes.c_int32, P]
    lib.mp_test_plan_hold.restype = ctypes.c_int32
    return lib


def _plan(lib, ts, policy, hold_trace, hold_pos):
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")
    need = mp.plan_workspace_bytes(db)
    ws = torch.empty(max(need, 256), dtype=torch.uint8, device="cuda")
    off = torch.full((ts.n_tensors,), -7, dtype=torch.int64, device="cuda")
    pk = torch.zeros(ts.n_traces, dtype=torch.int64, device="cuda")
    st = torch.full((ts.n_traces,), -7, dtype=torch.int32, device="cuda")
    s = db.struct()
    rc = lib.mp_test_plan_hold(ctypes.byref(s), policy, off.data_ptr(), pk.data_ptr(), st.data_ptr(), ws.data_ptr(),
                               ws.numel(), hold_trace, hold_pos, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return rc, off.cpu().numpy(), pk.cpu().numpy(), st.cpu().numpy()


def _held_position(ts, b, alloc_step):
    """Alloc-order position of trace b's tensor allocated at alloc_step (the
    only one there, so its position does not depend on the scatter order)."""
    _, a, _, _ = ts.trace(b)
    a = np.asarray(a)
    assert (a == alloc_step).sum() == 1
    return int((a < alloc_step).sum())


def _check(ts, pol, off, pk, st, held):
    o_off, o_pk, o_st = oracle.plan_greedy_by_size(ts, pol)
    assert (o_st == 0).all()
    expect = np.zeros(ts.n_traces, dtype=np.int32)
    if held is not None:
        expect[held] = ETIMEOUT
    assert st.tolist() == expect.tolist()
    for b in range(ts.n_traces):
        if b == held:
            continue
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        assert np.array_equal(off[lo:hi], o_off[lo:hi]), f"offsets of trace {b}"
        assert pk[b] == o_pk[b]


def _cta_tier_batch():
    """Three traces, each one component of 100 short-lived tensors allocated at
    distinct steps 100..199 around five long-lived ones: the CTA tier's runs."""
    rng = np.random.default_rng(3)
    traces = []
    for _ in range(3):
        a = np.concatenate([np.arange(100, 200), np.full(5, 100)])
        f = np.concatenate([np.arange(100, 200) + rng.integers(2, 6, size=100), np.full(5, 300)])
        s = rng.integers(1, 1 << 12, size=105) * 64
        traces.append((400, a, f, s))
    return tg.from_arrays(traces)


def _grid_batch():
    """Three traces of 1,500 tensors (the grid-wide planner), alloc steps
    distinct, with a sprinkle of long-lived tensors."""
    rng = np.random.default_rng(4)
    traces = []
    for _ in range(3):
        n, T = 1500, 2000
        a = np.sort(rng.choice(T - 40, size=n, replace=False))
        life = np.where(rng.random(n) < 0.03, rng.integers(33, 400, size=n), rng.integers(1, 6, size=n))
        f = np.minimum(a + life, T)
        s = rng.integers(1, 1 << 16, size=n) * 16
        traces.append((T, a, f, s))
    return tg.from_arrays(traces)


@pytest.mark.parametrize("pol", (oracle.FIT_FIRST, oracle.FIT_BEST))
def test_cta_tier_wait_runs_out(hooks_lib, pol):
    import paper_2203_00448_gb300 as mp

    ts = _cta_tier_batch()
    p = _held_position(ts, 1, 150)
    rc, off, pk, st = _plan(hooks_lib, ts, pol, 1, p)
    assert rc == mp.OK
    _check(ts, pol, off, pk, st, held=1)
    rc, off, pk, st = _plan(hooks_lib, ts, pol, -1, -1)  # nothing held: the same library, right after
    assert rc == mp.OK
    _check(ts, pol, off, pk, st, held=None)


@pytest.mark.parametrize("pol", (oracle.FIT_FIRST, oracle.FIT_BEST))
def test_grid_wait_runs_out(hooks_lib, pol):
    import paper_2203_00448_gb300 as mp

    ts = _grid_batch()
    assert ts.max_tensors > 1024
    _, a, _, _ = ts.trace(1)
    p = _held_position(ts, 1, int(np.asarray(a)[700]))
    rc, off, pk, st = _plan(hooks_lib, ts, pol, 1, p)
    assert rc == mp.OK
    _check(ts, pol, off, pk, st, held=1)
    rc, off, pk, st = _plan(hooks_lib, ts, pol, -1, -1)
    assert rc == mp.OK
    _check(ts, pol, off, pk, st, held=None)
