"""mp_plan_greedy_by_size_static: the planner for callers that cannot allocate
device memory (its scratch is a fixed array inside libmemplan.so).

It is called straight through the C ABI and must give exactly the offsets,
peaks and statuses of mp_plan_greedy_by_size, on two calls in a row over
different batches (the shared scratch keeps the previous call's bytes), and
must reject a batch whose scratch need exceeds the fixed array without
touching the outputs.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import tracegen as tg

pytestmark = pytest.mark.gpu


def _static_plan(lib, db, policy, sentinel=-7):
    off = torch.full((db.n_tensors,), sentinel, dtype=torch.int64, device="cuda")
    pk = torch.full((db.n_traces,), sentinel, dtype=torch.int64, device="cuda")
    st = torch.full((db.n_traces,), sentinel, dtype=torch.int32, device="cuda")
    s = db.struct()
    rc = lib.mp_plan_greedy_by_size_static(ctypes.byref(s), policy, off.data_ptr() if off.numel() else None,
                                           pk.data_ptr() if pk.numel() else None,
                                           st.data_ptr() if st.numel() else None,
                                           torch.cuda.current_stream().cuda_stream)
    return rc, off, pk, st


def _extreme_batch(seed):
    """Eight traces of up to 1,000 tensors over 60,000 steps with sizes up to
    2^40: the per-trace planner with its working set in the scratch and 64-bit
    bytes, so the first call leaves the scratch full of large values."""
    rng = np.random.default_rng(seed)
    traces = []
    T = 60000
    for k in range(8):
        n = 1000 - 37 * k
        a = np.sort(rng.integers(0, T - 400, size=n))
        busy = rng.integers(0, 3, size=n) == 0
        a[busy] = 30000 + rng.integers(0, 120, size=int(busy.sum()))
        life = np.where(rng.random(n) < 0.1, rng.integers(33, 400, size=n), rng.integers(1, 6, size=n))
        f = np.minimum(a + life, T)
        s = rng.integers(1, 1 << 20, size=n) << 20
        traces.append((T, a, f, s))
    return tg.from_arrays(traces)


def _mid_components(seed):
    """Traces of at most 1,024 tensors whose components of 33 to 300 tensors
    take the CTA tier, with the working set in the scratch (20,000 steps)."""
    rng = np.random.default_rng(seed)
    traces = []
    T = 20000
    for c in (33, 120, 300):
        a1 = np.sort(rng.choice(np.arange(0, 9000), size=600, replace=False))
        f1 = a1 + 1
        a2 = 10000 + rng.integers(0, 10, size=c)
        f2 = 10040 + rng.integers(0, 10, size=c)
        s = rng.integers(1, 1 << 14, size=600 + c) * 64
        traces.append((T, np.concatenate([a1, a2]), np.concatenate([f1, f2]), s))
    return tg.from_arrays(traces)


def test_static_scratch_matches_workspace_entry_point(cuda_lib):
    import paper_2203_00448_gb300 as mp

    lib = cuda_lib
    # Calls in a row share the scratch array, and no call clears it.  The first
    # batch fills it with large values; the next ones must not read any of
    # them: the grid-wide planner on a few large traces (16 seq2seq traces, a
    # 10,000-tensor long-tail trace), the per-trace planner with its data in the
    # scratch (128 seq2seq traces, mid-size components), ragged random traces.
    batches = [_extreme_batch(1), tg.config(4).select(range(16)),
               tg.long_tail(seed=11, n=10000, T=5000, n_long=500, long_hi=2500),
               tg.config(4).select(range(128)), _mid_components(2), tg.random_small(5, 200, 150, 400, 1 << 20),
               _extreme_batch(3)]
    for policy in (mp.FIT_FIRST, mp.FIT_BEST):
        for ts in batches:
            db = mp.DeviceBatch.from_host(ts, "cuda")
            assert 0 < mp.plan_workspace_bytes(db) <= 16 << 20
            rc, off, pk, st = _static_plan(lib, db, policy)
            assert rc == mp.OK, mp.status_string(rc)
            ref_off, ref_pk, ref_st = mp.plan_greedy_by_size(db, policy)
            torch.cuda.synchronize()
            assert torch.equal(st, ref_st) and bool((st == 0).all()), ts.name
            assert torch.equal(off, ref_off), ts.name
            assert torch.equal(pk, ref_pk), ts.name


def test_static_scratch_rejects_oversized_batch(cuda_lib):
    import paper_2203_00448_gb300 as mp

    ts = tg.random_batch(0, 8192, 512, 1024)  # needs 32 MiB of scratch, more than the 16 MiB array
    db = mp.DeviceBatch.from_host(ts, "cuda")
    assert mp.plan_workspace_bytes(db) > 16 << 20
    rc, off, pk, st = _static_plan(cuda_lib, db, mp.FIT_FIRST)
    torch.cuda.synchronize()
    assert rc == mp.ENOMEM
    assert bool((off == -7).all()) and bool((pk == -7).all()) and bool((st == -7).all())
    # a small batch right after still works
    small = mp.DeviceBatch.from_host(tg.config(0), "cuda")
    rc, off, pk, st = _static_plan(cuda_lib, small, mp.FIT_FIRST)
    ref_off, ref_pk, _ = mp.plan_greedy_by_size(small, "first")
    torch.cuda.synchronize()
    assert rc == mp.OK and torch.equal(off, ref_off) and torch.equal(pk, ref_pk)
    assert np.array_equal(st.cpu().numpy(), np.zeros(1, dtype=np.int32))
