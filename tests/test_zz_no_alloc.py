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


def test_static_scratch_matches_workspace_entry_point(cuda_lib):
    import paper_2203_00448_gb300 as mp

    lib = cuda_lib
    # the first 128 seq2seq traces, the long-tail trace, ragged random traces: each fits the 16 MiB array
    batches = [tg.config(4).select(range(128)), tg.config(3), tg.random_small(5, 200, 150, 400, 1 << 20)]
    for policy in (mp.FIT_FIRST, mp.FIT_BEST):
        for ts in batches:  # consecutive calls share the scratch array
            db = mp.DeviceBatch.from_host(ts, "cuda")
            assert mp.plan_workspace_bytes(db) <= 16 << 20
            rc, off, pk, st = _static_plan(lib, db, policy)
            assert rc == mp.OK, mp.status_string(rc)
            ref_off, ref_pk, ref_st = mp.plan_greedy_by_size(db, policy)
            torch.cuda.synchronize()
            assert torch.equal(st, ref_st) and bool((st == 0).all())
            assert torch.equal(off, ref_off)
            assert torch.equal(pk, ref_pk)


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
