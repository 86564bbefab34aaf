"""The live profile, greedy_by_size and the fused call on ragged batches whose
input arrays start off a 16-byte boundary, against the CPU oracle, bit-exact.

The kernels read each trace's first tensors with 16-byte vector loads when the
trace's slices allow it and element by element otherwise.  Ragged trace
lengths put the slices at every 4- and 8-byte phase; here the arrays
themselves also start 4 (alloc, free) or 8 (sizes) bytes past a 16-byte
boundary, and the batch mixes empty traces, traces of one step, traces longer
than the register-held part and traces whose sizes sum past 2^32 (the 64-bit
launch).
"""
import numpy as np
import pytest
import torch

import oracle
import tracegen as tg

from tests.test_gpu_parity import POLICIES

pytestmark = pytest.mark.gpu


def _ragged(seed, n_traces):
    rng = np.random.default_rng(seed)
    traces = []
    for b in range(n_traces):
        kind = b % 11
        if kind == 0:
            traces.append((int(rng.integers(0, 5)), [], [], []))  # empty
            continue
        T = 1 if kind == 1 else int(rng.integers(2, 1500))
        n = int(rng.integers(1, 900)) if kind != 2 else int(rng.integers(600, 1100))
        a = rng.integers(0, T, size=n)
        f = np.minimum(a + 1 + rng.geometric(0.3, size=n), T)
        big = kind == 3
        s = rng.integers(1, 1 << 14, size=n) * (1 << 19 if big else 16)
        traces.append((T, a, f, s))
    return tg.from_arrays(traces)


def _shifted(ts):
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")

    def moved(t):
        big = torch.empty(t.numel() + 1, dtype=t.dtype, device="cuda")
        big[1:].copy_(t)
        return big[1:]

    db.alloc_step, db.free_step, db.size_bytes = moved(db.alloc_step), moved(db.free_step), moved(db.size_bytes)
    assert db.alloc_step.data_ptr() % 16 == 4 and db.size_bytes.data_ptr() % 16 == 8
    return db


@pytest.mark.parametrize("name,pol", POLICIES)
def test_ragged_shifted_profile_plan_and_fused(cuda_lib, name, pol):
    import paper_2203_00448_gb300 as mp

    ts = _ragged(5, 700)
    assert ts.n_tensors % 4 != 0 and (np.diff(ts.trace_ptr) == 0).any()
    o_prof, o_lb, o_st_p = oracle.live_profile(ts)
    o_off, o_pk, o_st_g = oracle.plan_greedy_by_size(ts, pol)
    o_v, o_c, o_st_v = oracle.validate_plan(ts, o_off)
    assert (o_st_p == 0).all() and (o_st_g == 0).all() and (o_v == 1).all()
    # some traces need the 64-bit launch
    sums = np.add.reduceat(ts.size_bytes, ts.trace_ptr[:-1]) * (np.diff(ts.trace_ptr) > 0)
    assert (sums >= 1 << 32).any()
    db = _shifted(ts)
    h = lambda t: t.cpu().numpy()

    prof, lb, st = mp.live_profile(db)
    assert np.array_equal(h(st), o_st_p)
    assert np.array_equal(h(prof), o_prof) and np.array_equal(h(lb), o_lb)

    off, pk, st = mp.plan_greedy_by_size(db, name)
    assert np.array_equal(h(st), o_st_g)
    assert np.array_equal(h(off), o_off) and np.array_equal(h(pk), o_pk)

    res = mp.plan_and_validate(db, name)
    torch.cuda.synchronize()
    assert np.array_equal(h(res.status), o_st_g)
    for k, want in (("profile", o_prof), ("peak_lb", o_lb), ("offsets", o_off), ("plan_peak", o_pk),
                    ("verdict", o_v), ("conflict", o_c)):
        assert np.array_equal(h(getattr(res, k)), want), k
