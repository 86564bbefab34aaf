"""mp_validate_plan on ragged batches against the CPU oracle, bit-exact.

The kernel loads each trace's first tensors with 16-byte vector loads when the
trace's slices allow it, element loads otherwise, and reads the rest of a long
trace from memory twice.  These cases cover slices at every 4- and 8-byte
phase of a 16-byte boundary (ragged trace lengths), input arrays that
themselves start off a 16-byte boundary, traces longer than the register-held
part, empty traces and failing traces between valid ones, wide (64-bit)
addresses next to narrow ones, and the variant whose working set lives in the
workspace.
"""
import numpy as np
import pytest
import torch

import oracle
import tracegen as tg

pytestmark = pytest.mark.gpu


def _ragged(seed, n_traces, n_max, T_max):
    rng = np.random.default_rng(seed)
    traces = []
    for b in range(n_traces):
        n = int(rng.integers(0, n_max + 1)) if b % 17 else int(rng.integers(n_max, 2 * n_max))
        T = int(rng.integers(1, T_max + 1))
        a = rng.integers(0, T, size=n)
        f = np.minimum(a + 1 + rng.geometric(0.3, size=n), T)
        s = rng.integers(1, 1 << 14, size=n) * 16
        traces.append((T, a, f, s))
    return tg.from_arrays(traces)


def _offsets(ts, seed):
    """The oracle's FIRST plan, with conflicts planted in every third trace, one
    negative offset, and every fifth trace lifted past 2^32 (still valid)."""
    off, _, st = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
    assert (st == 0).all()
    rng = np.random.default_rng(seed)
    off = off.copy()
    tp = ts.trace_ptr
    for b in range(ts.n_traces):
        lo, hi = tp[b], tp[b + 1]
        if hi - lo >= 2 and b % 3 == 1:
            i, j = rng.integers(lo, hi, size=2)
            off[j] = off[i] + int(rng.integers(0, 3)) * 16
        if b % 5 == 2:
            off[lo:hi] += 1 << 33
    nonempty = [b for b in range(ts.n_traces) if tp[b + 1] > tp[b]]
    off[tp[nonempty[7]]] = -16
    return off


def _device(ts, shift):
    """The batch on the device; with shift, every per-tensor array starts one
    element past a fresh allocation (4 or 8 bytes off a 16-byte boundary)."""
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")
    if shift:
        def moved(t):
            big = torch.empty(t.numel() + 1, dtype=t.dtype, device="cuda")
            big[1:].copy_(t)
            return big[1:]

        db.alloc_step, db.free_step, db.size_bytes = moved(db.alloc_step), moved(db.free_step), moved(db.size_bytes)
    return db


def _dev_offsets(off, shift):
    t = torch.as_tensor(off, device="cuda")
    if not shift:
        return t
    big = torch.empty(t.numel() + 3, dtype=t.dtype, device="cuda")
    big[3:].copy_(t)
    return big[3:]


@pytest.mark.parametrize("shift", (False, True))
def test_validator_staged_ragged(cuda_lib, shift):
    import paper_2203_00448_gb300 as mp

    ts = _ragged(11, 3001, 600, 1200)
    assert ts.n_tensors % 4 != 0
    off = _offsets(ts, 12)
    ov, oc, ost = oracle.validate_plan(ts, off)
    assert (ost == 2).sum() == 0 and (ost == 1).sum() == 1 and (ov[ost == 0] == 0).sum() > 500
    db = _device(ts, shift)
    v, c, st = mp.validate_plan(db, _dev_offsets(off, shift))
    torch.cuda.synchronize()
    assert np.array_equal(st.cpu().numpy(), ost)
    okm = ost == 0
    assert np.array_equal(v.cpu().numpy()[okm], ov[okm])
    assert np.array_equal(c.cpu().numpy()[okm], oc[okm])


def test_validator_staged_failing_traces(cuda_lib):
    """Invalid tensors, end overflow and a broken CSR entry between valid traces."""
    import paper_2203_00448_gb300 as mp

    ts = _ragged(5, 700, 300, 500)
    off = _offsets(ts, 6)
    tp = ts.trace_ptr
    a = ts.alloc_step.copy()
    nonempty = [b for b in range(ts.n_traces) if tp[b + 1] - tp[b] >= 2]
    a[tp[nonempty[3]] + 1] = -1                       # EINVAL
    off[tp[nonempty[9]] + 1] = 2 ** 63 - 8             # EOVERFLOW
    ts = tg.TraceSet(ts.trace_ptr, ts.steps, ts.profile_ptr, a, ts.free_step, ts.size_bytes)
    ov, oc, ost = oracle.validate_plan(ts, off)
    db = mp.DeviceBatch.from_host(ts, "cuda")
    db.steps[nonempty[20]] = ts.max_steps + 1          # T past max_steps: EINVAL for that trace
    v, c, st = mp.validate_plan(db, torch.as_tensor(off, device="cuda"))
    torch.cuda.synchronize()
    ost = ost.copy()
    ost[nonempty[20]] = 1
    assert ost[nonempty[3]] == 1 and ost[nonempty[9]] == 2
    assert np.array_equal(st.cpu().numpy(), ost)
    okm = ost == 0
    assert np.array_equal(v.cpu().numpy()[okm], ov[okm])
    assert np.array_equal(c.cpu().numpy()[okm], oc[okm])


def test_validator_workspace_variant_staged(cuda_lib):
    """A trace too large for shared memory (the working set in the workspace)
    among small ones: the stage still carries every trace's first tensors."""
    import paper_2203_00448_gb300 as mp

    small = _ragged(9, 300, 200, 300)
    traces = [small.trace(b) for b in range(small.n_traces)]
    rng = np.random.default_rng(2)
    n, T = 9001, 4000
    a = rng.integers(0, T - 1, size=n)
    f = np.minimum(a + 1 + rng.geometric(0.3, size=n), T)
    traces.insert(100, (T, a, f, rng.integers(1, 1 << 10, size=n) * 16))
    ts = tg.from_arrays(traces)
    off = _offsets(ts, 4)
    db = mp.DeviceBatch.from_host(ts, "cuda")
    assert mp.validate_workspace_bytes(db) > 0
    v, c, st = mp.validate_plan(db, torch.as_tensor(off, device="cuda"))
    torch.cuda.synchronize()
    ov, oc, ost = oracle.validate_plan(ts, off)
    assert np.array_equal(st.cpu().numpy(), ost)
    okm = ost == 0
    assert np.array_equal(v.cpu().numpy()[okm], ov[okm])
    assert np.array_equal(c.cpu().numpy()[okm], oc[okm])
