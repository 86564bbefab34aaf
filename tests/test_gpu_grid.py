"""The grid-wide dataflow planner (batches of at most 32 traces, some of more
than 1,024 tensors) against the CPU oracle, bit-exact, through the C ABI.

Every tensor of every trace is a node of one dataflow executed by a persistent
grid: these cases cover ragged batches that mix small, large, empty and
failing traces; long-lived tensors with more predecessors than a CTA's shared
region holds (the gather, the FIRST jumps and the BEST sort spill to global
memory); traces where short-lived tensors meet hundreds of long-lived ones; and
the fused entry point (profile, plan, validation) on the same batches.
"""
import numpy as np
import pytest
import torch

import oracle
import tracegen as tg

from tests.test_gpu_parity import POLICIES, assert_parity, gpu_run, oracle_run

pytestmark = pytest.mark.gpu


def _fused(ts, policy):
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")
    assert mp.plan_workspace_bytes(db) > 0
    res = mp.plan_and_validate(db, policy)
    torch.cuda.synchronize()
    h = lambda t: t.cpu().numpy()
    return {k: h(getattr(res, k)) for k in ("profile", "peak_lb", "offsets", "plan_peak", "verdict", "conflict",
                                           "status")}


def _assert_fused(ts, g, o):
    st = o["st"]
    fused_st = np.where(st[0] != 0, st[0], st[1])
    assert np.array_equal(g["status"], fused_st)
    ok = fused_st == 0
    for b in np.nonzero(ok)[0]:
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        assert np.array_equal(g["offsets"][lo:hi], o["offsets"][lo:hi]), f"offsets of trace {b}"
        plo, phi = ts.profile_ptr[b], ts.profile_ptr[b + 1]
        assert np.array_equal(g["profile"][plo:phi], o["profile"][plo:phi]), f"profile of trace {b}"
    for k in ("peak_lb", "plan_peak", "verdict"):
        assert np.array_equal(g[k][ok], o[k][ok]), k
    assert np.array_equal(g["conflict"][ok], o["conflict"][ok])


def _mixed_batch(seed):
    rng = np.random.default_rng(seed)
    small = tg.random_small(seed, 24, 200, 300, 1 << 20)
    traces = [small.trace(b) for b in range(small.n_traces)]
    # one large trace: short lives with a sprinkle of long-lived tensors
    n, T = 2500, 3000
    a = rng.integers(0, T, size=n)
    life = np.where(rng.random(n) < 0.04, rng.integers(33, 900, size=n), 1 + rng.geometric(0.4, size=n) - 1)
    f = np.minimum(a + life, T)
    s = rng.integers(1, 1 << 18, size=n) * 64
    traces.insert(17, (T, a, f, s))
    traces.insert(5, (7, [], [], []))                                   # empty
    traces.insert(9, (0, [], [], []))                                   # no steps
    traces.insert(20, (4, np.array([0, 1]), np.array([2, 5]), np.array([8, 8])))        # free > T: EINVAL
    traces.insert(21, (4, np.array([0, 1]), np.array([2, 3]), np.array([2 ** 62, 2 ** 62])))  # EOVERFLOW
    return tg.from_arrays(traces)


@pytest.mark.parametrize("name,pol", POLICIES)
def test_grid_mixed_batch(cuda_lib, name, pol):
    """Small, large, empty and failing traces in one batch: the whole batch runs
    as one dataflow; every valid trace matches the oracle, both entry points."""
    import paper_2203_00448_gb300 as mp

    ts = _mixed_batch(3)
    assert ts.max_tensors > 1024 and ts.n_traces <= 32
    o = oracle_run(ts, pol)
    assert (o["st"][1] != 0).sum() == 2
    assert_parity(ts, gpu_run(ts, name), o)
    _assert_fused(ts, _fused(ts, name), o)
    # the same batch planned twice in a row gives the same bytes
    db = mp.DeviceBatch.from_host(ts, "cuda")
    a1 = [t.cpu().numpy() for t in mp.plan_greedy_by_size(db, name)]
    a2 = [t.cpu().numpy() for t in mp.plan_greedy_by_size(db, name)]
    assert all(np.array_equal(x, y) for x, y in zip(a1, a2))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_grid_predecessors_beyond_the_shared_region(cuda_lib, name, pol):
    """Long-lived tensors of small size spanning a trace of 14,000 short-lived
    ones: each has more than 12,288 predecessors, more pairs than a CTA's
    shared region holds, so the gather spills to the overflow buffer, FIRST
    jumps over both, and BEST sorts all pairs in global memory.  A second trace
    is a clique of 1,500 long-lived tensors, a dependency chain of CTA items
    as long as the trace."""
    rng = np.random.default_rng(21)
    T = 20000
    n1 = 14000
    a1 = rng.integers(0, T - 3, size=n1)
    f1 = a1 + rng.integers(1, 4, size=n1)
    s1 = rng.integers(1 << 10, 1 << 20, size=n1) * 16
    a2 = np.concatenate([np.zeros(4, dtype=np.int64), rng.integers(0, T - 6000, size=50)])
    f2 = np.concatenate([np.full(4, T), a2[4:] + rng.integers(33, 5000, size=50)])
    s2 = np.concatenate([np.array([16, 32, 48, 64]), rng.integers(1, 1 << 20, size=50) * 16])
    A, F, S = np.concatenate([a1, a2]), np.concatenate([f1, f2]), np.concatenate([s1, s2])
    nc, Tc = 1500, 3000
    ac = rng.integers(0, 1000, size=nc)
    fc = ac + 2000
    sc = rng.integers(1, 1 << 12, size=nc) * 64
    ts = tg.from_arrays([(T, A, F, S), (Tc, ac, fc, sc)])
    order = np.lexsort((np.arange(len(A)), A, -S))
    rank = np.empty(len(A), dtype=np.int64)
    rank[order] = np.arange(len(A))
    preds = max(int(((A < F[i]) & (F > A[i]) & (rank < rank[i])).sum()) for i in range(n1, n1 + 4))
    assert preds > 12288
    o = oracle_run(ts, pol)
    assert_parity(ts, gpu_run(ts, name), o)


@pytest.mark.parametrize("name,pol", POLICIES)
def test_grid_many_long_lived_neighbours(cuda_lib, name, pol):
    """Four traces of 3,000 short-lived tensors, each short one overlapping
    several hundred long-lived ones: those with more predecessors than a warp
    holds (512) become CTA items, the others stay warp items."""
    rng = np.random.default_rng(8)
    traces = []
    for k in range(4):
        n1, T = 3000, 1500
        a1 = rng.integers(0, T - 2, size=n1)
        f1 = a1 + rng.integers(1, 3, size=n1)
        nl = 900
        la = rng.integers(0, 100, size=nl)
        lf = np.minimum(la + rng.integers(1200, 1500, size=nl), T)
        s = rng.integers(1, 1 << 20, size=n1 + nl) * (4 if k % 2 else 64)
        traces.append((T, np.concatenate([a1, la]), np.concatenate([f1, lf]), s))
    ts = tg.from_arrays(traces)
    o = oracle_run(ts, pol)
    assert_parity(ts, gpu_run(ts, name), o)
    _assert_fused(ts, _fused(ts, name), o)


@pytest.mark.parametrize("name,pol", POLICIES)
def test_grid_offsets_past_the_merge_keys(cuda_lib, name, pol):
    """Sizes up to 2^45: offsets pass 2^50, beyond what the merge sort's 64-bit
    keys hold next to a 13-bit pair index, so long-lived tensors fall back to
    sorting (offset, end) records; a second trace of small sizes in the same
    batch takes the merge sort."""
    rng = np.random.default_rng(31)
    traces = []
    for big in (True, False):
        n, T = 1600, 2400
        a = rng.integers(0, T - 50, size=n)
        life = np.where(rng.random(n) < 0.25, rng.integers(40, 1500, size=n), rng.integers(1, 8, size=n))
        f = np.minimum(a + life, T)
        s = rng.integers(1, 1 << 12, size=n) * ((1 << 33) if big else 16)
        traces.append((T, a, f, s))
    ts = tg.from_arrays(traces)
    o = oracle_run(ts, pol)
    assert (o["st"] == 0).all()
    assert int(o["offsets"][: ts.trace_ptr[1]].max()) >= 1 << 50
    assert_parity(ts, gpu_run(ts, name), o)
