"""GPU path vs CPU oracle, bit-exact (all integer work: tolerance 0).

Every call goes through the C ABI (libmemplan.so) via the package binding.
Covers the five workloads at full size in the launch configuration the bench
uses, random ragged batches, shapes that force each placement tier and the
workspace (global-memory) variants, empty traces, planted plan conflicts and
every per-trace error code.
"""
import functools

import numpy as np
import pytest
import torch

import oracle
import tracegen as tg

pytestmark = pytest.mark.gpu

POLICIES = (("first", oracle.FIT_FIRST), ("best", oracle.FIT_BEST))


def gpu_run(ts, policy):
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")
    res = mp.run_path(db, policy)
    pk2, st_pk = mp.peak(db, res.offsets)
    torch.cuda.synchronize()
    h = lambda t: t.cpu().numpy()
    return dict(profile=h(res.profile), peak_lb=h(res.peak_lb), offsets=h(res.offsets), plan_peak=h(res.plan_peak),
                verdict=h(res.verdict), conflict=h(res.conflict), st=h(res.status), peak=h(pk2), st_peak=h(st_pk))


def oracle_run(ts, pol):
    prof, lb, st_p = oracle.live_profile(ts)
    off, pk, st_g = oracle.plan_greedy_by_size(ts, pol)
    v, c, st_v = oracle.validate_plan(ts, off)
    pk2, st_pk = oracle.peak(ts, off)
    return dict(profile=prof, peak_lb=lb, offsets=off, plan_peak=pk, verdict=v, conflict=c,
                st=np.stack([st_p, st_g, st_v]), peak=pk2, st_peak=st_pk)


@functools.lru_cache(maxsize=None)
def config_oracle(k, pol):
    return oracle_run(tg.config(k), pol)


def assert_parity(ts, g, o):
    assert np.array_equal(g["st"], o["st"]), "trace status differs"
    ok = (o["st"] == 0).all(axis=0)
    prof_ok = o["st"][0] == 0
    for b in np.nonzero(prof_ok)[0]:
        lo, hi = ts.profile_ptr[b], ts.profile_ptr[b + 1]
        assert np.array_equal(g["profile"][lo:hi], o["profile"][lo:hi]), f"profile of trace {b}"
    assert np.array_equal(g["peak_lb"][prof_ok], o["peak_lb"][prof_ok])
    plan_ok = o["st"][1] == 0
    for b in np.nonzero(plan_ok)[0]:
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        assert np.array_equal(g["offsets"][lo:hi], o["offsets"][lo:hi]), f"offsets of trace {b}"
    assert np.array_equal(g["plan_peak"][plan_ok], o["plan_peak"][plan_ok])
    assert np.array_equal(g["verdict"][ok], o["verdict"][ok])
    assert np.array_equal(g["conflict"][ok], o["conflict"][ok])
    assert np.array_equal(g["st_peak"], o["st_peak"])
    assert np.array_equal(g["peak"][ok], o["peak"][ok])


@pytest.mark.parametrize("name,pol", POLICIES)
@pytest.mark.parametrize("k", range(5))
def test_workload_parity(cuda_lib, k, name, pol):
    ts = tg.config(k)
    g = gpu_run(ts, name)
    o = config_oracle(k, pol)
    assert (o["st"] == 0).all() and (o["verdict"] == 1).all()
    assert_parity(ts, g, o)


def test_determinism(cuda_lib):
    ts = tg.config(4)
    a, b = gpu_run(ts, "best"), gpu_run(ts, "best")
    for key in a:
        assert np.array_equal(a[key], b[key]), key


@pytest.mark.parametrize("name,pol", POLICIES)
def test_random_ragged_batches(cuda_lib, name, pol):
    for seed, n_max, T_max, smax in ((1, 40, 30, 64), (2, 200, 300, 1 << 20), (3, 120, 12, 8), (4, 300, 2000, 1 << 30)):
        ts = tg.random_small(seed, 300, n_max, T_max, smax)
        assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_all_tiers_shared_memory_path(cuda_lib, name, pol):
    """Cliques and long-lived tensors: predecessor counts from 0 to ~n cover the
    thread, warp and CTA placement tiers inside one CTA."""
    rng = np.random.default_rng(100)
    traces = []
    for n in (1, 9, 33, 64, 150, 200):
        T = 50
        a = rng.integers(0, 10, size=n)
        f = rng.integers(40, 51, size=n)
        s = rng.integers(1, 4, size=n) * 64  # many equal sizes: exercises the tie-break
        traces.append((T, a, f, s))
        a2 = rng.integers(0, T, size=n)
        f2 = np.minimum(a2 + rng.integers(1, 60, size=n), T)
        traces.append((T, a2, f2, rng.integers(1, 5000, size=n)))
    ts = tg.from_arrays(traces)
    assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_global_memory_path(cuda_lib, name, pol):
    """A trace too large for shared memory runs on the workspace variant; the
    long tensors spanning ~17,000 short ones exceed the warp enumeration limit."""
    rng = np.random.default_rng(7)
    n_short, T = 17000, 9000
    a = rng.integers(0, T, size=n_short)
    f = np.minimum(a + 1 + rng.geometric(0.5, size=n_short) - 1, T)
    s = rng.integers(1, 1 << 16, size=n_short)
    la = np.array([0, 0, 100, 4000]); lf = np.array([T, T, 8000, 8999])
    ls = np.array([1 << 20, 64, 5000, 70000])
    ts = tg.from_arrays([(T, np.concatenate([a, la]), np.concatenate([f, lf]), np.concatenate([s, ls]))])
    assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


def test_long_horizon_global_variants(cuda_lib):
    """Traces of 40,000 steps: the profile's difference array no longer fits in
    shared memory (it is built and scanned in the output slice itself) and the
    validator's working set moves to the workspace; a short trace rides along."""
    rng = np.random.default_rng(17)
    T, n = 40000, 3000
    a = rng.integers(0, T, size=n)
    f = np.minimum(a + 1 + rng.geometric(0.01, size=n), T)
    s = rng.integers(1, 1 << 24, size=n) * 64
    ts = tg.from_arrays([(T, a, f, s), tg.config(0).trace(0), (T, a[:50], f[:50], s[:50] << 20)])
    assert_parity(ts, gpu_run(ts, "first"), oracle_run(ts, oracle.FIT_FIRST))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_long_lived_chain_workspace_path(cuda_lib, name, pol):
    """One component of 14,000 tensors that all live longer than 32 steps, on
    the workspace variant: the long-lived list is too long to stage in shared
    memory, and every member is placed by the whole CTA.  A second trace
    mixes short-lived members with about 200 long-lived ones around them, so
    that short-lived members gather more than 128 predecessors."""
    rng = np.random.default_rng(11)
    n = 14000
    a = np.arange(n) // 2
    T = int(a[-1]) + 80
    f = np.minimum(a + rng.integers(33, 70, size=n), T)
    s = rng.integers(1, 1 << 12, size=n) * 64
    n2, T2 = 3000, 1200
    a2 = rng.integers(0, T2, size=n2)
    f2 = np.minimum(a2 + rng.integers(1, 4, size=n2), T2)
    la = rng.integers(0, 100, size=200)
    lf = np.minimum(la + rng.integers(900, 1200, size=200), T2)
    s2 = rng.integers(1, 1 << 10, size=n2 + 200) * 4
    ts = tg.from_arrays([(T, a, f, s), (T2, np.concatenate([a2, la]), np.concatenate([f2, lf]), s2)])
    assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_mid_size_component_workspace_path(cuda_lib, name, pol):
    """A batch too large for shared memory whose traces hold components of 33
    to 256 tensors (placed by the CTA tier) among thousands of single ones."""
    rng = np.random.default_rng(5)
    traces = []
    for c in (33, 100, 256):
        n1, T = 13000, 16000
        a1 = np.sort(rng.choice(T - 200, size=n1, replace=False))
        a1 = a1[(a1 < 5000) | (a1 >= 5100)]  # keep clear of the block below
        f1 = a1 + 1
        a2 = 5000 + rng.integers(0, 10, size=c)
        f2 = 5040 + rng.integers(0, 10, size=c)
        s = rng.integers(1, 1 << 14, size=len(a1) + c) * 64
        traces.append((T, np.concatenate([a1, a2]), np.concatenate([f1, f2]), s))
    ts = tg.from_arrays(traces)
    assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_one_cta_per_trace_workspace_variants(cuda_lib, name, pol):
    """Traces of at most 1,024 tensors over 60,000 steps: one CTA per trace,
    with the working set in the workspace (too large for shared memory).  Sizes
    summing below and above 2^32 take the 32-bit and the 64-bit launch; each
    trace holds components of 33 to 700 tensors with long-lived members, so the
    CTA tier runs on both."""
    import paper_2203_00448_gb300 as mp

    rng = np.random.default_rng(40)
    T = 60000
    traces = []
    for n, scale in ((1000, 64), (1024, 1 << 26), (700, 4), (300, 1 << 30)):
        a = np.sort(rng.integers(0, T - 400, size=n))
        comp = rng.integers(0, 4, size=n) == 0  # a quarter of them crowd into one busy stretch
        a[comp] = 20000 + rng.integers(0, 200, size=int(comp.sum()))
        life = np.where(rng.random(n) < 0.1, rng.integers(33, 300, size=n), rng.integers(1, 6, size=n))
        f = np.minimum(a + life, T)
        s = rng.integers(1, 1 << 10, size=n) * scale
        traces.append((T, a, f, s))
    ts = tg.from_arrays(traces)
    db = mp.DeviceBatch.from_host(ts, "cuda")
    assert ts.max_tensors <= 1024 and mp.plan_workspace_bytes(db) > 0
    assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


def test_empty_and_degenerate(cuda_lib):
    ts = tg.from_tuples([(0, []), (5, []), (1, [(0, 1, 1)]), (3, [(0, 3, 7), (0, 3, 7), (1, 2, 7)]),
                         (4, [(0, 4, 2 ** 40), (0, 4, 2 ** 40)])])
    for name, pol in POLICIES:
        assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))


def test_zero_traces(cuda_lib):
    import paper_2203_00448_gb300 as mp

    ts = tg.from_tuples([])
    db = mp.DeviceBatch.from_host(ts, "cuda")
    res = mp.run_path(db, "first")
    torch.cuda.synchronize()
    assert res.offsets.numel() == 0 and res.verdict.numel() == 0


def test_error_codes(cuda_lib):
    traces = [
        (4, [(-1, 2, 8)]),                       # alloc < 0
        (4, [(2, 2, 8)]),                        # free <= alloc
        (4, [(1, 5, 8)]),                        # free > T
        (4, [(0, 1, 0)]),                        # size <= 0
        (4, [(0, 1, 2 ** 62), (0, 2, 2 ** 62)]),  # sizes overflow int64
        (4, [(0, 1, 2 ** 62), (0, 1, -5)]),       # EINVAL wins
        (6, [(0, 3, 64), (1, 4, 32)]),           # fine
    ]
    ts = tg.from_tuples(traces)
    for name, pol in POLICIES:
        g, o = gpu_run(ts, name), oracle_run(ts, pol)
        assert o["st"][1].tolist() == [1, 1, 1, 1, 2, 1, 0]
        assert_parity(ts, g, o)


def test_validator_error_codes(cuda_lib):
    """The validator's own status codes: offsets past INT64_MAX - size, size sums past INT64_MAX,
    negative offsets, and EINVAL winning over EOVERFLOW, each beside a valid trace."""
    import paper_2203_00448_gb300 as mp

    big = 2 ** 62
    traces = [
        (4, [(0, 2, 64), (1, 3, 64)]),                      # valid, no conflict
        (4, [(0, 2, 64), (1, 3, 64)]),                      # end past INT64_MAX
        (4, [(0, 1, big), (0, 2, big), (1, 3, 64)]),         # sizes sum past INT64_MAX
        (4, [(0, 2, 64), (1, 3, 64)]),                      # negative offset
        (4, [(0, 2, 64), (1, 3, 64), (2, 4, 64)]),          # end past INT64_MAX and an invalid offset
        (4, [(0, 2, 64), (1, 3, 64)]),                      # address clash
    ]
    ts = tg.from_tuples(traces)
    off = np.zeros(ts.n_tensors, dtype=np.int64)
    tp = ts.trace_ptr
    off[tp[0] + 1] = 64
    off[tp[1] + 1] = 2 ** 63 - 1 - 32
    off[tp[2] + 1] = 2 ** 62
    off[tp[3] + 1] = -64
    off[tp[4] + 1] = 2 ** 63 - 1
    off[tp[4] + 2] = -1
    off[tp[5] + 1] = 32
    db = mp.DeviceBatch.from_host(ts, "cuda")
    v, c, st = mp.validate_plan(db, torch.as_tensor(off, device="cuda"))
    ov, oc, ost = oracle.validate_plan(ts, off)
    assert ost.tolist() == [0, 2, 2, 1, 1, 0]
    assert np.array_equal(st.cpu().numpy(), ost)
    okm = ost == 0
    assert np.array_equal(v.cpu().numpy()[okm], ov[okm]) and ov[okm].tolist() == [1, 0]
    assert np.array_equal(c.cpu().numpy()[okm], oc[okm])


def test_declared_bounds_and_csr_checked(cuda_lib):
    """Traces breaking the host-declared bounds or the CSR are rejected per trace."""
    import paper_2203_00448_gb300 as mp

    ts = tg.from_tuples([(4, [(0, 2, 8), (1, 3, 8), (0, 4, 8)]), (3, [(0, 3, 5)])])
    db = mp.DeviceBatch.from_host(ts, "cuda")
    db.max_tensors = 2  # trace 0 has 3 tensors
    _, _, st = mp.plan_greedy_by_size(db)
    _, _, st2 = mp.validate_plan(db, torch.zeros(ts.n_tensors, dtype=torch.int64, device="cuda"))
    assert st.tolist() == [1, 0] and st2.tolist() == [1, 0]
    db = mp.DeviceBatch.from_host(ts, "cuda")
    db.max_steps = 3
    _, _, st = mp.live_profile(db)
    assert st.tolist() == [1, 0]
    db = mp.DeviceBatch.from_host(ts, "cuda")
    db.profile_ptr[1] = 3  # trace 0 claims 3 profile entries but T = 4
    _, _, st = mp.live_profile(db)
    assert st.tolist() == [1, 1]
    db = mp.DeviceBatch.from_host(ts, "cuda")
    db.trace_ptr[1] = 5  # beyond n_tensors = 4
    _, _, st = mp.plan_greedy_by_size(db)
    assert st.tolist() == [1, 1]


def test_validator_on_planted_conflicts(cuda_lib):
    import paper_2203_00448_gb300 as mp

    ts = tg.config(2).select(range(0, 4096, 8))
    off, _, _ = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
    rng = np.random.default_rng(3)
    bad = off.copy()
    for b in range(ts.n_traces):
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        if b % 3 == 0:
            continue  # leave some traces valid
        i, j = rng.integers(lo, hi, size=2)
        bad[j] = bad[i] + (rng.integers(0, 3) * 64)
    bad[ts.trace_ptr[5]] = -64  # one trace with a negative offset
    db = mp.DeviceBatch.from_host(ts, "cuda")
    v, c, st = mp.validate_plan(db, torch.as_tensor(bad, device="cuda"))
    pk, st_pk = mp.peak(db, torch.as_tensor(bad, device="cuda"))
    ov, oc, ost = oracle.validate_plan(ts, bad)
    opk, opst = oracle.peak(ts, bad)
    assert np.array_equal(st.cpu().numpy(), ost) and np.array_equal(st_pk.cpu().numpy(), opst)
    okm = ost == 0
    assert np.array_equal(v.cpu().numpy()[okm], ov[okm])
    assert np.array_equal(c.cpu().numpy()[okm], oc[okm])
    assert np.array_equal(pk.cpu().numpy()[okm], opk[okm])
    assert (ov[okm] == 0).sum() > 100


def test_generator_and_oracle_stable_on_this_host(cuda_lib):
    """The committed oracle summaries reproduce on the GPU host (its CPU may be
    another architecture), so the parity above compares like with like."""
    import json
    import os

    ref = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "config_summaries.json")))
    for k in (0, 1, 2):
        c = ref["configs"][k]
        ts = tg.config(k)
        assert tg.digest(ts) == c["sha256"]
        o = config_oracle(k, oracle.FIT_FIRST)
        assert int(o["offsets"].sum()) == c["first_offsets_sum"]
        assert int(o["plan_peak"].sum()) == c["first_plan_peak_sum"]


# ------------------------------------------------------------- fused entry point

def fused_run(ts, policy, profile=True):
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")
    res = mp.plan_and_validate(db, policy, profile=profile)
    torch.cuda.synchronize()
    h = lambda t: t.cpu().numpy()
    return dict(profile=h(res.profile), peak_lb=h(res.peak_lb), offsets=h(res.offsets), plan_peak=h(res.plan_peak),
                verdict=h(res.verdict), conflict=h(res.conflict), st=h(res.status))


def assert_fused_parity(ts, g, o, profile=True):
    st_expect = o["st"].max(axis=0)  # a trace's one status: its error, if any stage reports one
    assert np.array_equal(g["st"], st_expect), "trace status differs"
    ok = st_expect == 0
    for b in np.nonzero(ok)[0]:
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        assert np.array_equal(g["offsets"][lo:hi], o["offsets"][lo:hi]), f"offsets of trace {b}"
        if profile:
            plo, phi = ts.profile_ptr[b], ts.profile_ptr[b + 1]
            assert np.array_equal(g["profile"][plo:phi], o["profile"][plo:phi]), f"profile of trace {b}"
    for k in ("plan_peak", "verdict") + (("peak_lb",) if profile else ()):
        assert np.array_equal(g[k][ok], o[k][ok]), k
    assert np.array_equal(g["conflict"][ok], o["conflict"][ok])
    assert (g["verdict"][ok] == 1).all()


@pytest.mark.parametrize("name,pol", POLICIES)
@pytest.mark.parametrize("k", range(5))
def test_fused_workload_parity(cuda_lib, k, name, pol):
    ts = tg.config(k)
    assert_fused_parity(ts, fused_run(ts, name), config_oracle(k, pol))


@pytest.mark.parametrize("name,pol", POLICIES)
def test_fused_random_and_errors(cuda_lib, name, pol):
    for ts in (tg.random_small(11, 300, 120, 200, 1 << 20), tg.random_small(12, 100, 300, 2000, 1 << 30),
               tg.from_tuples([(4, [(-1, 2, 8)]), (4, [(0, 1, 2 ** 62), (0, 2, 2 ** 62)]), (0, []), (5, []),
                               (6, [(0, 3, 64), (1, 4, 32), (3, 6, 8)])])):
        assert_fused_parity(ts, fused_run(ts, name), oracle_run(ts, pol))


def test_fused_without_profile(cuda_lib):
    ts = tg.config(2).select(range(0, 4096, 16))
    o = oracle_run(ts, oracle.FIT_FIRST)
    assert_fused_parity(ts, fused_run(ts, "first", profile=False), o, profile=False)


def test_byte_width_boundary_and_mixed_batches(cuda_lib):
    """Traces whose sizes sum just below, at and above 2^32 (the kernel switches
    from 32-bit to 64-bit byte arithmetic there), interleaved with small ones in
    one call, through both entry points."""
    T, a, f, s = tg.config(0).trace(0)
    traces = []
    for target in (2 ** 32 - 1, 2 ** 32, 2 ** 32 + 1, 2 ** 33 + 12345):
        s2 = np.asarray(s, dtype=np.int64).copy()
        s2[0] += target - int(s2.sum())
        traces += [(T, a, f, s2), tg.config(0).trace(0)]
    ts = tg.from_arrays(traces)
    for name, pol in POLICIES:
        o = oracle_run(ts, pol)
        assert (o["st"] == 0).all()
        assert_parity(ts, gpu_run(ts, name), o)
        assert_fused_parity(ts, fused_run(ts, name), o)


# ------------------------------------------------------------- bump_allocation

def assert_bump_parity(ts):
    import paper_2203_00448_gb300 as mp

    db = mp.DeviceBatch.from_host(ts, "cuda")
    off, pk, st = mp.plan_bump(db)
    torch.cuda.synchronize()
    o_off, o_pk, o_st = oracle.plan_bump(ts)
    st, pk, off = st.cpu().numpy(), pk.cpu().numpy(), off.cpu().numpy()
    assert np.array_equal(st, o_st), "trace status differs"
    assert np.array_equal(pk, o_pk), "plan_peak differs"
    for b in np.nonzero(o_st == 0)[0]:
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        assert np.array_equal(off[lo:hi], o_off[lo:hi]), f"offsets of trace {b}"


@pytest.mark.parametrize("k", range(5))
def test_bump_workload_parity(cuda_lib, k):
    assert_bump_parity(tg.config(k))  # the long-tail trace keeps its working set in the workspace


def test_bump_buckets_errors_and_ragged(cuda_lib):
    rng = np.random.default_rng(3)
    same_step = (50, np.zeros(300, np.int64), rng.integers(1, 51, 300), rng.integers(1, 1 << 20, 300))
    for ts in (tg.random_small(21, 300, 120, 200, 1 << 20), tg.from_arrays([same_step, same_step]),
               tg.from_tuples([(4, [(-1, 2, 8)]), (4, [(0, 1, 2 ** 62), (0, 2, 2 ** 62)]), (0, []), (5, []),
                               (6, [(0, 3, 64), (1, 4, 32), (3, 6, 8), (1, 2, 16)])])):
        assert_bump_parity(ts)


# ------------------------------------------------------------- exact optimum (small traces)

def test_optimal_matches_oracle_brute_force(cuda_lib):
    """mp_plan_optimal against the oracle's exhaustive search: the optimum and
    the offsets of the first optimal order, on traces of 0..10 tensors with
    few distinct sizes (many ties); lb <= opt <= greedy; more than 10 tensors
    and invalid traces get their status codes."""
    import paper_2203_00448_gb300 as mp

    rng = np.random.default_rng(5)
    traces = []
    for n in (0, 1, 2, 3, 4, 5, 6, 7, 8, 8, 9, 9, 10, 6, 7):
        T = int(rng.integers(1, 10))
        a = rng.integers(0, T, n)
        f = np.minimum(a + rng.integers(1, 5, n), T)
        s = rng.integers(1, 5, n) * 64
        traces.append((T, a, f, s))
    big = traces[12]
    traces += [(5, np.zeros(11, np.int64), np.full(11, 5), np.full(11, 8)),  # 11 tensors: beyond the search
               (4, np.array([0, 2]), np.array([3, 1]), np.array([8, 8]))]     # free <= alloc
    ts = tg.from_arrays(traces)
    db = mp.DeviceBatch.from_host(ts, "cuda")
    off, pk, st = mp.plan_optimal(db)
    g_off, g_pk, g_st = mp.plan_greedy_by_size(db, "first")
    torch.cuda.synchronize()
    off, pk, st, g_pk = off.cpu().numpy(), pk.cpu().numpy(), st.cpu().numpy(), g_pk.cpu().numpy()
    _, lb, _ = oracle.live_profile(ts)
    assert list(st[-2:]) == [oracle.EINVAL, oracle.EINVAL]
    for b in range(ts.n_traces - 2):
        T, a, f, s = ts.trace(b)
        assert st[b] == 0
        opt, o_off = oracle.bruteforce_opt(a, f, s)
        lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
        assert pk[b] == opt, f"trace {b}"
        assert np.array_equal(off[lo:hi], o_off), f"offsets of trace {b}"
        assert lb[b] <= opt <= g_pk[b]
    assert len(big[1]) == 10


# ------------------------------------------------------------- plans replayed on device memory

def test_replay_on_device_slabs(cuda_lib):
    """Plans materialised on one device buffer (a slab per trace) and replayed:
    greedy and bump plans replay cleanly; plans with a planted address clash
    between lifetime-overlapping tensors fail exactly where the validator says
    so; a tensor outside its slab is rejected before anything is written."""
    import paper_2203_00448_gb300 as mp

    ts = tg.from_arrays([tg.config(0).trace(0), tg.config(1).trace(0)] +
                        [tg.config(2).trace(b) for b in range(0, 4096, 128)] +
                        [tg.random_small(31, 1, 60, 40, 1 << 12).trace(0), (3, [], [], [])])
    db = mp.DeviceBatch.from_host(ts, "cuda")
    counts = np.diff(ts.trace_ptr)
    for plan, ref in ((lambda: mp.plan_greedy_by_size(db, "first"), lambda: oracle.plan_greedy_by_size(ts, 0)),
                      (lambda: mp.plan_greedy_by_size(db, "best"), lambda: oracle.plan_greedy_by_size(ts, 1)),
                      (lambda: mp.plan_bump(db), lambda: oracle.plan_bump(ts))):
        off, pk, st = plan()
        slab, base, where = mp.materialize(db, off, pk, st)
        ok, first_bad, rst = mp.replay_plan(db, off, base, slab)
        torch.cuda.synchronize()
        assert bool((rst == 0).all()) and bool((ok == 1).all()) and bool((first_bad == -1).all())
        assert int(base[-1]) >= int(pk.sum())
        # the library's tensor addresses: each trace's slab base plus the oracle's offset
        o_off, o_pk, _ = ref()
        hb = base.cpu().numpy()
        sizes = (o_pk + mp.SLAB_ALIGN - 1) // mp.SLAB_ALIGN * mp.SLAB_ALIGN
        assert np.array_equal(hb, np.concatenate([[0], np.cumsum(sizes)]))
        assert np.array_equal(where.cpu().numpy(), np.repeat(hb[:-1], counts) + o_off)

    # planted clashes: in every other trace, one tensor moved onto a lifetime-overlapping one
    off, _, _ = mp.plan_greedy_by_size(db, "first")
    h = off.cpu().numpy().copy()
    rng = np.random.default_rng(9)
    for b in range(0, ts.n_traces, 2):
        T, a, f, s = ts.trace(b)
        pairs = [(i, j) for i in range(len(a)) for j in range(len(a)) if i != j and a[i] < f[j] and a[j] < f[i]]
        if pairs:
            i, j = pairs[int(rng.integers(len(pairs)))]
            h[ts.trace_ptr[b] + j] = h[ts.trace_ptr[b] + i]
    bad_off = torch.from_numpy(h).cuda()
    pk2, st2 = mp.peak(db, bad_off)
    # a failed trace gets an empty slab and address -1 for its tensors
    fst = torch.zeros_like(st2)
    fst[1] = oracle.EINVAL
    _, fbase, fwhere = mp.materialize(db, bad_off, pk2, fst)
    hb, hw = fbase.cpu().numpy(), fwhere.cpu().numpy()
    assert hb[2] == hb[1] and (hw[ts.trace_ptr[1]:ts.trace_ptr[2]] == -1).all()
    assert np.array_equal(hw[ts.trace_ptr[2]:], np.repeat(hb[2:-1], counts[2:]) + h[ts.trace_ptr[2]:])
    verdict, _, vst = mp.validate_plan(db, bad_off)
    slab, base, _ = mp.materialize(db, bad_off, pk2, st2)
    ok, first_bad, rst = mp.replay_plan(db, bad_off, base, slab)
    torch.cuda.synchronize()
    assert bool((rst == 0).all()) and bool((vst == 0).all())
    assert torch.equal(ok, verdict)
    assert int((verdict == 0).sum()) >= 10
    fb = first_bad.cpu().numpy()
    assert all((fb[b] >= 0) == (int(verdict[b]) == 0) for b in range(ts.n_traces))

    # a tensor past its trace's slab, and a buffer too small for the last slabs
    off, pk, st = mp.plan_greedy_by_size(db, "first")
    slab, base, _ = mp.materialize(db, off, pk, st)
    h = off.cpu().numpy().copy()
    h[ts.trace_ptr[1]] = int(pk[1]) + 1
    ok, _, rst = mp.replay_plan(db, torch.from_numpy(h).cuda(), base, slab)
    short = slab[: int(base[3])]
    ok2, _, rst2 = mp.replay_plan(db, off, base, short)
    torch.cuda.synchronize()
    assert int(rst[1]) == oracle.EINVAL and int(ok[1]) == 0 and bool((rst[2:] == 0).all())
    r2 = rst2.cpu().numpy()
    assert (r2[:3] == 0).all() and (r2[3:][np.diff(base.cpu().numpy())[3:] > 0] == oracle.EINVAL).all()


# ------------------------------------------------------------- end to end from host memory

def test_host_path_matches_the_device_path(cuda_lib):
    """HostPath (mp_plan_and_validate_host: pinned host buffers, chunked copies
    overlapping the planning, or none with the kernels reading and writing the
    pinned buffers directly) gives the fused call's results for every chunk
    count, also for a second batch of the same shape staged into the same
    buffers, and with empty, failing and more-chunks-than-traces cases."""
    import paper_2203_00448_gb300 as mp

    cases = ((tg.config(2).select(range(0, 4096, 8)), tg.config(2).select(range(1, 4096, 8))),
             (tg.random_small(41, 97, 120, 200, 1 << 30),),
             (tg.from_tuples([(4, [(-1, 2, 8)]), (0, []), (6, [(0, 3, 64), (1, 4, 32), (3, 6, 8)]), (5, [])]),))
    for batches in cases:
        for chunks in (0, 1, 3, 8):
            hp = mp.HostPath(batches[0], "cuda", "first", chunks=chunks)
            for ts in batches:
                ref = fused_run(ts, "first")
                out = hp.run(ts)
                ok = ref["st"] == 0
                assert np.array_equal(out["status"], ref["st"])
                for k, ptr in (("offsets", ts.trace_ptr), ("profile", ts.profile_ptr)):
                    for b in np.nonzero(ok)[0]:
                        assert np.array_equal(out[k][ptr[b]:ptr[b + 1]], ref[k][ptr[b]:ptr[b + 1]]), (k, b)
                for k in ("peak_lb", "plan_peak", "verdict"):
                    assert np.array_equal(out[k][ok], ref[k][ok]), k
                assert np.array_equal(out["conflict"].reshape(-1, 2)[ok], ref["conflict"][ok])


# ------------------------------------------------------------- greedy by breadth

@pytest.mark.parametrize("name,pol", POLICIES)
def test_breadth_parity(cuda_lib, name, pol):
    import paper_2203_00448_gb300 as mp

    hand = tg.from_tuples([(2, [(0, 2, 5)] + [(0, 1, 4)] * 6 + [(1, 2, 20)])])
    for ts in (tg.config(0), tg.config(1), tg.config(2).select(range(0, 4096, 16)), tg.config(3), hand,
               tg.random_small(17, 200, 100, 150, 1 << 24),
               tg.from_tuples([(4, [(-1, 2, 8)]), (4, [(0, 1, 2 ** 62), (0, 2, 2 ** 62)]), (0, []), (5, [])])):
        db = mp.DeviceBatch.from_host(ts, "cuda")
        off, pk, st = mp.plan_greedy_by_breadth(db, name)
        torch.cuda.synchronize()
        o_off, o_pk, o_st = oracle.plan_greedy_by_breadth(ts, pol)
        st, pk, off = st.cpu().numpy(), pk.cpu().numpy(), off.cpu().numpy()
        assert np.array_equal(st, o_st), ts.name
        assert np.array_equal(pk, o_pk), ts.name
        for b in np.nonzero(o_st == 0)[0]:
            lo, hi = ts.trace_ptr[b], ts.trace_ptr[b + 1]
            assert np.array_equal(off[lo:hi], o_off[lo:hi]), (ts.name, b)


@pytest.mark.parametrize("name,pol", POLICIES)
def test_breadth_component_tiers(cuda_lib, name, pol):
    """Greedy by breadth through its component kernel: components of 2..8
    tensors (a thread each), 9..32 (a warp each) and larger (the whole CTA),
    sizes drawn from two values so that breadths, steps and sizes tie often;
    traces whose large components outgrow the CTA tier's scratch (more than
    0.6 tensors per step) go to the per-tensor kernel in the same call."""
    import paper_2203_00448_gb300 as mp

    rng = np.random.default_rng(41)
    traces = []
    for b in range(300):
        n, T = int(rng.integers(20, 400)), int(rng.integers(100, 900))
        a = rng.integers(0, T - 1, size=n)
        life = 1 + rng.geometric(0.35 if b % 7 else 0.08, size=n)
        f = np.minimum(a + life, T)
        s = rng.choice([64, 128], size=n)
        traces.append((T, a, f, s))
    ts = tg.from_arrays(traces)
    big = 0
    for b in range(ts.n_traces):
        _, a, f, _ = ts.trace(b)
        o = np.lexsort((np.arange(len(a)), a))
        run = np.maximum.accumulate(np.asarray(f)[o])
        starts = np.flatnonzero(np.r_[True, run[:-1] <= np.asarray(a)[o][1:]])
        big += int(np.diff(np.r_[starts, len(a)]).max() > 32)
    assert 0 < big < ts.n_traces
    db = mp.DeviceBatch.from_host(ts, "cuda")
    off, pk, st = mp.plan_greedy_by_breadth(db, name)
    torch.cuda.synchronize()
    o_off, o_pk, o_st = oracle.plan_greedy_by_breadth(ts, pol)
    assert np.array_equal(st.cpu().numpy(), o_st) and (o_st == 0).all()
    assert np.array_equal(pk.cpu().numpy(), o_pk)
    assert np.array_equal(off.cpu().numpy(), o_off)


def test_host_path_against_the_oracle_unpacked(cuda_lib):
    """mp_plan_and_validate_host through the C ABI with host arrays spaced 64
    bytes apart and in another order (one copy per array both ways), and with
    conflict NULL, checked against the oracle directly."""
    import ctypes

    from paper_2203_00448_gb300 import _lib

    lib = _lib.load()
    ts = tg.random_small(43, 150, 300, 400, 1 << 28)
    B, N, S = ts.n_traces, ts.n_tensors, ts.n_steps
    arrays = [("size_bytes", ts.size_bytes, np.int64), ("steps", ts.steps, np.int32),
              ("trace_ptr", ts.trace_ptr, np.int64), ("free_step", ts.free_step, np.int32),
              ("profile_ptr", ts.profile_ptr, np.int64), ("alloc_step", ts.alloc_step, np.int32)]
    outs = [("status", B, np.int32), ("offsets", N, np.int64), ("verdict", B, np.int32), ("profile", S, np.int64),
            ("plan_peak", B, np.int64), ("peak_lb", B, np.int64)]
    total = sum(np.asarray(a).nbytes + 64 for _, a, _ in arrays) + sum(n * np.dtype(d).itemsize + 64 for _, n, d in outs)
    buf = torch.empty(total + 64, dtype=torch.uint8, pin_memory=True)
    pos, view = 64, {}
    for name, a, dt in arrays:
        a = np.asarray(a, dtype=dt)
        view[name] = buf[pos:pos + a.nbytes].view(torch.int64 if dt == np.int64 else torch.int32)
        view[name].numpy()[...] = a
        pos += a.nbytes + 64
    for name, n, dt in outs:
        nbytes = n * np.dtype(dt).itemsize
        view[name] = buf[pos:pos + nbytes].view(torch.int64 if dt == np.int64 else torch.int32)
        view[name].fill_(-3)
        pos += nbytes + 64
    p = lambda k: view[k].data_ptr()
    hb = _lib.MpBatch(B, int(ts.max_tensors), int(ts.max_steps), 0, N, S, p("trace_ptr"), p("steps"),
                      p("profile_ptr"), p("alloc_step"), p("free_step"), p("size_bytes"))
    res = _lib.MpHostResults(p("profile"), p("peak_lb"), p("offsets"), p("plan_peak"), p("verdict"), None, p("status"))
    for chunks in (1, 3):
        need = lib.mp_host_path_bytes(ctypes.byref(hb), chunks)
        dbuf = torch.empty(need, dtype=torch.uint8, device="cuda")
        s = torch.cuda.current_stream().cuda_stream
        st = lib.mp_plan_and_validate_host(ctypes.byref(hb), 0, ctypes.byref(res), chunks, dbuf.data_ptr(),
                                           dbuf.numel(), s, s, s)
        assert st == 0
        torch.cuda.synchronize()
        o_prof, o_lb, o_st_p = oracle.live_profile(ts)
        o_off, o_pk, o_st_g = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
        o_v, _, _ = oracle.validate_plan(ts, o_off)
        assert (o_st_p == 0).all() and (o_st_g == 0).all()
        got = {k: view[k].numpy().copy() for k, _, _ in outs}
        assert np.array_equal(got["status"], o_st_g)
        for k, want in (("profile", o_prof), ("peak_lb", o_lb), ("offsets", o_off), ("plan_peak", o_pk),
                        ("verdict", o_v)):
            assert np.array_equal(got[k], want), (chunks, k)


@pytest.mark.parametrize("name,pol", POLICIES)
def test_two_per_lane_warp_tier(cuda_lib, name, pol):
    """Components of 33..64 tensors, placed by one warp with two tensors per
    lane: overlap structures from chains to near-cliques, sizes drawn from few
    values (ties broken by alloc step and id), in 32-bit traces, traces whose
    sizes sum past 2^32 (the 64-bit launch), and a batch wide enough in steps
    to keep its working set in the workspace."""
    rng = np.random.default_rng(77)

    def comp_trace(c, T, big):
        a = np.sort(rng.integers(0, T // 2, size=c))
        f = np.minimum(a + rng.integers(1, T // 2, size=c), T)
        # keep it one component: every tensor overlaps the next in alloc order
        for i in range(c - 1):
            if f[i] <= a[i + 1]:
                f[i] = a[i + 1] + 1
        s = rng.choice([64, 128, 192], size=c) * ((1 << 26) if big else 1)
        return a, f, s

    traces = []
    for k, c in enumerate([33, 40, 47, 55, 63, 64] * 3):
        T0 = int(rng.integers(80, 300))
        a, f, s = comp_trace(c, T0, big=(k % 3 == 2))
        # a few tiny components after it
        extra = rng.integers(T0, T0 + 99, size=20)
        traces.append((T0 + 100, np.concatenate([a, extra]), np.concatenate([f, extra + 1]),
                       np.concatenate([s, rng.integers(1, 100, size=20) * 8])))
    ts = tg.from_arrays(traces)
    assert_parity(ts, gpu_run(ts, name), oracle_run(ts, pol))
    # the same components with the working set in the workspace (many steps)
    wide = tg.from_arrays([(T + 40000, a, f, s) for (T, a, f, s) in traces[:6]])
    assert_parity(wide, gpu_run(wide, name), oracle_run(wide, pol))
