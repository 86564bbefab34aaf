"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every check here is independent of the oracle's own code: hand-derived
fixtures (tests/golden/hand_cases.json), closed forms, special cases with
textbook answers, brute force over subsets / orderings / Eq. 2.1
orientations, invariants, and planted conflicts.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle
import tracegen as tg
from tests import refs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_cases.json")
CASES = json.load(open(GOLDEN))


def one(T, tensors):
    return tg.from_tuples([(T, tensors)])


def rand_trace(rng, n, T, smax=64, life_max=None):
    a = rng.integers(0, T, size=n)
    life = rng.integers(1, (life_max or T) + 1, size=n)
    f = np.minimum(a + life, T)
    s = rng.integers(1, smax + 1, size=n)
    return [(int(x), int(y), int(z)) for x, y, z in zip(a, f, s)]


# ------------------------------------------------------------- hand fixtures

@pytest.mark.parametrize("case", CASES["plan_cases"], ids=lambda c: c["name"])
def test_hand_plan_cases(case):
    ts = one(case["T"], case["tensors"])
    prof, lb, st = oracle.live_profile(ts)
    assert st.tolist() == [0]
    assert prof.tolist() == case["profile"]
    assert lb.tolist() == [case["peak_lb"]]
    for pol, key in ((oracle.FIT_FIRST, "first"), (oracle.FIT_BEST, "best")):
        off, pk, st = oracle.plan_greedy_by_size(ts, pol)
        assert st.tolist() == [0]
        assert off.tolist() == case[key], key
        assert pk.tolist() == [case["plan_peak_" + key]]


@pytest.mark.parametrize("case", CASES["validate_cases"], ids=lambda c: c["name"])
def test_hand_validate_cases(case):
    ts = one(case["T"], case["tensors"])
    v, c, st = oracle.validate_plan(ts, np.array(case["offsets"], dtype=np.int64))
    assert st.tolist() == [0]
    assert v.tolist() == [case["verdict"]]
    assert c[0].tolist() == case["conflict"]


# ------------------------------------------------------------- live profile

def test_profile_closed_form_sum():
    """sum_t profile[t] = sum_i size_i * (free_i - alloc_i)."""
    ts = tg.random_small(11, 40, 30, 50, 1 << 20)
    prof, lb, st = oracle.live_profile(ts)
    assert (st == 0).all()
    for b in range(ts.n_traces):
        T, a, f, s = ts.trace(b)
        p = prof[ts.profile_ptr[b]:ts.profile_ptr[b + 1]]
        assert int(p.sum()) == int(np.sum(s.astype(np.int64) * (f - a).astype(np.int64)))
        assert (p >= 0).all()
        assert lb[b] == (p.max() if T else 0)


def test_profile_single_tensor():
    ts = one(9, [(3, 7, 5000)])
    prof, lb, _ = oracle.live_profile(ts)
    assert prof.tolist() == [0, 0, 0, 5000, 5000, 5000, 5000, 0, 0]
    assert lb.tolist() == [5000]


def test_peak_lb_is_max_clique_weight():
    """max_t profile equals the heaviest pairwise-overlapping set (Helly)."""
    rng = np.random.default_rng(5)
    for _ in range(60):
        n, T = int(rng.integers(1, 10)), int(rng.integers(1, 12))
        tensors = rand_trace(rng, n, T, smax=1000)
        _, lb, _ = oracle.live_profile(one(T, tensors))
        assert lb[0] == refs.max_clique_weight(tensors)


# ------------------------------------------------------------- greedy special cases

def test_disjoint_lifetimes_all_at_zero():
    tensors = [(k, k + 1, 64 * (k % 7 + 1)) for k in range(20)]
    ts = one(20, tensors)
    for pol in (0, 1):
        off, pk, _ = oracle.plan_greedy_by_size(ts, pol)
        assert off.tolist() == [0] * 20
        assert pk[0] == max(s for _, _, s in tensors)


def test_clique_is_prefix_sum_in_priority_order():
    rng = np.random.default_rng(7)
    for _ in range(20):
        n, T = int(rng.integers(1, 30)), 10
        tensors = [(int(rng.integers(0, 5)), int(rng.integers(5, 11)), int(rng.integers(1, 50))) for _ in range(n)]
        order = sorted(range(n), key=lambda i: (-tensors[i][2], tensors[i][0], i))
        expect, acc = [0] * n, 0
        for i in order:
            expect[i] = acc
            acc += tensors[i][2]
        for pol in (0, 1):
            off, pk, _ = oracle.plan_greedy_by_size(one(T, tensors), pol)
            assert off.tolist() == expect
            assert pk[0] == acc


def test_equal_sizes_reach_lower_bound():
    """Equal sizes: priority = alloc order, and left-endpoint first fit colours
    an interval graph optimally, so the plan peak equals the live-bytes peak."""
    rng = np.random.default_rng(9)
    for _ in range(40):
        n, T = int(rng.integers(1, 60)), int(rng.integers(1, 40))
        tensors = [(a, f, 256) for a, f, _ in rand_trace(rng, n, T)]
        ts = one(T, tensors)
        _, lb, _ = oracle.live_profile(ts)
        for pol in (0, 1):
            _, pk, _ = oracle.plan_greedy_by_size(ts, pol)
            assert pk[0] == lb[0]


# ------------------------------------------------------------- greedy vs independent restatements

def test_first_fit_equals_lowest_feasible_offset():
    rng = np.random.default_rng(13)
    for _ in range(300):
        n, T = int(rng.integers(0, 25)), int(rng.integers(1, 20))
        tensors = rand_trace(rng, n, T, smax=int(rng.integers(1, 100)))
        off, _, _ = oracle.plan_greedy_by_size(one(T, tensors), oracle.FIT_FIRST)
        assert off.tolist() == refs.first_fit_in_priority_order(tensors)


def test_best_fit_equals_smallest_free_hole():
    rng = np.random.default_rng(17)
    for _ in range(300):
        n, T = int(rng.integers(0, 25)), int(rng.integers(1, 20))
        tensors = rand_trace(rng, n, T, smax=int(rng.integers(1, 100)))
        off, _, _ = oracle.plan_greedy_by_size(one(T, tensors), oracle.FIT_BEST)
        assert off.tolist() == refs.best_fit_in_priority_order(tensors)


# ------------------------------------------------------------- optimum

def test_bruteforce_matches_eq21_orientations():
    """For n <= 5 the all-orderings first-fit search equals the Eq. 2.1
    optimum found by enumerating every z_ij orientation."""
    rng = np.random.default_rng(19)
    for _ in range(80):
        n, T = int(rng.integers(1, 6)), int(rng.integers(1, 6))
        tensors = rand_trace(rng, n, T, smax=20)
        a, f, s = (np.array([t[k] for t in tensors]) for k in range(3))
        opt, offs = oracle.bruteforce_opt(a, f, s)
        assert opt == refs.mip_optimum(tensors)
        v, _, _ = oracle.validate_plan(one(T, tensors), offs)
        assert v[0] == 1 and max(int(o) + t[2] for o, t in zip(offs, tensors)) == opt


def test_lower_bound_le_optimum_le_greedy():
    rng = np.random.default_rng(23)
    gaps = []
    for _ in range(60):
        n, T = int(rng.integers(1, 8)), int(rng.integers(1, 10))
        tensors = rand_trace(rng, n, T, smax=100)
        ts = one(T, tensors)
        a, f, s = (np.array([t[k] for t in tensors]) for k in range(3))
        opt, _ = oracle.bruteforce_opt(a, f, s)
        _, lb, _ = oracle.live_profile(ts)
        for pol in (0, 1):
            _, pk, _ = oracle.plan_greedy_by_size(ts, pol)
            assert lb[0] <= opt <= pk[0]
            gaps.append(pk[0] / opt)
    assert min(gaps) == 1.0  # greedy is often exactly optimal on tiny traces


# ------------------------------------------------------------- invariants

def test_plans_validate_and_are_bounded():
    ts = tg.random_small(29, 60, 80, 60, 1 << 16)
    _, lb, _ = oracle.live_profile(ts)
    for pol in (0, 1):
        off, pk, st = oracle.plan_greedy_by_size(ts, pol)
        assert (st == 0).all()
        v, c, st = oracle.validate_plan(ts, off)
        assert (st == 0).all() and (v == 1).all() and (c == -1).all()
        sums = np.add.reduceat(ts.size_bytes, ts.trace_ptr[:-1]) if ts.n_tensors else None
        for b in range(ts.n_traces):
            n = ts.trace_ptr[b + 1] - ts.trace_ptr[b]
            total = int(sums[b]) if n else 0
            assert lb[b] <= pk[b] <= total


def test_homogeneity_and_shift_invariance():
    """Scaling every size by k scales every offset by k (the linearity in
    batch size noted in Ch. 7); shifting every step by c changes nothing."""
    rng = np.random.default_rng(31)
    for _ in range(40):
        n, T = int(rng.integers(1, 40)), int(rng.integers(1, 30))
        tensors = rand_trace(rng, n, T, smax=500)
        for pol in (0, 1):
            base, _, _ = oracle.plan_greedy_by_size(one(T, tensors), pol)
            k = int(rng.integers(2, 9))
            scaled, _, _ = oracle.plan_greedy_by_size(one(T, [(a, f, s * k) for a, f, s in tensors]), pol)
            assert (scaled == base * k).all()
            c = int(rng.integers(1, 9))
            shifted, _, _ = oracle.plan_greedy_by_size(one(T + c, [(a + c, f + c, s) for a, f, s in tensors]), pol)
            assert (shifted == base).all()


# ------------------------------------------------------------- validation

def test_planted_conflict_is_reported():
    rng = np.random.default_rng(37)
    found = 0
    for _ in range(200):
        n, T = int(rng.integers(2, 30)), int(rng.integers(1, 20))
        tensors = rand_trace(rng, n, T, smax=64)
        ts = one(T, tensors)
        off, _, _ = oracle.plan_greedy_by_size(ts, 0)
        pairs = [(i, j) for i, j in itertools.combinations(range(n), 2) if refs.overlap(tensors[i], tensors[j])]
        if not pairs:
            continue
        i, j = pairs[int(rng.integers(0, len(pairs)))]
        bad = off.copy()
        bad[j] = bad[i]  # j now starts where i starts: same bytes, overlapping lifetimes
        expect = min((p, q) for p, q in pairs
                     if bad[p] < bad[q] + tensors[q][2] and bad[q] < bad[p] + tensors[p][2])
        v, c, _ = oracle.validate_plan(ts, bad)
        assert v[0] == 0 and tuple(c[0]) == expect
        found += 1
    assert found > 100


def test_address_overlap_without_lifetime_overlap_is_legal():
    ts = one(6, [(0, 2, 100), (2, 4, 100), (4, 6, 100)])
    v, c, _ = oracle.validate_plan(ts, np.zeros(3, dtype=np.int64))
    assert v[0] == 1 and c[0].tolist() == [-1, -1]


# ------------------------------------------------------------- bump allocation

def test_bump_allocation_is_running_offset_in_alloc_order():
    ts = one(10, [(3, 5, 10), (0, 2, 20), (3, 4, 30), (1, 9, 40)])
    off, pk, _ = oracle.plan_bump(ts)
    # alloc order: id1 (0), id3 (1), id0 (3), id2 (3)
    assert off.tolist() == [60, 0, 70, 20]
    assert pk[0] == 100


# ------------------------------------------------------------- error codes

@pytest.mark.parametrize("tensors,T,code", [
    ([(-1, 2, 8)], 4, 1),            # alloc < 0
    ([(2, 2, 8)], 4, 1),             # free <= alloc
    ([(1, 5, 8)], 4, 1),             # free > T
    ([(0, 1, 0)], 4, 1),             # size <= 0
    ([(0, 1, 2 ** 62), (0, 1, 2 ** 62)], 4, 2),   # sizes sum to 2^63 > INT64_MAX
    ([(0, 1, 2 ** 62), (0, 1, -5)], 4, 1),        # EINVAL wins over EOVERFLOW
])
def test_trace_status_codes(tensors, T, code):
    ts = tg.from_tuples([(T, tensors), (3, [(0, 3, 7)])])
    for fn in (lambda: oracle.live_profile(ts)[2], lambda: oracle.plan_greedy_by_size(ts, 0)[2],
               lambda: oracle.validate_plan(ts, np.zeros(ts.n_tensors, dtype=np.int64))[2]):
        st = fn()
        assert st.tolist() == [code, 0]


def test_offset_status_codes():
    ts = one(4, [(0, 2, 8), (1, 3, 8)])
    _, _, st = oracle.validate_plan(ts, np.array([0, -1]))
    assert st.tolist() == [1]
    _, _, st = oracle.validate_plan(ts, np.array([0, 2 ** 63 - 4]))
    assert st.tolist() == [2]
    pk, st = oracle.peak(ts, np.array([0, 100]))
    assert st.tolist() == [0] and pk.tolist() == [108]


# ------------------------------------------------------------- greedy by breadth

def test_breadth_hand_case_orders_by_the_widest_operator():
    """T = 2.  x: 5 bytes over [0, 2); six tensors of 4 bytes over [0, 1);
    y: 20 bytes over [1, 2).  Operator 0 holds x and the six (29 bytes),
    operator 1 holds x and y (25): operator 0 goes first, x (its largest) at
    0 and the six stacked above it (5, 9, ..., 25); then y, overlapping only
    x, at 5.  greedy_by_size instead takes y first (0), x above it (20), and
    the six around x (0, 4, 8, 12, 16, 25)."""
    tensors = [(0, 2, 5)] + [(0, 1, 4)] * 6 + [(1, 2, 20)]
    ts = tg.from_tuples([(2, tensors)])
    off, pk, st = oracle.plan_greedy_by_breadth(ts, oracle.FIT_FIRST)
    assert st[0] == 0 and pk[0] == 29
    assert list(off) == [0, 5, 9, 13, 17, 21, 25, 5]
    off_s, pk_s, _ = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
    assert list(off_s) == [20, 0, 4, 8, 12, 16, 25, 0] and pk_s[0] == 29


def test_breadth_reads_operators_by_their_inputs_and_outputs():
    """T = 3, tensors (alloc, free, size): t0 (2, 3, 12), t1 (0, 3, 10), t2
    (1, 2, 9), t3 (0, 2, 3), t4 (0, 3, 8).  Operator 0 produces t1, t3, t4
    (21 bytes); operator 1 produces t2 and uses t3 last (12); operator 2
    produces t0 and uses t1 and t4 last (30).  So t0, t1, t4 go first (operator
    2, by size), then t3 (operator 0), then t2 (operator 1).  FIRST: t0 at 0,
    t1 above it at 12, t4 above both at 22, t3 at 0 (it meets t1 and t4 only),
    t2 at 3 (above t3, below t1): peak 30.  Reading an operator as every
    tensor live at its step would make operators 1 and 2 tie at 30 bytes and
    give [27, 0, 10, 27, 19]; greedy_by_size gives [0, 12, 0, 9, 22]."""
    ts = tg.from_tuples([(3, [(2, 3, 12), (0, 3, 10), (1, 2, 9), (0, 2, 3), (0, 3, 8)])])
    off, pk, st = oracle.plan_greedy_by_breadth(ts, oracle.FIT_FIRST)
    assert st[0] == 0 and list(off) == [0, 12, 3, 0, 22] and pk[0] == 30
    off_s, _, _ = oracle.plan_greedy_by_size(ts, oracle.FIT_FIRST)
    assert list(off_s) == [0, 12, 0, 9, 22]


def test_breadth_equals_size_when_one_operator_produces_everything():
    # every tensor is allocated at step 0: operator 0 produces all of them and
    # is at least as wide as any last user, so the order is the size order
    rng = np.random.default_rng(11)
    for _ in range(20):
        n = int(rng.integers(1, 12))
        f = rng.integers(1, 8, n)
        s = rng.integers(1, 100, n)
        ts = tg.from_tuples([(8, [(0, int(f[k]), int(s[k])) for k in range(n)])])
        for pol in (oracle.FIT_FIRST, oracle.FIT_BEST):
            assert np.array_equal(oracle.plan_greedy_by_breadth(ts, pol)[0], oracle.plan_greedy_by_size(ts, pol)[0])


def test_breadth_plans_are_valid_and_bounded():
    ts = tg.random_small(13, 40, 9, 12, 1 << 10)
    for pol in (oracle.FIT_FIRST, oracle.FIT_BEST):
        off, pk, st = oracle.plan_greedy_by_breadth(ts, pol)
        v, _, vst = oracle.validate_plan(ts, off)
        _, lb, _ = oracle.live_profile(ts)
        ok = st == 0
        assert (v[ok] == 1).all() and (vst[ok] == 0).all()
        assert (lb[ok] <= pk[ok]).all()
        for b in np.nonzero(ok)[0]:
            T, a, f, s = ts.trace(b)
            if len(a) <= 7:
                assert oracle.bruteforce_opt(a, f, s)[0] <= pk[b]
