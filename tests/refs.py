"""Independent pure-Python checks used to pin the oracle (small inputs only).

None of these restate the oracle's code: each computes a fact about the
planning problem by a different route (subset enumeration, orientation
enumeration of Eq. 2.1, permutation search).
"""
from __future__ import annotations

import itertools


def overlap(t1, t2) -> bool:
    (a1, f1, _), (a2, f2, _) = t1, t2
    return a1 < f2 and a2 < f1


def max_clique_weight(tensors) -> int:
    """Heaviest set of pairwise lifetime-overlapping tensors (subset enumeration).

    Intervals that pairwise overlap share a common step (Helly property of
    intervals), so this equals the maximum of the live-bytes profile.
    """
    n = len(tensors)
    best = 0
    for mask in range(1, 1 << n):
        idx = [i for i in range(n) if mask >> i & 1]
        if all(overlap(tensors[i], tensors[j]) for i, j in itertools.combinations(idx, 2)):
            best = max(best, sum(tensors[i][2] for i in idx))
    return best


def mip_optimum(tensors) -> int:
    """Optimum of Eq. 2.1 by enumerating the z_ij orientations of every
    lifetime-overlapping pair: for an acyclic orientation the least offsets
    satisfying offset_i + mem_i <= offset_j along each oriented pair are the
    longest-path values, and total_mem is their max end."""
    n = len(tensors)
    if n == 0:
        return 0
    pairs = [(i, j) for i, j in itertools.combinations(range(n), 2) if overlap(tensors[i], tensors[j])]
    best = None
    for z in range(1 << len(pairs)):
        succ = [[] for _ in range(n)]
        indeg = [0] * n
        for k, (i, j) in enumerate(pairs):
            u, v = (i, j) if not (z >> k & 1) else (j, i)  # u below v in address space
            succ[u].append(v)
            indeg[v] += 1
        off = [0] * n
        ready = [i for i in range(n) if indeg[i] == 0]
        seen = 0
        while ready:
            u = ready.pop()
            seen += 1
            for v in succ[u]:
                off[v] = max(off[v], off[u] + tensors[u][2])
                indeg[v] -= 1
                if indeg[v] == 0:
                    ready.append(v)
        if seen < n:
            continue  # cyclic orientation: infeasible
        total = max(off[i] + tensors[i][2] for i in range(n))
        best = total if best is None else min(best, total)
    return best


def lowest_feasible(size, placed) -> int:
    """Lowest o >= 0 with [o, o + size) disjoint from every (off, end) in placed,
    found by scanning o upward over candidate starts (0 and every end)."""
    cands = sorted({0} | {e for _, e in placed})
    for o in cands:
        if all(o + size <= off or end <= o for off, end in placed):
            return o
    raise AssertionError("unreachable: the max end is always feasible")


def first_fit_in_priority_order(tensors):
    """greedy_by_size with the first-fit criterion restated as 'lowest feasible
    offset among lifetime-overlapping placed tensors', in priority order."""
    n = len(tensors)
    order = sorted(range(n), key=lambda i: (-tensors[i][2], tensors[i][0], i))
    off = [None] * n
    for i in order:
        placed = [(off[j], off[j] + tensors[j][2]) for j in range(n)
                  if off[j] is not None and overlap(tensors[i], tensors[j])]
        off[i] = lowest_feasible(tensors[i][2], placed)
    return off


def best_fit_in_priority_order(tensors):
    """greedy_by_size with best fit restated via the free intervals: merge the
    lifetime-overlapping placed ranges, list the maximal free holes below the
    top, take the smallest hole that fits (lowest on ties), else the top."""
    n = len(tensors)
    order = sorted(range(n), key=lambda i: (-tensors[i][2], tensors[i][0], i))
    off = [None] * n
    for i in order:
        rng = sorted((off[j], off[j] + tensors[j][2]) for j in range(n)
                     if off[j] is not None and overlap(tensors[i], tensors[j]))
        merged = []
        for lo, hi in rng:
            if merged and lo <= merged[-1][1]:
                merged[-1][1] = max(merged[-1][1], hi)
            else:
                merged.append([lo, hi])
        holes, cur = [], 0
        for lo, hi in merged:
            if lo > cur:
                holes.append((cur, lo - cur))
            cur = max(cur, hi)
        fits = [(length, start) for start, length in holes if length >= tensors[i][2]]
        off[i] = min(fits)[1] if fits else cur
    return off
