/*
 * oracle.c -- plain, slow, obviously correct CPU reference of the
 * memory-planning path (live-bytes profile, greedy_by_size, plan validation).
 *
 * TEST INFRASTRUCTURE ONLY: used by the tests, the package's smoke check and
 * the bench's CPU-baseline leg, never by the product path.  It shares no code
 * with the CUDA library and deliberately uses different algorithms from it:
 * the profile adds each tensor to every step it is live at (no difference
 * array, no scan), greedy_by_size sorts with qsort and scans all placed
 * tensors for every tensor, and validation is the literal double loop.
 *
 * Passages followed:
 *   Eq. 2.1 and its pairwise constraints (Sec. 2.3): a plan is feasible when
 *     every pair of lifetime-overlapping tensors is ordered in address space,
 *     and total_mem >= offset_i + mem_i for every i.
 *   Sec. 2.3, strategy list: greedy_by_size sorts the intermediates by size and
 *     assigns offsets among lifetime-overlapping tensors by a fit criterion;
 *     bump_allocation gives every allocation the running offset.
 *   Sec. 3.2: greedy_by_size is the default strategy.
 *
 * Readings where the paper is silent (each is part of the public contract):
 *   - lifetimes are half-open [alloc, free): a tensor freed at step t and one
 *     allocated at t do not overlap;
 *   - priority ties: size descending, then alloc step ascending, then id;
 *   - gaps are measured against the running maximum end of the placed
 *     tensors taken in (offset, id) order, the region [0, first offset) is a
 *     gap, and the region above everything is used only if no gap fits;
 *   - FIRST takes the first gap that fits (the lowest feasible offset), BEST
 *     the smallest gap that fits, the lowest such gap on ties;
 *   - touching address ranges (offset_i + size_i == offset_j) are legal,
 *     as Eq. 2.1 uses <=.
 */
#include "oracle.h"

#include <stdlib.h>
#include <string.h>

#define OR_EXPORT __attribute__((visibility("default")))

/* ------------------------------------------------------------ per-trace checks */

/* Status of trace b from its metadata and tensors (and offsets when given):
 * EINVAL for a bad CSR range, T < 0, alloc < 0, free <= alloc, free > T,
 * size <= 0 or offset < 0; otherwise EOVERFLOW when the sizes sum, or some
 * offset + size, exceeds INT64_MAX; otherwise OK. */
static int32_t trace_check(const or_batch *B, int32_t b, const int64_t *offsets, int need_profile)
{
    int64_t lo = B->trace_ptr[b], hi = B->trace_ptr[b + 1];
    int32_t T = B->steps[b];
    if (lo < 0 || hi < lo || T < 0) return OR_EINVAL;
    if (need_profile && B->profile_ptr[b + 1] - B->profile_ptr[b] != (int64_t)T) return OR_EINVAL;
    int overflow = 0;
    int64_t total = 0;
    for (int64_t k = lo; k < hi; ++k) {
        int32_t a = B->alloc_step[k], f = B->free_step[k];
        int64_t s = B->size_bytes[k];
        if (a < 0 || f <= a || f > T || s <= 0) return OR_EINVAL;
        if (offsets && offsets[k] < 0) return OR_EINVAL;
        if (total > INT64_MAX - s) overflow = 1;
        else total += s;
        if (offsets && offsets[k] > INT64_MAX - s) overflow = 1;
    }
    return overflow ? OR_EOVERFLOW : OR_OK;
}

static int lifetimes_overlap(int32_t ai, int32_t fi, int32_t aj, int32_t fj)
{
    return ai < fj && aj < fi;
}

/* -------------------------------------------------------------- live profile */

OR_EXPORT int or_live_profile(const or_batch *B, int64_t *profile, int64_t *peak_lb, int32_t *trace_status)
{
    for (int32_t b = 0; b < B->n_traces; ++b) {
        int32_t st = trace_check(B, b, NULL, 1);
        trace_status[b] = st;
        int32_t T = B->steps[b];
        int64_t *prof = profile + B->profile_ptr[b];
        if (st != OR_OK) {
            peak_lb[b] = 0;
            if (T > 0 && B->profile_ptr[b + 1] - B->profile_ptr[b] == (int64_t)T)
                for (int32_t t = 0; t < T; ++t) prof[t] = 0;
            continue;
        }
        for (int32_t t = 0; t < T; ++t) prof[t] = 0;
        for (int64_t k = B->trace_ptr[b]; k < B->trace_ptr[b + 1]; ++k)
            for (int32_t t = B->alloc_step[k]; t < B->free_step[k]; ++t) prof[t] += B->size_bytes[k];
        int64_t m = 0;
        for (int32_t t = 0; t < T; ++t)
            if (prof[t] > m) m = prof[t];
        peak_lb[b] = m;
    }
    return 0;
}

/* ----------------------------------------------------------- greedy_by_size */

/* qsort has no context argument; the oracle is single-threaded, so the trace
 * being sorted is reached through these file-scope pointers. */
static const int32_t *g_a;
static const int64_t *g_s;
static const int64_t *g_off;

/* Priority: larger size first, then earlier alloc step, then smaller id. */
static int cmp_priority(const void *x, const void *y)
{
    int32_t i = *(const int32_t *)x, j = *(const int32_t *)y;
    if (g_s[i] != g_s[j]) return g_s[i] > g_s[j] ? -1 : 1;
    if (g_a[i] != g_a[j]) return g_a[i] < g_a[j] ? -1 : 1;
    return (i > j) - (i < j);
}

/* Address order of placed tensors: offset ascending, then id. */
static int cmp_offset(const void *x, const void *y)
{
    int32_t i = *(const int32_t *)x, j = *(const int32_t *)y;
    if (g_off[i] != g_off[j]) return g_off[i] < g_off[j] ? -1 : 1;
    return (i > j) - (i < j);
}

/* Allocation order: alloc step ascending, then id. */
static int cmp_alloc(const void *x, const void *y)
{
    int32_t i = *(const int32_t *)x, j = *(const int32_t *)y;
    if (g_a[i] != g_a[j]) return g_a[i] < g_a[j] ? -1 : 1;
    return (i > j) - (i < j);
}

/* Offset of a tensor of the given size among the lifetime-overlapping
 * placed tensors listed in `nb` (already in (offset, id) order). */
static int64_t fit_in_gaps(int32_t policy, int64_t size, const int32_t *nb, int32_t n_nb,
                           const int64_t *off, const int64_t *s)
{
    int64_t prev = 0;          /* running maximum end of the tensors seen so far */
    int64_t best_gap = -1, best_off = 0;
    for (int32_t k = 0; k < n_nb; ++k) {
        int32_t x = nb[k];
        int64_t gap = off[x] - prev;
        if (gap >= size) {
            if (policy == OR_FIT_FIRST) return prev;
            if (best_gap < 0 || gap < best_gap) {
                best_gap = gap;
                best_off = prev;
            }
        }
        int64_t end = off[x] + s[x];
        if (end > prev) prev = end;
    }
    if (policy == OR_FIT_BEST && best_gap >= 0) return best_off;
    return prev;
}

/* Places the tensors of one trace in the given order: each at the first or
 * the smallest gap among the already placed, lifetime-overlapping tensors
 * (the placement rule of greedy_by_size); returns the plan's peak. */
static int64_t place_in_order(int32_t policy, int32_t n, const int32_t *order, const int32_t *a,
                              const int32_t *f, const int64_t *s, int64_t *off)
{
    int32_t *placed = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n ? n : 1));
    int32_t *nb = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n ? n : 1));
    int32_t n_placed = 0;
    for (int32_t r = 0; r < n; ++r) {
        int32_t i = order[r];
        int32_t n_nb = 0;
        for (int32_t k = 0; k < n_placed; ++k) {
            int32_t j = placed[k];
            if (lifetimes_overlap(a[i], f[i], a[j], f[j])) nb[n_nb++] = j;
        }
        g_off = off;
        qsort(nb, (size_t)n_nb, sizeof(int32_t), cmp_offset);
        off[i] = fit_in_gaps(policy, s[i], nb, n_nb, off, s);
        placed[n_placed++] = i;
    }
    int64_t peak = 0;
    for (int32_t i = 0; i < n; ++i)
        if (off[i] + s[i] > peak) peak = off[i] + s[i];
    free(placed);
    free(nb);
    return peak;
}

OR_EXPORT int or_plan_greedy_by_size(const or_batch *B, int32_t policy, int64_t *offsets,
                                     int64_t *plan_peak, int32_t *trace_status)
{
    for (int32_t b = 0; b < B->n_traces; ++b) {
        int32_t st = trace_check(B, b, NULL, 0);
        trace_status[b] = st;
        int64_t lo = B->trace_ptr[b];
        int32_t n = st == OR_EINVAL && (lo < 0 || B->trace_ptr[b + 1] < lo)
                        ? 0 : (int32_t)(B->trace_ptr[b + 1] - lo);
        const int32_t *a = B->alloc_step + lo, *f = B->free_step + lo;
        const int64_t *s = B->size_bytes + lo;
        int64_t *off = offsets + lo;
        if (st != OR_OK) {
            for (int32_t i = 0; i < n; ++i) off[i] = 0;
            plan_peak[b] = 0;
            continue;
        }
        int32_t *order = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n ? n : 1));
        for (int32_t i = 0; i < n; ++i) order[i] = i;
        g_a = a;
        g_s = s;
        qsort(order, (size_t)n, sizeof(int32_t), cmp_priority);
        plan_peak[b] = place_in_order(policy, n, order, a, f, s, off);
        free(order);
    }
    return 0;
}

/* ------------------------------------------------------ greedy by breadth */

static const uint64_t *g_m; /* per tensor: the larger breadth of its two operators */
static const int32_t *g_t;  /* per tensor: the step of that operator (the earlier on ties) */

/* Breadth order: the widest operator first (earlier step on ties), then the
 * greedy_by_size priority inside an operator. */
static int cmp_breadth(const void *x, const void *y)
{
    int32_t i = *(const int32_t *)x, j = *(const int32_t *)y;
    if (g_m[i] != g_m[j]) return g_m[i] > g_m[j] ? -1 : 1;
    if (g_t[i] != g_t[j]) return g_t[i] < g_t[j] ? -1 : 1;
    return cmp_priority(x, y);
}

OR_EXPORT int or_plan_greedy_by_breadth(const or_batch *B, int32_t policy, int64_t *offsets,
                                        int64_t *plan_peak, int32_t *trace_status)
{
    for (int32_t b = 0; b < B->n_traces; ++b) {
        int32_t st = trace_check(B, b, NULL, 0);
        trace_status[b] = st;
        int64_t lo = B->trace_ptr[b];
        int32_t n = st == OR_EINVAL && (lo < 0 || B->trace_ptr[b + 1] < lo)
                        ? 0 : (int32_t)(B->trace_ptr[b + 1] - lo);
        const int32_t *a = B->alloc_step + lo, *f = B->free_step + lo;
        const int64_t *s = B->size_bytes + lo;
        int64_t *off = offsets + lo;
        if (st != OR_OK) {
            for (int32_t i = 0; i < n; ++i) off[i] = 0;
            plan_peak[b] = 0;
            continue;
        }
        int32_t T = B->steps[b];
        /* The operator at step t produces the tensors allocated at t and uses
         * for the last time the tensors freed at t + 1: its breadth is the
         * bytes of both (a tensor of one step counts once).  Every tensor
         * counts for at most two operators, so a breadth stays below 2^64. */
        uint64_t *breadth = (uint64_t *)calloc((size_t)(T > 0 ? T : 1), sizeof(uint64_t));
        for (int32_t i = 0; i < n; ++i) {
            breadth[a[i]] += (uint64_t)s[i];
            if (f[i] - 1 != a[i]) breadth[f[i] - 1] += (uint64_t)s[i];
        }
        const size_t cap = (size_t)(n > 0 ? n : 1);
        uint64_t *m = (uint64_t *)malloc(sizeof(uint64_t) * cap);
        int32_t *tm = (int32_t *)malloc(sizeof(int32_t) * cap);
        int32_t *order = (int32_t *)malloc(sizeof(int32_t) * cap);
        for (int32_t i = 0; i < n; ++i) {
            /* a tensor is placed by the wider of its producer and its last user */
            m[i] = breadth[a[i]];
            tm[i] = a[i];
            if (breadth[f[i] - 1] > m[i]) {
                m[i] = breadth[f[i] - 1];
                tm[i] = f[i] - 1;
            }
            order[i] = i;
        }
        g_a = a;
        g_s = s;
        g_m = m;
        g_t = tm;
        qsort(order, (size_t)n, sizeof(int32_t), cmp_breadth);
        plan_peak[b] = place_in_order(policy, n, order, a, f, s, off);
        free(breadth);
        free(m);
        free(tm);
        free(order);
    }
    return 0;
}

/* ----------------------------------------------------------- bump_allocation */

OR_EXPORT int or_plan_bump(const or_batch *B, int64_t *offsets, int64_t *plan_peak, int32_t *trace_status)
{
    for (int32_t b = 0; b < B->n_traces; ++b) {
        int32_t st = trace_check(B, b, NULL, 0);
        trace_status[b] = st;
        int64_t lo = B->trace_ptr[b];
        int32_t n = st == OR_EINVAL && (lo < 0 || B->trace_ptr[b + 1] < lo)
                        ? 0 : (int32_t)(B->trace_ptr[b + 1] - lo);
        int64_t *off = offsets + lo;
        if (st != OR_OK) {
            for (int32_t i = 0; i < n; ++i) off[i] = 0;
            plan_peak[b] = 0;
            continue;
        }
        int32_t *order = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n ? n : 1));
        for (int32_t i = 0; i < n; ++i) order[i] = i;
        g_a = B->alloc_step + lo;
        qsort(order, (size_t)n, sizeof(int32_t), cmp_alloc);
        int64_t bump = 0;
        for (int32_t r = 0; r < n; ++r) {
            off[order[r]] = bump;
            bump += B->size_bytes[lo + order[r]];
        }
        plan_peak[b] = bump;
        free(order);
    }
    return 0;
}

/* ---------------------------------------------------------------- validation */

OR_EXPORT int or_validate_plan(const or_batch *B, const int64_t *offsets, int32_t *verdict,
                               int32_t *conflict, int32_t *trace_status)
{
    for (int32_t b = 0; b < B->n_traces; ++b) {
        int32_t st = trace_check(B, b, offsets, 0);
        trace_status[b] = st;
        verdict[b] = 0;
        if (conflict) conflict[2 * b] = conflict[2 * b + 1] = -1;
        if (st != OR_OK) continue;
        int64_t lo = B->trace_ptr[b];
        int32_t n = (int32_t)(B->trace_ptr[b + 1] - lo);
        const int32_t *a = B->alloc_step + lo, *f = B->free_step + lo;
        const int64_t *s = B->size_bytes + lo, *off = offsets + lo;
        int ok = 1;
        for (int32_t i = 0; i < n && ok; ++i)
            for (int32_t j = i + 1; j < n; ++j) {
                if (!lifetimes_overlap(a[i], f[i], a[j], f[j])) continue;
                int disjoint = off[i] + s[i] <= off[j] || off[j] + s[j] <= off[i];
                if (!disjoint) {
                    ok = 0;
                    if (conflict) {
                        conflict[2 * b] = i;
                        conflict[2 * b + 1] = j;
                    }
                    break;
                }
            }
        verdict[b] = ok;
    }
    return 0;
}

OR_EXPORT int or_peak(const or_batch *B, const int64_t *offsets, int64_t *plan_peak, int32_t *trace_status)
{
    for (int32_t b = 0; b < B->n_traces; ++b) {
        int32_t st = trace_check(B, b, offsets, 0);
        trace_status[b] = st;
        plan_peak[b] = 0;
        if (st != OR_OK) continue;
        int64_t m = 0;
        for (int64_t k = B->trace_ptr[b]; k < B->trace_ptr[b + 1]; ++k)
            if (offsets[k] + B->size_bytes[k] > m) m = offsets[k] + B->size_bytes[k];
        plan_peak[b] = m;
    }
    return 0;
}

/* ------------------------------------------------------- exact DSA optimum */

/* Lowest offset at which tensor i fits among the tensors placed so far
 * (those with placed_flag set): the smallest candidate among 0 and the ends
 * of lifetime-overlapping placed tensors that conflicts with none of them. */
static int64_t lowest_fit(int32_t i, int32_t n, const int32_t *a, const int32_t *f, const int64_t *s,
                          const int64_t *off, const uint8_t *placed_flag)
{
    int64_t best = -1;
    for (int32_t c = -1; c < n; ++c) {
        int64_t cand;
        if (c < 0) cand = 0;
        else if (placed_flag[c] && lifetimes_overlap(a[i], f[i], a[c], f[c])) cand = off[c] + s[c];
        else continue;
        if (best >= 0 && cand >= best) continue;
        int ok = 1;
        for (int32_t j = 0; j < n && ok; ++j) {
            if (!placed_flag[j] || !lifetimes_overlap(a[i], f[i], a[j], f[j])) continue;
            if (cand < off[j] + s[j] && off[j] < cand + s[i]) ok = 0;
        }
        if (ok) best = cand;
    }
    return best;
}

OR_EXPORT int64_t or_bruteforce_opt(int32_t n, const int32_t *a, const int32_t *f, const int64_t *s,
                                    int64_t *best_offsets)
{
    if (n > 10 || n < 0) return -1;
    if (n == 0) return 0;
    int32_t perm[10];
    int64_t off[10];
    uint8_t placed[10];
    for (int32_t i = 0; i < n; ++i) perm[i] = i;
    int64_t best = -1;
    for (;;) {
        memset(placed, 0, sizeof(placed));
        int64_t peak = 0;
        for (int32_t r = 0; r < n; ++r) {
            int32_t i = perm[r];
            off[i] = lowest_fit(i, n, a, f, s, off, placed);
            placed[i] = 1;
            if (off[i] + s[i] > peak) peak = off[i] + s[i];
        }
        if (best < 0 || peak < best) {
            best = peak;
            if (best_offsets)
                for (int32_t i = 0; i < n; ++i) best_offsets[i] = off[i];
        }
        /* next permutation in lexicographic order */
        int32_t k = n - 2;
        while (k >= 0 && perm[k] >= perm[k + 1]) --k;
        if (k < 0) break;
        int32_t l = n - 1;
        while (perm[l] <= perm[k]) --l;
        int32_t t = perm[k];
        perm[k] = perm[l];
        perm[l] = t;
        for (int32_t x = k + 1, y = n - 1; x < y; ++x, --y) {
            t = perm[x];
            perm[x] = perm[y];
            perm[y] = t;
        }
    }
    return best;
}
