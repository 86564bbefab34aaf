// plan.cu -- stage 2: greedy_by_size offset assignment (Sec. 2.3; the default
// strategy of Sec. 3.2).
//
// Definition (sequential): take tensors in priority order -- size descending,
// alloc step ascending, id ascending -- and give each, among the already
// placed tensors whose lifetimes overlap its own, the first (FIRST) or the
// smallest fitting (BEST) gap in address order; above them all if none fits.
//
// Parallel form used here (exactly the same result).  Tensor i's offset is a
// function of the offsets of P_i = { j : overlap(i, j), j precedes i in
// priority } and of nothing else, because a placed tensor that does not
// overlap i in lifetime never constrains i.  The priority order orients every
// lifetime-overlap edge, giving a DAG; a tensor can be placed as soon as all
// of P_i are placed.  One CTA per trace runs Kahn's algorithm over that DAG:
// PEND[i] counts unplaced predecessors, each round places the whole frontier
// (tensors in one frontier never overlap each other, so they are
// independent) and decrements the successors' counters, which queues the
// tensors that became ready.  The number of rounds is the DAG's depth, not N.
// No sort is materialised: the priority order is used only as a comparator.
//
// Overlap pairs.  Short-lived tensors (life <= kLongLife) are counting-sorted
// by alloc step, so each short-short overlapping pair is found once, from the
// member that starts first (its forward window alloc_j < free_i), and stored
// in exact per-tensor predecessor / successor lists (count pass, prefix sum,
// fill pass).  Pairs with a long-lived tensor are found from the long side:
// the short tensors with alloc in [alloc - Lshort + 1, free) (Lshort = longest
// short lifetime) and the long tensors after it in the long list.  A short
// tensor meets its long neighbours by scanning the (small) long list; a long
// tensor, or every tensor of a trace whose lists exceed their capacity,
// enumerates its alloc-step window instead.
//
// Gap search.  FIRST is the lowest offset o at which [o, o + s_i) meets no
// predecessor [off_j, end_j).  Thread tier: start at o = 0 and jump to the
// largest end among the predecessors that conflict with [o, o + s_i) until
// none does (every feasible offset >= o is >= each conflicting end, so the
// first conflict-free o is the lowest feasible one).  BEST walks the maximal
// free holes below the top (max end) in address order -- jump off covered
// points, measure the hole to the next predecessor start -- and keeps the
// smallest hole that fits, the lowest on ties, else the top.  Warp and CTA
// tiers (many predecessors) test all candidates {0} U {end_j} in parallel
// instead: FIRST is the smallest conflict-free candidate; BEST scores each
// uncovered candidate c below the top by min{off_j >= c} - c.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int32_t kLongLife = 32;         // lifetimes above this are "long" (performance knob only)
constexpr int32_t kListCap = 2;           // list capacity per tensor (pairs), else window mode
constexpr int32_t kRegPred = 4;           // thread tier keeps up to this many predecessors in registers
constexpr int32_t kThreadMaxPred = 16;    // thread tier: at most this many predecessors,
constexpr int32_t kThreadMaxScan = 64;    // ... a predecessor scan of at most this many items
constexpr int32_t kThreadMaxRange = 512;  // ... and a successor scan of at most this many items
constexpr int32_t kWarpMaxRange = 16384;  // warp tier: enumeration items
constexpr int32_t kListedBit = 4;         // INFO: predecessors / successors come from the lists
enum : int32_t { kTierThread = 0, kTierWarp = 1, kTierCta = 2 };

__host__ __device__ constexpr size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

template <typename I>
struct PlanLayout {
    size_t s, off, pend, pre, sue, aux, bend, a, f, bys, longl, queue, predl, succl, info, total;
    __host__ __device__ PlanLayout(int64_t n, int64_t T) {
        s = 0;
        off = s + align16((size_t)n * 8);
        pend = off + align16((size_t)n * 8);
        pre = pend + align16((size_t)n * 4);
        sue = pre + align16((size_t)n * 4);
        aux = sue + align16((size_t)n * 4);
        bend = aux + align16((size_t)n * 4);
        a = bend + align16((size_t)T * 4);
        f = a + align16((size_t)n * sizeof(I));
        bys = f + align16((size_t)n * sizeof(I));
        longl = bys + align16((size_t)n * sizeof(I));
        queue = longl + align16((size_t)n * sizeof(I));
        predl = queue + align16((size_t)n * sizeof(I));
        succl = predl + align16((size_t)n * kListCap * sizeof(I));
        info = succl + align16((size_t)n * kListCap * sizeof(I));
        total = align_up(info + align16((size_t)n));
    }
};

template <typename I>
struct Trace {
    int64_t* S;
    int64_t* OFF;
    int32_t* PEND;  // unplaced predecessors (|P_i| once the pairs are counted)
    int32_t* PRE;   // end of i's predecessor list in PREDL (start: PRE[i - 1], or 0)
    int32_t* SUE;   // end of i's successor list in SUCCL
    int32_t* AUX;   // per-round tier lists
    int32_t* BEND;  // BEND[t] = number of short tensors with alloc <= t
    I* A;
    I* F;
    I* BYS;    // short tensors sorted by alloc step
    I* LONGL;  // long tensors, any order
    I* QUEUE;  // topological order as it is discovered
    I* PREDL;  // short predecessors of short tensors, grouped by tensor
    I* SUCCL;  // short successors of short tensors, grouped by tensor
    uint8_t* INFO;  // tier | kListedBit
    int32_t n, nlong, lshort;
};

// j strictly precedes i in priority (size desc, alloc asc, id asc).
template <typename I>
__device__ __forceinline__ bool precedes(const Trace<I>& m, int32_t j, int32_t i) {
    const int64_t sj = m.S[j], si = m.S[i];
    if (sj != si) return sj > si;
    const int32_t aj = m.A[j], ai = m.A[i];
    if (aj != ai) return aj < ai;
    return j < i;
}

// Enumeration of all of i's lifetime neighbours: items [0, nshort) are the
// short tensors with alloc in [alloc_i - lshort + 1, free_i), items
// [nshort, nshort + nlong) the long list.
struct Window {
    int32_t ai, fi, p0, nshort, range;
};

template <typename I>
__device__ __forceinline__ Window window_of(const Trace<I>& m, int32_t i) {
    Window w;
    w.ai = m.A[i];
    w.fi = m.F[i];
    int32_t lo = w.ai - m.lshort + 1;
    if (lo < 0) lo = 0;
    w.p0 = lo > 0 ? m.BEND[lo - 1] : 0;
    w.nshort = m.BEND[w.fi - 1] - w.p0;
    w.range = w.nshort + m.nlong;
    return w;
}

// Item k of i's window: the neighbour's id if it overlaps i in lifetime, else -1.
template <typename I>
__device__ __forceinline__ int32_t neighbour(const Trace<I>& m, int32_t i, const Window& w, int32_t k) {
    if (k < w.nshort) {
        const int32_t j = m.BYS[w.p0 + k];  // alloc_j < free_i by the window
        return (j != i && m.F[j] > w.ai) ? j : -1;
    }
    const int32_t j = m.LONGL[k - w.nshort];
    return (j != i && m.A[j] < w.fi && m.F[j] > w.ai) ? j : -1;
}

// Appends j to the queue; every tensor is pushed exactly once, so the slot is
// always < n -- the guard only keeps a defect from writing out of bounds.
template <typename I>
__device__ __forceinline__ void enqueue(const Trace<I>& m, int32_t j, int32_t* s_tail) {
    const int32_t pos = atomicAdd(s_tail, 1);
    if (pos < m.n) m.QUEUE[pos] = (I)j;
}

template <typename I>
__device__ __forceinline__ void push_ready(const Trace<I>& m, int32_t j, int32_t* s_tail) {
    if (atomicSub(m.PEND + j, 1) == 1) enqueue(m, j, s_tail);
}

// Calls fn(j) for every predecessor j of i (listed: short ones from the list,
// long ones from the long list; else the whole window).
template <typename I, typename Fn>
__device__ __forceinline__ void for_each_pred(const Trace<I>& m, int32_t i, bool listed, Fn&& fn) {
    if (listed) {
        const int32_t e = m.PRE[i];
        for (int32_t x = i ? m.PRE[i - 1] : 0; x < e; ++x) fn((int32_t)m.PREDL[x]);
        const int32_t ai = m.A[i], fi = m.F[i];
        for (int32_t u = 0; u < m.nlong; ++u) {
            const int32_t L = m.LONGL[u];
            if (m.A[L] < fi && m.F[L] > ai && precedes(m, L, i)) fn(L);
        }
    } else {
        const Window w = window_of(m, i);
        for (int32_t k = 0; k < w.range; ++k) {
            const int32_t j = neighbour(m, i, w, k);
            if (j >= 0 && precedes(m, j, i)) fn(j);
        }
    }
}

// Calls fn(j) for every successor j of i.
template <typename I, typename Fn>
__device__ __forceinline__ void for_each_succ(const Trace<I>& m, int32_t i, bool listed, Fn&& fn) {
    if (listed) {
        const int32_t e = m.SUE[i];
        for (int32_t x = i ? m.SUE[i - 1] : 0; x < e; ++x) fn((int32_t)m.SUCCL[x]);
        const int32_t ai = m.A[i], fi = m.F[i];
        for (int32_t u = 0; u < m.nlong; ++u) {
            const int32_t L = m.LONGL[u];
            if (m.A[L] < fi && m.F[L] > ai && precedes(m, i, L)) fn(L);
        }
    } else {
        const Window w = window_of(m, i);
        for (int32_t k = 0; k < w.range; ++k) {
            const int32_t j = neighbour(m, i, w, k);
            if (j >= 0 && precedes(m, i, j)) fn(j);
        }
    }
}

// ------------------------------------------------------------- gap search

constexpr int64_t kNone = INT64_MAX;

// FIRST by jumping: `each(fn)` calls fn(off, end) for every predecessor.
template <typename Each>
__device__ __forceinline__ int64_t fit_first_scan(int64_t s, Each&& each) {
    int64_t o = 0;
    for (;;) {
        int64_t next = o;
        each([&](int64_t po, int64_t pe) {
            if (po < o + s && o < pe && pe > next) next = pe;
        });
        if (next == o) return o;
        o = next;
    }
}

// BEST by walking the free holes below the top in address order.
template <typename Each>
__device__ __forceinline__ int64_t fit_best_scan(int64_t s, int64_t top, Each&& each) {
    int64_t c = 0, best_len = kNone, best = top;
    while (c < top) {
        for (;;) {  // move c off any predecessor that covers it
            int64_t next = c;
            each([&](int64_t po, int64_t pe) {
                if (po <= c && c < pe && pe > next) next = pe;
            });
            if (next == c) break;
            c = next;
        }
        if (c >= top) break;
        int64_t ns = kNone;  // c is uncovered and below the top: some start lies above it
        each([&](int64_t po, int64_t) {
            if (po > c && po < ns) ns = po;
        });
        const int64_t len = ns - c;
        if (len >= s && len < best_len) {
            best_len = len;
            best = c;
        }
        c = ns;
    }
    return best;
}

// Candidate test over buffered predecessors po/pe of length c (any memory space).
__device__ __forceinline__ bool span_free(const int64_t* po, const int64_t* pe, int32_t c, int64_t cand,
                                          int64_t s) {
    for (int32_t x = 0; x < c; ++x)
        if (po[x] < cand + s && cand < pe[x]) return false;
    return true;
}

__device__ __forceinline__ int64_t gap_at(const int64_t* po, const int64_t* pe, int32_t c, int64_t cand) {
    int64_t next = INT64_MAX;
    for (int32_t x = 0; x < c; ++x) {
        const int64_t o = po[x];
        if (o <= cand && cand < pe[x]) return -1;  // covered: not a gap start
        if (o >= cand && o < next) next = o;
    }
    return next - cand;
}

// Evaluates candidates k = first, first + stride, ... <= c (k = 0 is offset 0,
// k >= 1 is pe[k - 1]); returns this participant's best as (key, val):
// FIRST -> (cand, cand); BEST -> (gap length, cand).
__device__ __forceinline__ void eval_candidates(int32_t policy, const int64_t* po, const int64_t* pe, int32_t c,
                                                int64_t s, int64_t top, int32_t first, int32_t stride,
                                                int64_t& key, int64_t& val) {
    key = kNone;
    val = kNone;
    for (int32_t k = first; k <= c; k += stride) {
        const int64_t cand = k == 0 ? 0 : pe[k - 1];
        if (policy == MP_FIT_FIRST) {
            if (cand < key && span_free(po, pe, c, cand, s)) key = val = cand;
        } else {
            if (cand >= top) continue;
            const int64_t len = gap_at(po, pe, c, cand);
            if (len >= s && (len < key || (len == key && cand < val))) {
                key = len;
                val = cand;
            }
        }
    }
}

__device__ __forceinline__ int64_t resolve(int32_t policy, int64_t key, int64_t val, int64_t top) {
    if (policy == MP_FIT_FIRST) return key;  // offset `top` always fits, so key is finite
    return key == kNone ? top : val;
}

// ------------------------------------------------------------- tiers
// Each tier places one frontier tensor i and decrements the pending count of
// every successor.  A successor that reaches zero is queued for the next
// round, which starts after a barrier, i.e. after OFF[i] is visible.

// Thread tier: few predecessors; up to kRegPred are kept in registers, more
// are re-read from the lists (or the short window) on every pass.
template <typename I>
__device__ __forceinline__ void place_thread(const Trace<I>& m, int32_t policy, int32_t i, int32_t* s_tail) {
    const bool listed = (m.INFO[i] & kListedBit) != 0;
    const int64_t s = m.S[i];
    int64_t po[kRegPred], pe[kRegPred];
#pragma unroll
    for (int x = 0; x < kRegPred; ++x) po[x] = pe[x] = kNone;
    int32_t c = 0;
    int64_t top = 0;
    for_each_pred(m, i, listed, [&](int32_t j) {
        const int64_t o = m.OFF[j], e = o + m.S[j];
#pragma unroll
        for (int x = 0; x < kRegPred; ++x)
            if (x == c) {
                po[x] = o;
                pe[x] = e;
            }
        ++c;
        top = e > top ? e : top;
    });
    int64_t off;
    if (c <= kRegPred) {
        auto each = [&](auto&& fn) {
#pragma unroll
            for (int x = 0; x < kRegPred; ++x)
                if (x < c) fn(po[x], pe[x]);
        };
        off = policy == MP_FIT_FIRST ? fit_first_scan(s, each) : fit_best_scan(s, top, each);
    } else {
        auto each = [&](auto&& fn) {
            for_each_pred(m, i, listed, [&](int32_t j) { fn(m.OFF[j], m.OFF[j] + m.S[j]); });
        };
        off = policy == MP_FIT_FIRST ? fit_first_scan(s, each) : fit_best_scan(s, top, each);
    }
    m.OFF[i] = off;
    for_each_succ(m, i, listed, [&](int32_t j) { push_ready(m, j, s_tail); });
}

// Warp tier: predecessors gathered into this warp's buffer slice (capacity wcap).
template <typename I>
__device__ __forceinline__ void place_warp(const Trace<I>& m, int32_t policy, int32_t i, int64_t* bo, int64_t* be, int32_t wcap,
                           int32_t* s_tail, int32_t* s_err) {
    const int lane = threadIdx.x & 31;
    const Window w = window_of(m, i);
    int32_t cnt = 0;
    int64_t top = 0;
    for (int32_t kb = 0; kb < w.range; kb += 32) {
        const int32_t k = kb + lane;
        const int32_t j = k < w.range ? neighbour(m, i, w, k) : -1;
        bool hit = false;
        if (j >= 0) {
            hit = precedes(m, j, i);
            if (!hit) push_ready(m, j, s_tail);
        }
        const unsigned mask = __ballot_sync(0xffffffffu, hit);
        if (hit) {
            const int32_t pos = cnt + __popc(mask & ((1u << lane) - 1u));
            const int64_t o = m.OFF[j], e = o + m.S[j];
            if (pos < wcap) {
                bo[pos] = o;
                be[pos] = e;
            }
            top = e > top ? e : top;
        }
        cnt += __popc(mask);
    }
    if (cnt > wcap) {
        if (lane == 0) *s_err = 1;
        cnt = wcap;
    }
    top = warp_max_i64(top);
    __syncwarp();
    int64_t key, val;
    eval_candidates(policy, bo, be, cnt, m.S[i], top, lane, 32, key, val);
    warp_min_pair(key, val);
    if (lane == 0) m.OFF[i] = resolve(policy, key, val, top);
    __syncwarp();
}

// CTA tier: every thread of the block takes part (uniform control flow).
template <typename I>
__device__ __forceinline__ void place_cta(const Trace<I>& m, int32_t policy, int32_t i, int64_t* bo, int64_t* be, int32_t cap,
                          int32_t* s_tail, int32_t* s_cnt, unsigned long long* s_top, int32_t* s_err,
                          int64_t* red) {
    const Window w = window_of(m, i);
    if (threadIdx.x == 0) {
        *s_cnt = 0;
        *s_top = 0;
    }
    __syncthreads();
    for (int32_t k = threadIdx.x; k < w.range; k += blockDim.x) {
        const int32_t j = neighbour(m, i, w, k);
        if (j < 0) continue;
        if (!precedes(m, j, i)) {
            push_ready(m, j, s_tail);
            continue;
        }
        const int64_t o = m.OFF[j], e = o + m.S[j];
        const int32_t pos = atomicAdd(s_cnt, 1);
        if (pos < cap) {
            bo[pos] = o;
            be[pos] = e;
        } else {
            *s_err = 1;
        }
        atomicMax(s_top, (unsigned long long)e);
    }
    __syncthreads();
    int32_t c = *s_cnt;
    c = c < cap ? c : cap;
    const int64_t top = (int64_t)*s_top;
    int64_t key, val;
    eval_candidates(policy, bo, be, c, m.S[i], top, threadIdx.x, blockDim.x, key, val);
    block_min_pair(key, val, red);
    if (threadIdx.x == 0) m.OFF[i] = resolve(policy, key, val, top);
    __syncthreads();
}

template <typename I, bool kSmem>
__global__ void __launch_bounds__(kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal, kSmem ? 8 : 1)
k_plan(mp_batch bt, int32_t policy, int64_t* __restrict__ offsets, int64_t* __restrict__ plan_peak,
       int32_t* __restrict__ status, unsigned char* __restrict__ ws, size_t data_stride, size_t buf_offset,
       size_t buf_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[64];
    __shared__ int32_t s_nlong, s_lshort, s_tail, s_cnt, s_err, s_nw, s_nc;
    __shared__ unsigned long long s_top;
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const PlanLayout<I> L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * data_stride;
    Trace<I> m;
    m.S = reinterpret_cast<int64_t*>(base + L.s);
    m.OFF = reinterpret_cast<int64_t*>(base + L.off);
    m.PEND = reinterpret_cast<int32_t*>(base + L.pend);
    m.PRE = reinterpret_cast<int32_t*>(base + L.pre);
    m.SUE = reinterpret_cast<int32_t*>(base + L.sue);
    m.AUX = reinterpret_cast<int32_t*>(base + L.aux);
    m.BEND = reinterpret_cast<int32_t*>(base + L.bend);
    m.A = reinterpret_cast<I*>(base + L.a);
    m.F = reinterpret_cast<I*>(base + L.f);
    m.BYS = reinterpret_cast<I*>(base + L.bys);
    m.LONGL = reinterpret_cast<I*>(base + L.longl);
    m.QUEUE = reinterpret_cast<I*>(base + L.queue);
    m.PREDL = reinterpret_cast<I*>(base + L.predl);
    m.SUCCL = reinterpret_cast<I*>(base + L.succl);
    m.INFO = reinterpret_cast<uint8_t*>(base + L.info);
    m.n = n;
    const int32_t cap = bt.max_tensors;
    int64_t* bo = reinterpret_cast<int64_t*>(ws + buf_offset + (size_t)b * buf_stride);
    int64_t* be = bo + cap;
    const int nwarps = blockDim.x >> 5, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t wcap = cap / nwarps;

    // ---- phase 1: load, check, classify short / long
    for (int t = threadIdx.x; t < T; t += blockDim.x) m.BEND[t] = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        m.PEND[k] = 0;
        m.PRE[k] = 0;
        m.SUE[k] = 0;
    }
    if (threadIdx.x == 0) {
        s_nlong = 0;
        s_lshort = 0;
        s_tail = 0;
        s_err = 0;
        s_nw = 0;
        s_nc = 0;
    }
    __syncthreads();
    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    bool bad = false;
    uint64_t sum = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t s = __ldg(Sg + k);
        if (!tensor_ok(a, f, s, T)) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        m.A[k] = (I)a;
        m.F[k] = (I)f;
        m.S[k] = s;
        const int32_t life = f - a;
        if (life > kLongLife) {
            m.LONGL[atomicAdd(&s_nlong, 1)] = (I)k;
        } else {
            atomicAdd(m.BEND + a, 1);
            atomicMax(&s_lshort, life);
        }
    }
    bad = __syncthreads_or(bad);
    sum = block_sat_sum(sum, reinterpret_cast<uint64_t*>(red));
    if (bad || sum > (uint64_t)INT64_MAX) {
        if (threadIdx.x == 0) status[b] = bad ? MP_EINVAL : MP_EOVERFLOW;
        return;
    }
    m.nlong = s_nlong;
    m.lshort = s_lshort;
    const int32_t nshort = n - m.nlong;

    // ---- phase 2: counting sort of the short tensors by alloc step
    block_excl_scan_array<int32_t, 4>(m.BEND, T, reinterpret_cast<int32_t*>(red));
    for (int k = threadIdx.x; k < n; k += blockDim.x)
        if (m.F[k] - m.A[k] <= kLongLife) m.BYS[atomicAdd(m.BEND + m.A[k], 1)] = (I)k;
    __syncthreads();

    // ---- phase 3: every overlapping pair once.  Short-short pairs from the
    // earlier-starting member's forward window (one thread per short tensor),
    // counted, then written into exact lists after a prefix sum; pairs with a
    // long tensor from the long side (one warp per long tensor), counted only.
    auto short_pairs = [&](auto&& on_pair) {
        for (int32_t p = threadIdx.x; p < nshort; p += blockDim.x) {
            const int32_t i = m.BYS[p];
            const int32_t stop = m.BEND[m.F[i] - 1];
            for (int32_t q = p + 1; q < stop; ++q) {
                const int32_t j = m.BYS[q];
                if (precedes(m, i, j)) on_pair(i, j);
                else on_pair(j, i);
            }
        }
    };
    short_pairs([&](int32_t hi, int32_t lo) {
        atomicAdd(m.PRE + lo, 1);
        atomicAdd(m.SUE + hi, 1);
    });
    for (int32_t u = warp; u < m.nlong; u += nwarps) {
        const int32_t Lt = m.LONGL[u];
        const Window w = window_of(m, Lt);
        for (int32_t k = lane; k < w.nshort; k += 32) {
            const int32_t j = m.BYS[w.p0 + k];
            if (m.F[j] > w.ai) atomicAdd(m.PEND + (precedes(m, Lt, j) ? j : Lt), 1);
        }
        for (int32_t v = u + 1 + lane; v < m.nlong; v += 32) {
            const int32_t j = m.LONGL[v];
            if (m.A[j] < w.fi && m.F[j] > w.ai) atomicAdd(m.PEND + (precedes(m, Lt, j) ? j : Lt), 1);
        }
    }
    __syncthreads();
    for (int k = threadIdx.x; k < n; k += blockDim.x) m.PEND[k] += m.PRE[k];
    __syncthreads();
    const int32_t n_short_pairs = block_excl_scan_array<int32_t, 4>(m.PRE, n, reinterpret_cast<int32_t*>(red));
    block_excl_scan_array<int32_t, 4>(m.SUE, n, reinterpret_cast<int32_t*>(red));
    const bool lists = n_short_pairs <= kListCap * n;
    if (lists) {
        short_pairs([&](int32_t hi, int32_t lo) {
            m.PREDL[atomicAdd(m.PRE + lo, 1)] = (I)hi;
            m.SUCCL[atomicAdd(m.SUE + hi, 1)] = (I)lo;
        });
    }
    __syncthreads();

    // ---- phase 4: tiers and the first frontier
    for (int32_t i = threadIdx.x; i < n; i += blockDim.x) {
        const int32_t P = m.PEND[i];
        const bool listed = lists && (m.F[i] - m.A[i] <= kLongLife);
        int32_t pred_scan, succ_scan, range = 0;
        if (listed) {
            pred_scan = m.PRE[i] - (i ? m.PRE[i - 1] : 0) + m.nlong;
            succ_scan = m.SUE[i] - (i ? m.SUE[i - 1] : 0) + m.nlong;
        } else {
            range = window_of(m, i).range;
            pred_scan = succ_scan = range;
        }
        if (range == 0 && !(P <= kThreadMaxPred && pred_scan <= kThreadMaxScan && succ_scan <= kThreadMaxRange))
            range = window_of(m, i).range;
        const int32_t tier =
            (P <= kThreadMaxPred && pred_scan <= kThreadMaxScan && succ_scan <= kThreadMaxRange) ? kTierThread
            : (P <= wcap && range <= kWarpMaxRange)                                               ? kTierWarp
                                                                                                   : kTierCta;
        m.INFO[i] = (uint8_t)(tier | (listed ? kListedBit : 0));
        if (P == 0) enqueue(m, i, &s_tail);
    }

    // ---- phase 5: frontier rounds (at most n; each places >= 1 tensor).
    // Warp-tier tensors of the round are listed at the front of AUX, CTA-tier
    // tensors at the back.
    int32_t qh = 0;
    for (;;) {
        __syncthreads();
        const int32_t qt = s_tail < n ? s_tail : n;
        if (threadIdx.x == 0) {
            s_nw = 0;
            s_nc = 0;
        }
        __syncthreads();
        if (qt == qh) break;
        for (int32_t q = qh + threadIdx.x; q < qt; q += blockDim.x) {
            const int32_t i = m.QUEUE[q];
            const int32_t tier = m.INFO[i] & 3;
            if (tier == kTierThread) place_thread(m, policy, i, &s_tail);
            else if (tier == kTierWarp) m.AUX[atomicAdd(&s_nw, 1)] = i;
            else m.AUX[n - 1 - atomicAdd(&s_nc, 1)] = i;
        }
        __syncthreads();
        const int32_t nw = s_nw, nc = s_nc;
        for (int32_t q = warp; q < nw; q += nwarps)
            place_warp(m, policy, m.AUX[q], bo + (size_t)warp * wcap, be + (size_t)warp * wcap, wcap, &s_tail,
                       &s_err);
        if (nc > 0) {
            __syncthreads();
            for (int32_t q = 0; q < nc; ++q)
                place_cta(m, policy, m.AUX[n - 1 - q], bo, be, cap, &s_tail, &s_cnt, &s_top, &s_err, red);
        }
        qh = qt;
    }

    // ---- phase 6: offsets out, plan peak
    int64_t mx = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int64_t e = m.OFF[k] + m.S[k];
        offsets[tv.lo + k] = m.OFF[k];
        mx = e > mx ? e : mx;
    }
    mx = block_max_i64(mx, red);
    if (threadIdx.x == 0) {
        plan_peak[b] = mx;
        status[b] = (qh != n || s_tail != n || s_err) ? MP_EINTERNAL : MP_OK;
    }
}

struct PlanGeometry {
    bool smem, narrow;
    size_t data, data_stride, buf_offset, buf_stride, workspace;
};

// 16-bit indices when every id and step fits; shared memory when the trace's
// working set fits under the ceiling, else a workspace slice per trace.
PlanGeometry plan_geometry(const mp_batch& bt) {
    PlanGeometry g;
    g.narrow = bt.max_tensors <= 32767 && bt.max_steps <= 32767;
    g.data = g.narrow ? PlanLayout<int16_t>(bt.max_tensors, bt.max_steps).total
                      : PlanLayout<int32_t>(bt.max_tensors, bt.max_steps).total;
    g.smem = g.data <= kPlanSmemLimit;
    g.data_stride = g.smem ? 0 : g.data;
    g.buf_offset = (size_t)bt.n_traces * g.data_stride;
    g.buf_stride = align_up((size_t)bt.max_tensors * 16);
    g.workspace = bt.n_traces == 0 ? 0 : g.buf_offset + (size_t)bt.n_traces * g.buf_stride;
    return g;
}

template <typename I, bool kSmem>
cudaError_t launch_variant(const mp_batch& bt, const PlanGeometry& g, int32_t policy, int64_t* offsets,
                           int64_t* plan_peak, int32_t* status, unsigned char* ws, cudaStream_t stream) {
    const size_t smem = kSmem ? g.data : 0;
    if (kSmem) {
        cudaError_t e = set_smem_limit((const void*)k_plan<I, kSmem>, smem);
        if (e != cudaSuccess) return e;
    }
    k_plan<I, kSmem><<<(unsigned)bt.n_traces, kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal, smem, stream>>>(
        bt, policy, offsets, plan_peak, status, ws, g.data_stride, g.buf_offset, g.buf_stride);
    return cudaGetLastError();
}

}  // namespace

size_t plan_workspace_bytes(const mp_batch& bt) { return plan_geometry(bt).workspace; }

cudaError_t launch_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                        int32_t* status, void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const PlanGeometry g = plan_geometry(bt);
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    if (g.narrow)
        return g.smem ? launch_variant<int16_t, true>(bt, g, policy, offsets, plan_peak, status, ws, stream)
                      : launch_variant<int16_t, false>(bt, g, policy, offsets, plan_peak, status, ws, stream);
    return g.smem ? launch_variant<int32_t, true>(bt, g, policy, offsets, plan_peak, status, ws, stream)
                  : launch_variant<int32_t, false>(bt, g, policy, offsets, plan_peak, status, ws, stream);
}

}  // namespace mp
