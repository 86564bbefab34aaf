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
// PEND[i] = |P_i| counts unplaced predecessors, each round places the whole
// frontier (tensors in one frontier never overlap each other, so they are
// independent) and decrements the successors' counters, which pushes the
// tensors that became ready.  The number of rounds is the DAG's depth, not N.
// No sort is materialised: the priority order is used only as a comparator.
//
// Neighbour enumeration: short-lived tensors (life <= kLongLife) are
// counting-sorted by alloc step, so the short tensors overlapping i lie in the
// alloc-step window [alloc_i - Lshort + 1, free_i) (Lshort = longest short
// lifetime); long-lived tensors sit in a separate list scanned in full.
//
// Gap search without sorting: FIRST is the lowest offset o at which
// [o, o + s_i) meets no predecessor's [off_j, end_j); the answer is 0 or some
// end_j, so it is the smallest candidate c in {0} U {end_j} that conflicts
// with no predecessor.  BEST: a gap of the address-ordered scan starts at a
// candidate c that no predecessor covers (off_j <= c < end_j) and below the
// top (max end), and has length min{off_j >= c} - c; the smallest length
// >= s_i wins, the lowest start on ties, else the top.  Both forms are
// evaluated in parallel over candidates (thread, warp or CTA per tensor,
// chosen by |P_i| and the enumeration length).
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int32_t kLongLife = 32;           // lifetimes above this are "long" (performance knob only)
constexpr int32_t kThreadMaxPred = 4;       // thread tier: at most this many predecessors ...
constexpr int32_t kThreadMaxRange = 512;    // ... and at most this many enumeration items
constexpr int32_t kWarpMaxRange = 16384;    // warp tier: enumeration items
constexpr int32_t kTierShift = 28;             // NPRED = |P_i| | tier << 28 (|P_i| < 2^28)
enum : int32_t { kTierThread = 0, kTierWarp = 1, kTierCta = 2 };

struct PlanLayout {
    size_t s, off, a, f, bys, longl, pend, npred, queue, aux, bend, total;
    __host__ __device__ PlanLayout(int64_t n, int64_t T) {
        s = 0;
        off = s + align_up((size_t)n * 8);
        a = off + align_up((size_t)n * 8);
        f = a + align_up((size_t)n * 4);
        bys = f + align_up((size_t)n * 4);
        longl = bys + align_up((size_t)n * 4);
        pend = longl + align_up((size_t)n * 4);
        npred = pend + align_up((size_t)n * 4);
        queue = npred + align_up((size_t)n * 4);
        aux = queue + align_up((size_t)n * 4);
        bend = aux + align_up((size_t)n * 4);
        total = bend + align_up((size_t)T * 4);
    }
};

struct Trace {
    int64_t* S;
    int64_t* OFF;
    int32_t* A;
    int32_t* F;
    int32_t* BYS;    // short tensors sorted by alloc step
    int32_t* LONGL;  // long tensors, any order
    int32_t* PEND;   // unplaced predecessors
    int32_t* NPRED;  // |P_i| | tier << kTierShift, non-negative
    int32_t* QUEUE;  // topological order as it is discovered
    int32_t* BEND;   // BEND[t] = number of short tensors with alloc <= t
    int32_t n, nlong, lshort;
};

// j strictly precedes i in priority (size desc, alloc asc, id asc).
__device__ __forceinline__ bool precedes(const Trace& m, int32_t j, int32_t i) {
    const int64_t sj = m.S[j], si = m.S[i];
    if (sj != si) return sj > si;
    const int32_t aj = m.A[j], ai = m.A[i];
    if (aj != ai) return aj < ai;
    return j < i;
}

// Enumeration of i's lifetime neighbours: items [0, nshort) are the short
// tensors with alloc in [alloc_i - lshort + 1, free_i), items
// [nshort, nshort + nlong) the long list.
struct Window {
    int32_t ai, fi, p0, nshort, range;
};

__device__ __forceinline__ Window window_of(const Trace& m, int32_t i) {
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
__device__ __forceinline__ int32_t neighbour(const Trace& m, int32_t i, const Window& w, int32_t k) {
    if (k < w.nshort) {
        const int32_t j = m.BYS[w.p0 + k];  // alloc_j < free_i by the window
        return (j != i && m.F[j] > w.ai) ? j : -1;
    }
    const int32_t j = m.LONGL[k - w.nshort];
    return (j != i && m.A[j] < w.fi && m.F[j] > w.ai) ? j : -1;
}

// Appends j to the queue; every tensor is pushed exactly once, so the slot is
// always < n -- the guard only keeps a defect from writing out of bounds.
__device__ __forceinline__ void enqueue(const Trace& m, int32_t j, int32_t* s_tail) {
    const int32_t pos = atomicAdd(s_tail, 1);
    if (pos < m.n) m.QUEUE[pos] = j;
}

__device__ __forceinline__ void push_ready(const Trace& m, int32_t j, int32_t* s_tail) {
    if (atomicSub(m.PEND + j, 1) == 1) enqueue(m, j, s_tail);
}

// ------------------------------------------------------------- gap search

// Candidate test over predecessor arrays po/pe of length c (any memory space).
// FIRST: does [cand, cand + s) avoid every predecessor?
__device__ __forceinline__ bool span_free(const int64_t* po, const int64_t* pe, int32_t c, int64_t cand,
                                          int64_t s) {
    for (int32_t x = 0; x < c; ++x)
        if (po[x] < cand + s && cand < pe[x]) return false;
    return true;
}

// BEST: is cand uncovered, and how far is the next predecessor start >= cand?
__device__ __forceinline__ int64_t gap_at(const int64_t* po, const int64_t* pe, int32_t c, int64_t cand) {
    int64_t next = INT64_MAX;
    for (int32_t x = 0; x < c; ++x) {
        const int64_t o = po[x];
        if (o <= cand && cand < pe[x]) return -1;  // covered: not a gap start
        if (o >= cand && o < next) next = o;
    }
    return next - cand;
}

constexpr int64_t kNone = INT64_MAX;

// Evaluates candidates k = first, first + stride, ... < c + 1 (k = 0 is
// offset 0, k >= 1 is pe[k - 1]) and returns this participant's best as a
// (key, val) pair: FIRST -> (cand, cand); BEST -> (gap length, cand).
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
// Each tier places one frontier tensor i and, in the same pass over i's
// neighbours, decrements the pending count of every successor (a neighbour
// that i precedes).  A successor that reaches zero is queued for the next
// round, which starts after a barrier, i.e. after OFF[i] is visible.

// Thread tier: at most kThreadMaxPred predecessors, kept in registers.
__device__ void place_thread(const Trace& m, int32_t policy, int32_t i, int32_t* s_tail) {
    const Window w = window_of(m, i);
    int64_t po[kThreadMaxPred], pe[kThreadMaxPred];
#pragma unroll
    for (int x = 0; x < kThreadMaxPred; ++x) po[x] = pe[x] = 0;
    int32_t c = 0;
    int64_t top = 0;
    for (int32_t k = 0; k < w.range; ++k) {
        const int32_t j = neighbour(m, i, w, k);
        if (j < 0) continue;
        if (!precedes(m, j, i)) {
            push_ready(m, j, s_tail);
            continue;
        }
        const int64_t o = m.OFF[j], e = o + m.S[j];
#pragma unroll
        for (int x = 0; x < kThreadMaxPred; ++x)
            if (x == c) {
                po[x] = o;
                pe[x] = e;
            }
        ++c;
        top = e > top ? e : top;
    }
    const int64_t s = m.S[i];
    int64_t best_key = kNone, best_val = kNone;
#pragma unroll
    for (int k = 0; k <= kThreadMaxPred; ++k) {
        if (k > c) break;
        const int64_t cand = k == 0 ? 0 : pe[k - 1];
        bool ok = true;
        int64_t next = INT64_MAX;
#pragma unroll
        for (int x = 0; x < kThreadMaxPred; ++x) {
            if (x >= c) break;
            if (policy == MP_FIT_FIRST) {
                if (po[x] < cand + s && cand < pe[x]) ok = false;
            } else {
                if (po[x] <= cand && cand < pe[x]) ok = false;
                if (po[x] >= cand && po[x] < next) next = po[x];
            }
        }
        if (!ok) continue;
        if (policy == MP_FIT_FIRST) {
            if (cand < best_key) best_key = best_val = cand;
        } else if (cand < top) {
            const int64_t len = next - cand;
            if (len >= s && (len < best_key || (len == best_key && cand < best_val))) {
                best_key = len;
                best_val = cand;
            }
        }
    }
    m.OFF[i] = resolve(policy, best_key, best_val, top);
}

// Warp tier: predecessors gathered into this warp's buffer slice (capacity wcap).
__device__ void place_warp(const Trace& m, int32_t policy, int32_t i, int64_t* bo, int64_t* be, int32_t wcap,
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
__device__ void place_cta(const Trace& m, int32_t policy, int32_t i, int64_t* bo, int64_t* be, int32_t cap,
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

// Records |P_i| and the tier of tensor i, and seeds the queue with tensors
// that have no predecessor.
__device__ __forceinline__ void finish_count(const Trace& m, int32_t i, const Window& w, int32_t cnt, int32_t wcap,
                                             int32_t* s_tail) {
    const int32_t tier = (cnt <= kThreadMaxPred && w.range <= kThreadMaxRange) ? kTierThread
                         : (cnt <= wcap && w.range <= kWarpMaxRange)             ? kTierWarp
                                                                                 : kTierCta;
    m.NPRED[i] = cnt | (tier << kTierShift);
    m.PEND[i] = cnt;
    if (cnt == 0) enqueue(m, i, s_tail);
}

__device__ __forceinline__ int32_t count_preds(const Trace& m, int32_t i, const Window& w, int32_t first,
                                               int32_t stride) {
    int32_t cnt = 0;
    for (int32_t k = first; k < w.range; k += stride) {
        const int32_t j = neighbour(m, i, w, k);
        cnt += (j >= 0 && precedes(m, j, i)) ? 1 : 0;
    }
    return cnt;
}

template <bool kSmem>
__global__ void __launch_bounds__(kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal)
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
    const PlanLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * data_stride;
    Trace m;
    m.S = reinterpret_cast<int64_t*>(base + L.s);
    m.OFF = reinterpret_cast<int64_t*>(base + L.off);
    m.A = reinterpret_cast<int32_t*>(base + L.a);
    m.F = reinterpret_cast<int32_t*>(base + L.f);
    m.BYS = reinterpret_cast<int32_t*>(base + L.bys);
    m.LONGL = reinterpret_cast<int32_t*>(base + L.longl);
    m.PEND = reinterpret_cast<int32_t*>(base + L.pend);
    m.NPRED = reinterpret_cast<int32_t*>(base + L.npred);
    m.QUEUE = reinterpret_cast<int32_t*>(base + L.queue);
    m.BEND = reinterpret_cast<int32_t*>(base + L.bend);
    int32_t* AUX = reinterpret_cast<int32_t*>(base + L.aux);  // deferred (warp / CTA) tensors
    m.n = n;
    const int32_t cap = bt.max_tensors;
    int64_t* bo = reinterpret_cast<int64_t*>(ws + buf_offset + (size_t)b * buf_stride);
    int64_t* be = bo + cap;
    const int nwarps = blockDim.x >> 5, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t wcap = cap / nwarps;

    // ---- phase 1: load, check, classify short / long
    for (int t = threadIdx.x; t < T; t += blockDim.x) m.BEND[t] = 0;
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
        m.A[k] = a;
        m.F[k] = f;
        m.S[k] = s;
        const int32_t life = f - a;
        if (life > kLongLife) {
            m.LONGL[atomicAdd(&s_nlong, 1)] = k;
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

    // ---- phase 2: counting sort of the short tensors by alloc step
    block_excl_scan_array<int32_t, 4>(m.BEND, T, reinterpret_cast<int32_t*>(red));
    for (int k = threadIdx.x; k < n; k += blockDim.x)
        if (m.F[k] - m.A[k] <= kLongLife) m.BYS[atomicAdd(m.BEND + m.A[k], 1)] = k;
    __syncthreads();

    // ---- phase 3: |P_i| per tensor, tier, and the first frontier.  Tensors
    // with long enumeration windows are listed in AUX and counted by a warp
    // (or by the whole CTA) afterwards.
    for (int32_t i = threadIdx.x; i < n; i += blockDim.x) {
        const Window w = window_of(m, i);
        if (w.range > kThreadMaxRange) {
            AUX[atomicAdd(&s_nw, 1)] = i;
            continue;
        }
        finish_count(m, i, w, count_preds(m, i, w, 0, 1), wcap, &s_tail);
    }
    __syncthreads();
    const int32_t naux = s_nw;
    for (int32_t q = warp; q < naux; q += nwarps) {
        const int32_t i = AUX[q];
        const Window w = window_of(m, i);
        if (w.range > kWarpMaxRange) continue;
        int32_t cnt = count_preds(m, i, w, lane, 32);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
        if (lane == 0) finish_count(m, i, w, cnt, wcap, &s_tail);
    }
    __syncthreads();
    for (int32_t q = 0; q < naux; ++q) {
        const int32_t i = AUX[q];
        const Window w = window_of(m, i);
        if (w.range <= kWarpMaxRange) continue;
        if (threadIdx.x == 0) s_cnt = 0;
        __syncthreads();
        atomicAdd(&s_cnt, count_preds(m, i, w, threadIdx.x, blockDim.x));
        __syncthreads();
        if (threadIdx.x == 0) finish_count(m, i, w, s_cnt, wcap, &s_tail);
        __syncthreads();
    }

    // ---- phase 4: frontier rounds (at most n; each places >= 1 tensor).
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
            const int32_t tier = m.NPRED[i] >> kTierShift;
            if (tier == kTierThread) place_thread(m, policy, i, &s_tail);
            else if (tier == kTierWarp) AUX[atomicAdd(&s_nw, 1)] = i;
            else AUX[n - 1 - atomicAdd(&s_nc, 1)] = i;
        }
        __syncthreads();
        const int32_t nw = s_nw, nc = s_nc;
        for (int32_t q = warp; q < nw; q += nwarps)
            place_warp(m, policy, AUX[q], bo + (size_t)warp * wcap, be + (size_t)warp * wcap, wcap, &s_tail, &s_err);
        if (nc > 0) {
            __syncthreads();
            for (int32_t q = 0; q < nc; ++q)
                place_cta(m, policy, AUX[n - 1 - q], bo, be, cap, &s_tail, &s_cnt, &s_top, &s_err, red);
        }
        qh = qt;
    }

    // ---- phase 5: offsets out, plan peak
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
    bool smem;
    size_t data_stride, buf_offset, buf_stride, workspace;
};

PlanGeometry plan_geometry(const mp_batch& bt) {
    PlanGeometry g;
    const size_t data = PlanLayout(bt.max_tensors, bt.max_steps).total;
    g.smem = data <= kPlanSmemLimit;
    g.data_stride = g.smem ? 0 : data;
    g.buf_offset = (size_t)bt.n_traces * g.data_stride;
    g.buf_stride = align_up((size_t)bt.max_tensors * 16);
    g.workspace = bt.n_traces == 0 ? 0 : g.buf_offset + (size_t)bt.n_traces * g.buf_stride;
    return g;
}

}  // namespace

size_t plan_workspace_bytes(const mp_batch& bt) { return plan_geometry(bt).workspace; }

cudaError_t launch_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                        int32_t* status, void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const PlanGeometry g = plan_geometry(bt);
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    if (g.smem) {
        const size_t smem = PlanLayout(bt.max_tensors, bt.max_steps).total;
        cudaError_t e = set_smem_limit((const void*)k_plan<true>, smem);
        if (e != cudaSuccess) return e;
        k_plan<true><<<(unsigned)bt.n_traces, kPlanThreadsSmem, smem, stream>>>(
            bt, policy, offsets, plan_peak, status, ws, 0, g.buf_offset, g.buf_stride);
    } else {
        k_plan<false><<<(unsigned)bt.n_traces, kPlanThreadsGlobal, 0, stream>>>(
            bt, policy, offsets, plan_peak, status, ws, g.data_stride, g.buf_offset, g.buf_stride);
    }
    return cudaGetLastError();
}

}  // namespace mp
