// plan.cu -- stage 2: greedy_by_size offset assignment (Sec. 2.3; the default
// strategy of Sec. 3.2), and the fused pass that also builds the live profile
// (stage 1) and validates the plan (stage 3).
//
// Definition (sequential): take tensors in priority order -- size descending,
// alloc step ascending, id ascending -- and give each, among the already
// placed tensors whose lifetimes overlap its own, the first (FIRST) or the
// smallest fitting (BEST) gap in address order; above them all if none fits.
//
// Decomposition used here (exactly the same result).  Tensors whose lifetimes
// are linked by a chain of overlaps form a connected component; a tensor's
// offset depends only on tensors of its own component, so components are
// independent.  Sorted by alloc step (a counting sort into packed records),
// each component is a contiguous run: a new one starts at position p when no
// earlier tensor is still live at alloc(p) (the running maximum of free steps
// is <= alloc(p)).  Each component is then placed by the sequential
// definition itself:
//   - one tensor: offset 0;
//   - at most kThreadComp tensors: one thread.  First, one thread per member
//     (taken in the size-sorted component list, so that a warp's members
//     mostly share one component size) finds its priority rank inside its
//     component and the mask of members that both precede it and overlap its
//     lifetime (inside an alloc-ordered run, j < i overlaps i iff f_j > a_i,
//     and j > i iff a_j < f_i); then one thread per component visits the
//     members in rank order;
//   - at most kWarpComp tensors: one warp, a tensor per lane (two per lane
//     above 32); each lane counts the members that precede it, then the warp
//     places rank 0, 1, ... in turn with single-instruction warp reductions;
//   - larger: the whole CTA bitonic-sorts the component into priority order,
//     then places it tensor by tensor with a CTA-wide gather of the
//     overlapping placed tensors and a CTA-wide gap search.
// Thread-tier components are handed out largest size class first, so the
// lanes of a warp carry similar work.
//
// Gap search.  FIRST is the lowest offset o at which [o, o + s_i) meets no
// predecessor [off_j, end_j).  One thread: start at o = 0 and jump to the
// largest end among the predecessors that conflict with [o, o + s_i) until
// none does (every feasible offset >= o is >= each conflicting end, so the
// first conflict-free o is the lowest feasible one).  BEST walks the maximal
// free holes below the top (max end) in address order and keeps the smallest
// that fits, the lowest on ties, else the top.  CTA, few predecessors: every
// candidate in {0} U {end_j} is tested in parallel (FIRST: smallest
// conflict-free candidate; BEST: uncovered candidates c below the top scored
// by min{off_j >= c} - c).  CTA, many predecessors: FIRST by the jump method
// with block reductions; BEST by sorting the predecessors by offset and
// scanning the running maximum end, which exposes every gap at once.
//
// Byte width.  Every offset the method produces is 0 or the end of another
// tensor, so every offset, end and live-bytes value of a trace is at most the
// sum of its sizes.  Each call therefore launches the kernel twice: first with
// 32-bit byte arithmetic (W = uint32_t), which handles every trace whose sizes
// sum below 2^32 and marks the others deferred; then with 64-bit arithmetic,
// whose CTAs return at once unless their trace was deferred.
//
// Fused pass (mp_plan_and_validate): the difference array of the profile is
// built while the inputs are first read, scanned and written out before the
// records are scattered over the same shared memory; after placement every
// lifetime-overlapping pair is checked once, from its earlier member in alloc
// order, for address overlap.
#include <algorithm>

#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int32_t kThreadComp = 8;   // components up to this size: one thread
constexpr int32_t kWarpComp = 64;    // ... up to this size: one warp (a tensor or two per lane); else the CTA
constexpr int kCached = 4;           // tensors per thread kept in registers between the two input passes
constexpr int32_t kLongLife = 32;    // CTA tier: members living longer than this many steps are listed apart
constexpr int32_t kPredBuf = 512;    // CTA tier, data in the workspace: predecessors gathered per warp
constexpr int32_t kLongStage = 2048; // CTA tier, data in the workspace: long-lived members staged in shared memory
#ifdef MP_TEST_SPIN_CYCLES
constexpr long long kSpinCycles = MP_TEST_SPIN_CYCLES;  // test builds: a short bound
#else
constexpr long long kSpinCycles = 1ll << 31;  // a wait for another warp longer than this is a fault
#endif
constexpr int32_t kValWide = 64;     // validation: windows longer than this get a warp each
constexpr int32_t kFlowWarps = 16;   // warps that take members from a run's ready queue
constexpr int32_t kDeferComp = 1024;  // the 32-bit launch (data in shared memory) defers larger components
constexpr int32_t kSpinPolls = 64;   // polls of a queue slot before the waiting warp starts to sleep between them
constexpr int32_t kDeferred = -1;    // trace status between the two launches: needs 64-bit bytes

// Component size classes for the counting sort of the component list:
// classes 0 .. kThreadComp - 2 hold sizes kThreadComp down to 2 (thread tier,
// largest first), then one class for the warp tier and one for the CTA tier.
constexpr int kBinWarp = kThreadComp - 1;
constexpr int kBinCta = kThreadComp;
constexpr int kBins = kThreadComp + 1;

__host__ __device__ constexpr size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

__host__ __device__ inline int64_t pow2_at_least(int64_t x) {
    int64_t p = 1;
    while (p < x) p <<= 1;
    return p;
}

// Largest value of a byte word: "none" in minimum searches.
template <typename W>
__host__ __device__ constexpr W w_none() {
    return sizeof(W) == 4 ? (W)UINT32_MAX : (W)INT64_MAX;
}

// Difference-array layout: runs of kRun entries, each followed by kPad
// entries of padding, so that the 16-byte reads of eight lanes that scan
// kLane consecutive steps each fall in distinct banks.
template <typename W>
struct ProfGeom;
template <>
struct ProfGeom<int64_t> {
    static constexpr int kRun = 16, kPad = 2, kLane = 8;
};
template <>
struct ProfGeom<uint32_t> {
    static constexpr int kRun = 8, kPad = 4, kLane = 8;
};
template <typename W>
__host__ __device__ constexpr int32_t dpos(int32_t t) {
    return t + ProfGeom<W>::kPad * (int32_t)((uint32_t)t / ProfGeom<W>::kRun);
}
template <typename W>
__host__ __device__ constexpr size_t dpadded(size_t T) {
    return T + ProfGeom<W>::kPad * ((T + ProfGeom<W>::kRun - 1) / ProfGeom<W>::kRun);
}

// A tensor in alloc-step order.
template <typename I, typename W>
struct ARec {
    W s;
    I a, f, id, pad;
};

// Per-trace working set.  The records and the offsets (by alloc-order
// position) share their bytes with the profile's difference array, which is
// dead before the records are written.
template <typename I, typename W>
struct PlanLayout {
    size_t arec, offp, dprof, bend, sb, wt, lst, rp, ord, cnt, que, total;
    __host__ __device__ PlanLayout(int64_t n, int64_t T, bool fused) {
        constexpr bool cta_tier = true;
        arec = 0;
        offp = arec + align16((size_t)n * sizeof(ARec<I, W>));
        const size_t main_end = offp + align16((size_t)n * sizeof(W));
        dprof = 0;
        const size_t dend = fused ? align16(dpadded<W>((size_t)T) * sizeof(W)) : 0;
        bend = main_end > dend ? main_end : dend;
        sb = bend + align16((size_t)T * 4);
        wt = sb + align16((size_t)((n + 31) / 32) * 4);
        lst = wt + align16((size_t)((n + 31) / 32) * 4);
        rp = lst + align16((size_t)n * 4);  // the thread tier's ranks; later the CTA tier's long-lived ranks
        ord = rp + align16((size_t)n * (cta_tier ? 4 : 2));  // the CTA tier's priority order (int32)
        cnt = ord + (cta_tier ? align16((size_t)n * 4) : 0);  // the CTA tier's predecessor counts (int32)
        que = cnt + (cta_tier ? align16((size_t)n * 4) : 0);  // the CTA tier's ready queue (int32)
        total = align_up(que + (cta_tier ? align16((size_t)n * 4) : 0));
    }
};

// Outputs of one launch; the fused kernel also fills the profile, its peak,
// the verdict and the conflict pair (the last three pointers may be null).
struct PlanOut {
    int32_t policy;
    int64_t* offsets;
    int64_t* plan_peak;
    int32_t* status;
    int64_t* profile;
    int64_t* peak_lb;
    int32_t* verdict;
    int32_t* conflict;
};

// x strictly precedes y in priority (size desc, alloc asc, id asc).
template <typename R>
__device__ __forceinline__ bool precedes(const R& x, const R& y) {
    if (x.s != y.s) return x.s > y.s;
    if (x.a != y.a) return x.a < y.a;
    return x.id < y.id;
}

// The same order for 16-bit ids and steps and 32-bit sizes as one unsigned
// key, smallest first: the complemented size, then the alloc step, then the id.
template <typename R>
__device__ __forceinline__ uint64_t prio_key(const R& r) {
    return ((uint64_t)(~(uint32_t)r.s) << 32) | ((uint32_t)(uint16_t)r.a << 16) | (uint32_t)(uint16_t)r.id;
}
template <typename R>
__device__ __forceinline__ bool precedes_key(const R& x, uint64_t key_y) {
    constexpr bool kPacked = sizeof(x.s) == 4 && sizeof(x.a) == 2;
    if constexpr (kPacked) return prio_key(x) < key_y;
    return false;  // unused
}

// ------------------------------------------------------------- gap search

// FIRST by jumping: `each(fn)` calls fn(off, end) for every predecessor.
template <typename W, typename Each>
__device__ __forceinline__ W fit_first_scan(W s, Each&& each) {
    W o = 0;
    for (;;) {
        W next = o;
        each([&](W po, W pe) {
            if (po < o + s && o < pe && pe > next) next = pe;
        });
        if (next == o) return o;
        o = next;
    }
}

// BEST by walking the free holes below the top in address order.
template <typename W, typename Each>
__device__ __forceinline__ W fit_best_scan(W s, W top, Each&& each) {
    W c = 0, best_len = w_none<W>(), best = top;
    while (c < top) {
        for (;;) {  // move c off any predecessor that covers it
            W next = c;
            each([&](W po, W pe) {
                if (po <= c && c < pe && pe > next) next = pe;
            });
            if (next == c) break;
            c = next;
        }
        if (c >= top) break;
        W ns = w_none<W>();  // c is uncovered and below the top: some start lies above it
        each([&](W po, W) {
            if (po > c && po < ns) ns = po;
        });
        const W len = ns - c;
        if (len >= s && len < best_len) {
            best_len = len;
            best = c;
        }
        c = ns;
    }
    return best;
}

// ------------------------------------------------------------- one thread

__device__ __forceinline__ int nib(uint32_t x, int k) { return (int)((x >> (4 * k)) & 15u); }

// Places the component at alloc-order positions [p0, p0 + c), 2 <= c <=
// kThreadComp, with one thread, from its members' precomputed ranks and
// predecessor masks (RP[p] = rank | mask << 4); writes OFFP[p0 .. p0 + c) and
// returns the largest end.
template <typename I, typename W>
__device__ W place_thread(const ARec<I, W>* AR, const uint16_t* RP, W* OFFP, int32_t p0, int32_t c,
                          int32_t policy) {
    static_assert(kThreadComp <= 8, "ranks are packed into 4-bit fields of 32 bits, masks into 12 bits");
    uint32_t order = 0;  // field r = the member of rank r
    for (int k = 0; k < c; ++k) order |= (uint32_t)k << (4 * (RP[p0 + k] & 15));
    W mx = 0;
    for (int r = 0; r < c; ++r) {
        const int k = nib(order, r);
        const uint32_t m = RP[p0 + k] >> 4;  // placed already: they precede it
        const W s = AR[p0 + k].s;
        auto each = [&](auto&& fn) {
            for (uint32_t t = m; t; t &= t - 1) {
                const int q = __ffs(t) - 1;
                const W o = OFFP[p0 + q];
                fn(o, o + AR[p0 + q].s);
            }
        };
        W o;
        if (policy == MP_FIT_FIRST) {
            o = fit_first_scan<W>(s, each);
        } else {
            W top = 0;
            each([&](W, W pe) { top = pe > top ? pe : top; });
            o = fit_best_scan<W>(s, top, each);
        }
        OFFP[p0 + k] = o;
        mx = o + s > mx ? o + s : mx;
    }
    return mx;
}

// ------------------------------------------------------------- one warp

// Warp max / min of non-negative byte values: one 32-bit reduction, or two
// for 64-bit values (high words first, then the low words of the lanes
// holding the top high word).
__device__ __forceinline__ uint32_t warp_max_w(uint32_t v) { return __reduce_max_sync(0xffffffffu, v); }
__device__ __forceinline__ uint32_t warp_min_w(uint32_t v) { return __reduce_min_sync(0xffffffffu, v); }
__device__ __forceinline__ int64_t warp_max_w(int64_t v) {
    const unsigned hi = __reduce_max_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32));
    const unsigned lo = __reduce_max_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32) == hi ? (unsigned)v : 0u);
    return (int64_t)(((uint64_t)hi << 32) | lo);
}
__device__ __forceinline__ int64_t warp_min_w(int64_t v) {
    const unsigned hi = __reduce_min_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32));
    const unsigned lo = __reduce_min_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32) == hi ? (unsigned)v : ~0u);
    return (int64_t)(((uint64_t)hi << 32) | lo);
}

// BEST by one warp over the predecessor pairs each lane supplies through
// each(fn): the free holes below the top walked in address order, the
// smallest that fits kept, the lowest on ties, else the top.
template <typename W, typename Each>
__device__ W warp_best_fit(W s, Each&& each) {
    W top = 0;
    each([&](W, W pe) { top = pe > top ? pe : top; });
    top = warp_max_w(top);
    W c = 0, best_len = w_none<W>(), best = top;
    while (c < top) {
        for (;;) {  // move c off any predecessor that covers it
            W cov = 0;
            each([&](W po, W pe) {
                if (po <= c && c < pe && pe > cov) cov = pe;
            });
            cov = warp_max_w(cov);
            if (cov <= c) break;
            c = cov;
        }
        if (c >= top) break;
        W ns = w_none<W>();
        each([&](W po, W) {
            if (po > c && po < ns) ns = po;
        });
        ns = warp_min_w(ns);
        const W len = ns - c;
        if (len >= s && len < best_len) {
            best_len = len;
            best = c;
        }
        c = ns;
    }
    return best;
}

// Places the component at positions [p0, p0 + c), 32 < c <= 64, with one
// warp, two tensors per lane (positions lane and lane + 32), as place_warp
// does with one.  A single component of this size in a CTA holding tiny ones
// would otherwise go to the CTA tier and outlast every other CTA of its wave.
// Out of line: rarely taken, its code would crowd the hot loop's.
template <typename I, typename W>
__device__ __noinline__ W place_warp2(const ARec<I, W>* AR, W* OFFP, int32_t p0, int32_t c, int32_t policy) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    bool act[2];
    W s[2];
    int32_t a[2], f[2], id[2];
    int rank[2] = {0, 0};
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int32_t m = lane + 32 * k;
        act[k] = m < c;
        s[k] = 0;
        a[k] = f[k] = 0;
        id[k] = -1;
        if (act[k]) {
            const ARec<I, W> me = AR[p0 + m];
            s[k] = me.s;
            a[k] = (int32_t)me.a;
            f[k] = (int32_t)me.f;
            id[k] = (int32_t)me.id;
        }
    }
    for (int l = 0; l < 32; ++l) {
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const W sl = __shfl_sync(full, s[kk], l);
            const int32_t al = __shfl_sync(full, a[kk], l), il = __shfl_sync(full, id[kk], l);
            if (l + 32 * kk >= c) continue;
#pragma unroll
            for (int k = 0; k < 2; ++k)
                if (act[k] && !(l == lane && kk == k))
                    rank[k] += (sl != s[k] ? sl > s[k] : (al != a[k] ? al < a[k] : il < id[k])) ? 1 : 0;
        }
    }
    W off[2] = {0, 0}, end[2] = {0, 0};
    bool placed[2] = {false, false};
    for (int r = 0; r < c; ++r) {
        const unsigned b0 = __ballot_sync(full, act[0] && rank[0] == r);
        const unsigned b1 = __ballot_sync(full, act[1] && rank[1] == r);
        const int slot = b0 ? 0 : 1;
        const int src = __ffs(b0 ? b0 : b1) - 1;
        const int32_t ai = __shfl_sync(full, slot ? a[1] : a[0], src), fi = __shfl_sync(full, slot ? f[1] : f[0], src);
        const W si = __shfl_sync(full, slot ? s[1] : s[0], src);
        bool pred[2];
#pragma unroll
        for (int k = 0; k < 2; ++k) pred[k] = placed[k] && a[k] < fi && ai < f[k];  // placed: ranks below r
        W o = 0;
        if (policy == MP_FIT_FIRST) {
            for (;;) {
                W v = 0;
#pragma unroll
                for (int k = 0; k < 2; ++k)
                    if (pred[k] && off[k] < o + si && o < end[k] && end[k] > v) v = end[k];
                const W mx = warp_max_w(v);
                if (mx <= o) break;
                o = mx;
            }
        } else {
            W t = 0;
#pragma unroll
            for (int k = 0; k < 2; ++k)
                if (pred[k] && end[k] > t) t = end[k];
            const W top = warp_max_w(t);
            W cc = 0, best_len = w_none<W>();
            o = top;
            while (cc < top) {
                for (;;) {  // move cc off any predecessor that covers it
                    W v = 0;
#pragma unroll
                    for (int k = 0; k < 2; ++k)
                        if (pred[k] && off[k] <= cc && cc < end[k] && end[k] > v) v = end[k];
                    const W mx = warp_max_w(v);
                    if (mx <= cc) break;
                    cc = mx;
                }
                if (cc >= top) break;
                W v = w_none<W>();
#pragma unroll
                for (int k = 0; k < 2; ++k)
                    if (pred[k] && off[k] > cc && off[k] < v) v = off[k];
                const W ns = warp_min_w(v);
                const W len = ns - cc;
                if (len >= si && len < best_len) {
                    best_len = len;
                    o = cc;
                }
                cc = ns;
            }
        }
        if (lane == src) {
            if (slot == 0) {
                off[0] = o;
                end[0] = o + si;
                placed[0] = true;
            } else {
                off[1] = o;
                end[1] = o + si;
                placed[1] = true;
            }
        }
    }
    W mx = 0;
#pragma unroll
    for (int k = 0; k < 2; ++k)
        if (act[k]) {
            OFFP[p0 + lane + 32 * k] = off[k];
            mx = end[k] > mx ? end[k] : mx;
        }
    return warp_max_w(mx);
}

// Places the component at positions [p0, p0 + c), c <= 32, with one warp (a
// tensor per lane); every lane must call it.  Writes OFFP; returns the
// largest end.
template <typename I, typename W>
__device__ W place_warp(const ARec<I, W>* AR, W* OFFP, int32_t p0, int32_t c, int32_t policy) {
    if (c > 32) return place_warp2(AR, OFFP, p0, c, policy);
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    const bool act = lane < c;
    ARec<I, W> me;
    if (act) me = AR[p0 + lane];
    const W s = act ? me.s : 0;
    const int32_t a = act ? (int32_t)me.a : 0, f = act ? (int32_t)me.f : 0, id = act ? (int32_t)me.id : -1;
    int rank = 0;  // members that precede this one
    for (int l = 0; l < c; ++l) {
        const W sl = __shfl_sync(full, s, l);
        const int32_t al = __shfl_sync(full, a, l), il = __shfl_sync(full, id, l);
        if (act && l != lane) rank += (sl != s ? sl > s : (al != a ? al < a : il < id)) ? 1 : 0;
    }
    W off = 0, end = 0;
    bool placed = false;
    for (int r = 0; r < c; ++r) {
        const int src = __ffs(__ballot_sync(full, act && rank == r)) - 1;
        const int32_t ai = __shfl_sync(full, a, src), fi = __shfl_sync(full, f, src);
        const W si = __shfl_sync(full, s, src);
        const bool pred = placed && a < fi && ai < f;  // placed: ranks below r
        W o = 0;
        if (policy == MP_FIT_FIRST) {
            for (;;) {
                const W mx = warp_max_w((pred && off < o + si && o < end) ? end : (W)0);
                if (mx <= o) break;
                o = mx;
            }
        } else {
            const W top = warp_max_w(pred ? end : (W)0);
            W cc = 0, best_len = w_none<W>();
            o = top;
            while (cc < top) {
                for (;;) {  // move cc off any predecessor that covers it
                    const W mx = warp_max_w((pred && off <= cc && cc < end) ? end : (W)0);
                    if (mx <= cc) break;
                    cc = mx;
                }
                if (cc >= top) break;
                const W ns = warp_min_w((pred && off > cc) ? off : w_none<W>());
                const W len = ns - cc;
                if (len >= si && len < best_len) {
                    best_len = len;
                    o = cc;
                }
                cc = ns;
            }
        }
        if (lane == src) {
            off = o;
            end = o + si;
            placed = true;
        }
    }
    if (act) OFFP[p0 + lane] = off;
    return warp_max_w(act ? end : (W)0);
}

// ------------------------------------------------------------- whole CTA

// In-place bitonic sort of keys[0, len) (len a power of two) by `before`;
// every thread of the block must call it.
template <typename K, typename Before>
__device__ void block_bitonic_sort(K* keys, int32_t len, Before&& before) {
    for (int32_t k = 2; k <= len; k <<= 1) {
        for (int32_t j = k >> 1; j > 0; j >>= 1) {
            for (int32_t t = threadIdx.x; t < (len >> 1); t += blockDim.x) {
                const int32_t lo = 2 * t - (t & (j - 1));  // index with bit j clear
                const int32_t hi = lo + j;
                const bool up = (lo & k) == 0;
                const K x = keys[lo], y = keys[hi];
                if (up ? before(y, x) : before(x, y)) {
                    keys[lo] = y;
                    keys[hi] = x;
                }
            }
            __syncthreads();
        }
    }
}

// Exclusive prefix maximum (identity 0) of one value per thread; the block
// maximum is left in *total.  red: >= 33 slots.
__device__ __forceinline__ int64_t block_excl_max(int64_t v, int64_t* red, int64_t* total) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int64_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl = u > incl ? u : incl;
    }
    if (lane == 31) red[w] = incl;
    __syncthreads();
    if (w == 0) {
        int64_t xi = lane < nw ? red[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t u = __shfl_up_sync(0xffffffffu, xi, o);
            if (lane >= o) xi = u > xi ? u : xi;
        }
        const int64_t ex = __shfl_up_sync(0xffffffffu, xi, 1);
        if (lane < nw) red[lane] = lane == 0 ? 0 : ex;
        if (lane == nw - 1) red[32] = xi;
    }
    __syncthreads();
    const int64_t up = __shfl_up_sync(0xffffffffu, incl, 1);
    const int64_t wex = red[w];
    const int64_t r = lane == 0 ? wex : (up > wex ? up : wex);
    *total = red[32];
    __syncthreads();
    return r;
}

// Waits until another warp fills *slot (-1 until then) and returns it.
// Gives up after kSpinCycles, or at once when another warp has given up,
// and then sets *fail and returns -1.
__device__ __forceinline__ int32_t wait_slot(const volatile int32_t* slot, volatile int32_t* fail) {
    int32_t v = *slot;
    if (v >= 0) return v;
    const long long t0 = clock64();
    for (int32_t polls = 0;; ++polls) {
        if (polls >= kSpinPolls) __nanosleep(32);  // a short wait is the common case: poll first
        v = *slot;
        if (v >= 0) return v;
        if (*fail || clock64() - t0 > kSpinCycles) {
            *fail = 1;
            return -1;
        }
    }
}

// Position of the (n + 1)-th set bit of m (n < popc(m)).
__device__ __forceinline__ int nth_set_bit(unsigned m, int n) {
    int pos = 0;
#pragma unroll
    for (int step = 16; step > 0; step >>= 1)
        if (__popc(m & ((1u << (pos + step)) - 1u)) <= n) pos += step;
    return pos;
}

// A large component in the CTA tier.  Its members in priority order are
// ord[0, c) (positions); the long-lived ones (life above kLongLife steps) are
// at the ranks hr[0, nl), ascending.  With lw the longest life among the
// short-lived members (at most kLongLife), a short-lived member y overlaps x
// only if a_y > a_x - lw, so x can only overlap short-lived members allocated
// in (a_x - lw, f_x) -- a window of alloc order (BEND[t] = tensors allocated
// at or before t) -- or long-lived ones.  The
// variant with its data in the workspace stages the first kLongStage
// long-lived members in shared memory, by list index.
template <typename W>
struct LongStage {
    W* s;
    W* off;
    int32_t* a;
    int32_t* f;
    int32_t* id;
};
template <typename I, typename W>
struct Comp {
    const ARec<I, W>* AR;
    W* OFFP;
    const int32_t* BEND;
    const int32_t* ord;
    const int32_t* hr;
    int32_t p0, c, nl, lw;
    int32_t hold;  // test builds: a member never queued (-1: none)
    LongStage<W> st;
    bool staged;

    __device__ __forceinline__ void window(const ARec<I, W>& me, int32_t& w0, int32_t& w1) const {
        w0 = max(p0, (int32_t)me.a >= lw ? BEND[(int32_t)me.a - lw] : 0);
        w1 = min(p0 + c, BEND[(int32_t)me.f - 1]);
    }
    // The k-th long-lived member (record and offset; the offset once placed).
    __device__ __forceinline__ ARec<I, W> long_rec(int32_t k, int32_t& pos) const {
        pos = ord[hr[k]];
        if (staged) {
            ARec<I, W> o;
            o.s = st.s[k];
            o.a = (I)st.a[k];
            o.f = (I)st.f[k];
            o.id = (I)st.id[k];
            return o;
        }
        return AR[pos];
    }
    __device__ __forceinline__ W long_off(int32_t k, int32_t pos) const { return staged ? st.off[k] : OFFP[pos]; }
};

// Shared memory of the workspace variant: the long-lived stage, then a
// scratch area -- one predecessor buffer of kPredBuf (offset, end) pairs per
// warp while short-lived members are placed, the predecessors of a
// long-lived member while it is placed.
constexpr size_t kScratchBytes = 128 * 1024;
static_assert((kPlanThreadsWide / 32) * kPredBuf * 2 * sizeof(int64_t) <= kScratchBytes,
              "the per-warp predecessor buffers of the 64-bit launch fit in the scratch");
template <typename W>
__host__ __device__ constexpr size_t flow_smem_bytes() {
    return (size_t)kLongStage * (2 * sizeof(W) + 12) + kScratchBytes;
}
template <typename W>
__device__ __forceinline__ LongStage<W> long_stage(unsigned char* smem, W** scratch) {
    LongStage<W> st;
    W* w = reinterpret_cast<W*>(smem);
    st.s = w;
    st.off = w + kLongStage;
    *scratch = w + 2 * kLongStage;
    int32_t* i = reinterpret_cast<int32_t*>(reinterpret_cast<unsigned char*>(*scratch) + kScratchBytes);
    st.a = i;
    st.f = i + kLongStage;
    st.id = i + 2 * kLongStage;
    return st;
}

// Places the short-lived members of ranks [r0, r1) of a component (a run
// between two long-lived members; every lower rank is placed) with every
// warp of the CTA, in dependency order.  Each member counts its predecessors
// inside the run (the members that come first in priority and overlap its
// lifetime); members with none are queued.  A warp takes the next queued
// member, places it -- its offset depends on its predecessors' alone, so it
// is the sequential definition's -- publishes the offset, and decrements
// its successors inside the run, queuing those that reach zero.  Every
// member is queued exactly once, and the lowest unplaced rank is always
// ready, so the queue always fills.  Predecessors are gathered once: into a
// register per lane when there are at most 32, else into the warp's buffer
// pb (kPredBuf pairs) when there is one, else every pass of the gap search
// visits the candidates again.  Returns the largest end placed (lane 0).
template <typename I, typename W>
__device__ W place_run(const Comp<I, W>& cp, int32_t r0, int32_t r1, int32_t nl_placed, int32_t* CNT,
                       int32_t* QUE, W* pb, int32_t policy, int32_t* head, int32_t* tail, volatile int32_t* fail) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const unsigned lt_mask = (1u << lane) - 1u;
    const int32_t len = r1 - r0;
    volatile W* voff = cp.OFFP;
    volatile int32_t* vque = QUE;
    for (int32_t i = threadIdx.x; i < len; i += blockDim.x) QUE[i] = -1;
    if (threadIdx.x == 0) {
        *head = 0;
        *tail = 0;
    }
    __syncthreads();
    const ARec<I, W> R0 = cp.AR[cp.ord[r0]];
    const bool last = r1 == cp.c;
    const ARec<I, W> R1 = cp.AR[cp.ord[last ? r0 : r1]];
    auto is_short = [](const ARec<I, W>& o) { return (int32_t)o.f - (int32_t)o.a <= kLongLife; };
    auto overlaps = [](const ARec<I, W>& o, const ARec<I, W>& me) {
        return (int32_t)o.a < (int32_t)me.f && (int32_t)me.a < (int32_t)o.f;
    };
    auto push = [&](int32_t x) {
        if (x == cp.hold) return;  // only in test builds: the run then starves and its waits run out
        const int32_t at = atomicAdd(tail, 1);
        vque[at] = x;
    };
    // predecessors inside the run, a warp per member
    for (int32_t r = r0 + warp; r < r1; r += nwarps) {
        const int32_t x = cp.ord[r];
        const ARec<I, W> me = cp.AR[x];
        int32_t w0, w1;
        cp.window(me, w0, w1);
        int32_t cnt = 0;
        for (int32_t q0 = w0; q0 < w1; q0 += 32) {
            const int32_t q = q0 + lane;
            bool hit = false;
            if (q < w1 && q != x) {
                const ARec<I, W> o = cp.AR[q];
                hit = is_short(o) && overlaps(o, me) && precedes(o, me) && !precedes(o, R0);
            }
            cnt += __popc(__ballot_sync(full, hit));
        }
        if (lane == 0) {
            CNT[x] = cnt;
            if (cnt == 0) push(x);
        }
    }
    __syncthreads();

    W mx = 0;
    for (;;) {
        if (warp >= kFlowWarps) break;  // the rest wait at the barrier instead of polling the queue
        int32_t idx = 0;
        if (lane == 0) idx = atomicAdd(head, 1);
        idx = __shfl_sync(full, idx, 0);
        if (idx >= len) break;
        int32_t x = 0;
        if (lane == 0) x = wait_slot(vque + idx, fail);
        x = __shfl_sync(full, x, 0);
        if (x < 0) break;
        __threadfence_block();  // the predecessors' offsets after the queue entry
        const ARec<I, W> me = cp.AR[x];
        const W s = me.s;
        int32_t w0, w1;
        cp.window(me, w0, w1);
        // scan(fn): fn(is_pred, off, end) on every lane for each candidate, in
        // warp-uniform rounds
        auto scan = [&](auto&& fn) {
            for (int32_t q0 = w0; q0 < w1; q0 += 32) {
                const int32_t q = q0 + lane;
                bool hit = false;
                W po = 0, pe = 0;
                if (q < w1 && q != x) {
                    const ARec<I, W> o = cp.AR[q];
                    if (is_short(o) && overlaps(o, me) && precedes(o, me)) {
                        hit = true;
                        po = voff[q];
                        pe = po + o.s;
                    }
                }
                fn(hit, po, pe);
            }
            for (int32_t k0 = 0; k0 < nl_placed; k0 += 32) {
                const int32_t k = k0 + lane;
                bool hit = false;
                W po = 0, pe = 0;
                if (k < nl_placed) {
                    int32_t q;
                    const ARec<I, W> o = cp.long_rec(k, q);
                    if (overlaps(o, me)) {  // placed before this run: it precedes
                        hit = true;
                        po = cp.long_off(k, q);
                        pe = po + o.s;
                    }
                }
                fn(hit, po, pe);
            }
        };
        W rpo = 0, rpe = 0;  // register mode: lane l holds predecessor l
        int32_t np = 0;
        scan([&](bool hit, W po, W pe) {
            const unsigned bal = __ballot_sync(full, hit);
            if (bal == 0) return;
            const int32_t cnt = __popc(bal), rel = lane - np;
            const bool mine = rel >= 0 && rel < cnt;
            const int src = mine ? nth_set_bit(bal, rel) : lane;
            const W so = __shfl_sync(full, po, src), se = __shfl_sync(full, pe, src);
            if (mine) {
                rpo = so;
                rpe = se;
            }
            if (pb != nullptr) {
                const int32_t at = np + __popc(bal & lt_mask);
                if (hit && at < kPredBuf) {
                    pb[2 * at] = po;
                    pb[2 * at + 1] = pe;
                }
            }
            np += cnt;
        });
        __syncwarp();
        const int mode = np <= 32 ? 0 : (pb != nullptr && np <= kPredBuf ? 1 : 2);
        // each(fn): fn(off, end) for every predecessor held by this lane
        auto each = [&](auto&& fn) {
            if (mode == 0) {
                if (lane < np) fn(rpo, rpe);
            } else if (mode == 1) {
                for (int32_t k = lane; k < np; k += 32) fn(pb[2 * k], pb[2 * k + 1]);
            } else {
                scan([&](bool hit, W po, W pe) {
                    if (hit) fn(po, pe);
                });
            }
        };
        W o = 0;
        if (policy == MP_FIT_FIRST) {
            for (;;) {
                W hit = 0;
                each([&](W po, W pe) {
                    if (po < o + s && o < pe && pe > hit) hit = pe;
                });
                hit = warp_max_w(hit);
                if (hit <= o) break;
                o = hit;
            }
        } else {
            W top = 0;
            each([&](W, W pe) { top = pe > top ? pe : top; });
            top = warp_max_w(top);
            W cc = 0, best_len = w_none<W>();
            o = top;
            while (cc < top) {
                for (;;) {  // move cc off any predecessor that covers it
                    W cov = 0;
                    each([&](W po, W pe) {
                        if (po <= cc && cc < pe && pe > cov) cov = pe;
                    });
                    cov = warp_max_w(cov);
                    if (cov <= cc) break;
                    cc = cov;
                }
                if (cc >= top) break;
                W ns = w_none<W>();
                each([&](W po, W) {
                    if (po > cc && po < ns) ns = po;
                });
                ns = warp_min_w(ns);
                const W len2 = ns - cc;
                if (len2 >= s && len2 < best_len) {
                    best_len = len2;
                    o = cc;
                }
                cc = ns;
            }
        }
        if (lane == 0) {
            voff[x] = o;
            __threadfence_block();  // the offset before any successor can be queued
            mx = o + s > mx ? o + s : mx;
        }
        __syncwarp();
        // successors inside the run
        for (int32_t q0 = w0; q0 < w1; q0 += 32) {
            const int32_t q = q0 + lane;
            if (q < w1 && q != x) {
                const ARec<I, W> oq = cp.AR[q];
                if (is_short(oq) && overlaps(oq, me) && precedes(me, oq) && (last || precedes(oq, R1)) &&
                    atomicSub(CNT + q, 1) == 1)
                    push(q);
            }
        }
        __syncwarp();
    }
    return mx;
}

// Gap search over P predecessors already sorted by offset (off(x), end(x)):
// the gap before the x-th is its offset minus the largest end before it.
// FIRST takes the lowest offset whose gap fits, BEST the smallest fitting gap
// (the lowest offset on ties); with no fitting gap, the largest end.
template <typename Off, typename End>
__device__ int64_t sorted_gap(int32_t P, int64_t s, int32_t policy, Off&& off, End&& end, int64_t* red) {
    const int32_t chunk = (P + blockDim.x - 1) / blockDim.x;
    const int32_t k0 = min(P, (int32_t)threadIdx.x * chunk), k1 = min(P, k0 + chunk);
    int64_t local = 0;
    for (int32_t x = k0; x < k1; ++x) local = max(local, end(x));
    int64_t top;
    int64_t prev = block_excl_max(local, red, &top);
    int64_t key = INT64_MAX, val = INT64_MAX;
    for (int32_t x = k0; x < k1; ++x) {
        const int64_t gl = off(x) - prev;
        if (gl >= s) {
            const int64_t kx = policy == MP_FIT_FIRST ? prev : gl;  // prev grows with x
            if (kx < key || (kx == key && prev < val)) {
                key = kx;
                val = prev;
            }
        }
        prev = max(prev, end(x));
    }
    block_min_pair(key, val, red);
    return key == INT64_MAX ? top : val;
}

// Places the k-th long-lived member of a component (every lower rank placed)
// with the whole CTA.  Its predecessors -- the short-lived members of its
// window that precede it and every long-lived member of lower rank, hr[0, k),
// that overlaps it -- are gathered: with the data in shared memory as
// positions in idx (2n entries), otherwise as (offset, end) pairs in the
// shared scratch (sbuf, up to scap pairs) or else in bo / be.  FIRST then
// jumps to the largest conflicting end until nothing conflicts (a block
// reduction per jump); BEST sorts them by offset and searches the gaps in
// one pass.  Returns the offset (every thread).
template <typename I, typename W, bool kSmem>
__device__ W place_heavy(const Comp<I, W>& cp, int32_t k, int32_t policy, int32_t* idx, W* sbuf, int32_t scap,
                         int64_t* bo, int64_t* be, int64_t* red, int32_t* cnt) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    int32_t p;
    const ARec<I, W> me = cp.long_rec(k, p);
    const int32_t a = me.a, f = me.f;
    const int64_t s = (int64_t)me.s;
    int32_t w0, w1;
    cp.window(me, w0, w1);
    const int32_t nw = max(0, w1 - w0), ncand = nw + k;
    if (threadIdx.x == 0) *cnt = 0;
    __syncthreads();
    for (int32_t x0 = (int32_t)(threadIdx.x & ~31u); x0 < ncand; x0 += blockDim.x) {  // warp-uniform rounds
        const int32_t x = x0 + lane;
        bool hit = false;
        int32_t q = -1;
        int64_t po = 0, pe = 0;
        if (x < nw) {
            q = w0 + x;
            if (q != p) {
                const ARec<I, W> o = cp.AR[q];
                hit = (int32_t)o.f - (int32_t)o.a <= kLongLife && (int32_t)o.a < f && a < (int32_t)o.f &&
                      precedes(o, me);
                if (hit && !kSmem) {
                    po = (int64_t)cp.OFFP[q];
                    pe = po + (int64_t)o.s;
                }
            }
        } else if (x < ncand) {
            const ARec<I, W> o = cp.long_rec(x - nw, q);
            hit = (int32_t)o.a < f && a < (int32_t)o.f;
            if (hit && !kSmem) {
                po = (int64_t)cp.long_off(x - nw, q);
                pe = po + (int64_t)o.s;
            }
        }
        const unsigned bal = __ballot_sync(full, hit);
        if (bal) {
            int32_t at = 0;
            if (lane == 0) at = atomicAdd(cnt, __popc(bal));
            at = __shfl_sync(full, at, 0) + __popc(bal & ((1u << lane) - 1u));
            if (hit) {
                if (kSmem) {
                    idx[at] = q;
                } else if (at < scap) {
                    sbuf[2 * at] = (W)po;
                    sbuf[2 * at + 1] = (W)pe;
                } else {
                    bo[at] = po;
                    be[at] = pe;
                }
            }
        }
    }
    __syncthreads();
    const int32_t P = *cnt;
    const int32_t plen = (int32_t)pow2_at_least(P);
    int64_t off;
    if (kSmem && policy == MP_FIT_FIRST) {  // jump over the gathered positions
        const W* O = cp.OFFP;
        int64_t o = 0;
        for (;;) {
            int64_t next = o;
            for (int32_t x = threadIdx.x; x < P; x += blockDim.x) {
                const int32_t q = idx[x];
                const int64_t po = (int64_t)O[q], pe = po + (int64_t)cp.AR[q].s;
                if (po < o + s && o < pe && pe > next) next = pe;
            }
            next = block_max_i64(next, red);
            if (next == o) break;
            o = next;
        }
        off = o;
    } else if (policy == MP_FIT_FIRST) {  // jump over the gathered pairs
        int64_t o = 0;
        for (;;) {
            int64_t next = o;
            for (int32_t x = threadIdx.x; x < P; x += blockDim.x) {
                const int64_t po = x < scap ? (int64_t)sbuf[2 * x] : bo[x];
                const int64_t pe = x < scap ? (int64_t)sbuf[2 * x + 1] : be[x];
                if (po < o + s && o < pe && pe > next) next = pe;
            }
            next = block_max_i64(next, red);
            if (next == o) break;
            o = next;
        }
        off = o;
    } else if (kSmem) {  // sort positions by offset (-1 pads sort last)
        for (int32_t x = P + threadIdx.x; x < plen; x += blockDim.x) idx[x] = -1;
        __syncthreads();
        const W* O = cp.OFFP;
        block_bitonic_sort(idx, plen, [&](int32_t x, int32_t y) { return y < 0 ? x >= 0 : (x >= 0 && O[x] < O[y]); });
        off = sorted_gap(P, s, policy, [&](int32_t x) { return (int64_t)O[idx[x]]; },
                         [&](int32_t x) { return (int64_t)O[idx[x]] + (int64_t)cp.AR[idx[x]].s; }, red);
    } else if (plen <= scap) {  // sort the pairs in shared memory
        for (int32_t x = P + threadIdx.x; x < plen; x += blockDim.x) {
            sbuf[2 * x] = w_none<W>();
            sbuf[2 * x + 1] = w_none<W>();
        }
        __syncthreads();
        for (int32_t kk = 2; kk <= plen; kk <<= 1) {
            for (int32_t j = kk >> 1; j > 0; j >>= 1) {
                for (int32_t t = threadIdx.x; t < (plen >> 1); t += blockDim.x) {
                    const int32_t lo = 2 * t - (t & (j - 1)), hi = lo + j;
                    const bool up = (lo & kk) == 0;
                    const W xo = sbuf[2 * lo], yo = sbuf[2 * hi];
                    if (up ? yo < xo : xo < yo) {
                        const W xe = sbuf[2 * lo + 1];
                        sbuf[2 * lo] = yo;
                        sbuf[2 * hi] = xo;
                        sbuf[2 * lo + 1] = sbuf[2 * hi + 1];
                        sbuf[2 * hi + 1] = xe;
                    }
                }
                __syncthreads();
            }
        }
        off = sorted_gap(P, s, policy, [&](int32_t x) { return (int64_t)sbuf[2 * x]; },
                         [&](int32_t x) { return (int64_t)sbuf[2 * x + 1]; }, red);
    } else {  // too many for the scratch: all pairs to bo / be, sorted there
        for (int32_t x = threadIdx.x; x < min(P, scap); x += blockDim.x) {
            bo[x] = (int64_t)sbuf[2 * x];
            be[x] = (int64_t)sbuf[2 * x + 1];
        }
        for (int32_t x = P + threadIdx.x; x < plen; x += blockDim.x) {
            bo[x] = INT64_MAX;
            be[x] = INT64_MAX;
        }
        __syncthreads();
        for (int32_t kk = 2; kk <= plen; kk <<= 1) {
            for (int32_t j = kk >> 1; j > 0; j >>= 1) {
                for (int32_t t = threadIdx.x; t < (plen >> 1); t += blockDim.x) {
                    const int32_t lo = 2 * t - (t & (j - 1)), hi = lo + j;
                    const bool up = (lo & kk) == 0;
                    const int64_t xo = bo[lo], yo = bo[hi];
                    if (up ? yo < xo : xo < yo) {
                        const int64_t xe = be[lo];
                        bo[lo] = yo;
                        bo[hi] = xo;
                        be[lo] = be[hi];
                        be[hi] = xe;
                    }
                }
                __syncthreads();
            }
        }
        off = sorted_gap(P, s, policy, [&](int32_t x) { return bo[x]; }, [&](int32_t x) { return be[x]; }, red);
    }
    if (threadIdx.x == 0) {
        cp.OFFP[p] = (W)off;
        if (cp.staged) cp.st.off[k] = (W)off;
    }
    __syncthreads();
    return (W)off;
}

// ------------------------------------------------------------- components

// Component lookups over the start flags SB (n positions, one bit each).
// Traces of more than kWordWalk words have a per-word table instead of walks
// over SB: -NW[w] is the first start in words w.. (n if none); without the
// table NW is null.
constexpr int32_t kWordWalk = 32;

// Size of the component starting at position p: distance to the next start.
__device__ __forceinline__ int32_t comp_size(const uint32_t* SB, const int32_t* NW, int32_t p, int32_t n) {
    int32_t w = p >> 5;
    const int32_t nwords = (n + 31) >> 5;
    uint32_t m = SB[w] & ~((2u << (p & 31)) - 1u);  // start flags after p in its word
    if (m) return (w << 5) + __ffs(m) - 1 - p;
    if (NW) return (w + 1 < nwords ? -NW[w + 1] : n) - p;
    while (m == 0) {
        if (++w >= nwords) return n - p;
        m = SB[w];
    }
    return (w << 5) + __ffs(m) - 1 - p;
}

// In-place inclusive prefix maximum of x[0, len) by the whole block; with
// `reverse`, taken from x[len - 1] down to x[0].  red: >= 33 slots.
__device__ void block_scan_max_i32(int32_t* x, int32_t len, bool reverse, int32_t* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    int32_t carry = INT32_MIN;
    for (int32_t base = 0; base < len; base += blockDim.x) {
        const int32_t i = base + (int32_t)threadIdx.x;
        const int32_t at = reverse ? len - 1 - i : i;
        int32_t v = i < len ? x[at] : INT32_MIN;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t u = __shfl_up_sync(0xffffffffu, v, o);
            if (lane >= o) v = max(v, u);
        }
        if (lane == 31) red[w] = v;
        __syncthreads();
        if (w == 0) {
            int32_t xi = lane < nw ? red[lane] : INT32_MIN;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t u = __shfl_up_sync(0xffffffffu, xi, o);
                if (lane >= o) xi = max(xi, u);
            }
            if (lane < nw) red[lane] = xi;
        }
        __syncthreads();
        v = max(v, max(carry, w == 0 ? INT32_MIN : red[w - 1]));
        if (i < len) x[at] = v;
        carry = max(carry, red[nw - 1]);
        __syncthreads();
    }
}

// Size class of a component of c >= 2 tensors.
__device__ __forceinline__ int comp_bin(int32_t c) {
    return c > kWarpComp ? kBinCta : c > kThreadComp ? kBinWarp : kThreadComp - c;
}

// Adds v into a difference-array entry: 64-bit as two 32-bit atomics, 32-bit
// modulo 2^32 (exact once every add is in, since the true value fits).
__device__ __forceinline__ void d_add(int64_t* d, int64_t v) { atomic_add_u64_split(d, (uint64_t)v); }
__device__ __forceinline__ void d_add(uint32_t* d, int64_t v) { atomicAdd(d, (uint32_t)v); }

// Block exclusive scan of one byte word per thread (uint32 words may not
// wrap: every prefix of a trace's profile is below 2^32 on the 32-bit path).
template <typename W>
__device__ __forceinline__ W block_excl_scan_w(W v, int64_t* red, W* total) {
    return block_excl_scan<W>(v, reinterpret_cast<W*>(red), total);
}

// Components of more than kWalkMin members without long-lived ones are walked
// by one warp (walk_comp): cheapest when the dependencies form long chains,
// as in a network whose activations are all alike.  Smaller ones go to the
// ready-queue runs, whose warps overlap the independent members of a shallow
// dependency graph.
constexpr int32_t kWalkMin = 64;

// A window of more than this many alloc-order positions has no predecessor
// mask; the walk then tests its candidates on every pass.
constexpr int32_t kMaskBits = 64;
constexpr int32_t kUnmasked = 1 << 30;  // flag in the window start word

// Walks a component none of whose members lives longer than kLongLife steps
// with one warp, in priority order: ord[r] is the member of rank r, W0[x] the
// first position of member x's window (with kUnmasked when it has no mask) and
// PM[x] the mask of its predecessors in the window, both computed beforehand
// by the whole CTA.  Every predecessor of a member was placed earlier in the
// same walk, so the gap search sees final offsets: this is the sequential
// definition itself.  Lane l holds the predecessors at window positions l and
// l + 32, so a member costs one parallel load and a few warp reductions.  The
// next member's entries are loaded while the current one is placed (they do
// not depend on any offset).  Every lane must call it; returns this lane's
// largest end.
template <typename I, typename W>
__device__ W walk_comp(const ARec<I, W>* AR, W* OFFP, const int32_t* BEND, const int32_t* ord, const int32_t* W0,
                       const uint64_t* PM, int32_t p0, int32_t c, int32_t policy) {
    const int lane = threadIdx.x & 31;
    volatile W* voff = OFFP;
    W mx = 0;
    int32_t xn = c > 0 ? ord[0] : 0;
    ARec<I, W> men = AR[xn];
    int32_t wvn = W0[xn];
    uint64_t pmn = PM[xn];
    for (int32_t r = 0; r < c; ++r) {
        const int32_t x = xn;
        const ARec<I, W> me = men;
        const int32_t wv = wvn;
        const uint64_t pm = pmn;
        if (r + 1 < c) {
            xn = ord[r + 1];
            men = AR[xn];
            wvn = W0[xn];
            pmn = PM[xn];
        }
        const int32_t w0 = wv & (kUnmasked - 1);
        W o;
        if (!(wv & kUnmasked)) {
            // this lane's predecessors: window positions lane and lane + 32
            const bool h1 = (pm >> lane) & 1ull, h2 = (pm >> (lane + 32)) & 1ull;
            W o1 = 0, e1 = 0, o2 = 0, e2 = 0;  // an empty [0, 0) never conflicts
            if (h1) {
                o1 = voff[w0 + lane];
                e1 = (W)(o1 + AR[w0 + lane].s);
            }
            if (h2) {
                o2 = voff[w0 + lane + 32];
                e2 = (W)(o2 + AR[w0 + lane + 32].s);
            }
            auto each = [&](auto&& fn) {
                fn(o1, e1);
                fn(o2, e2);
            };
            if (policy == MP_FIT_FIRST) {
                o = 0;
                for (;;) {
                    W hit = 0;
                    each([&](W po, W pe) {
                        if (po < o + me.s && o < pe && pe > hit) hit = pe;
                    });
                    hit = warp_max_w(hit);
                    if (hit <= o) break;
                    o = hit;
                }
            } else {
                o = warp_best_fit<W>(me.s, each);
            }
        } else {  // a window too wide for a mask: its candidates tested on every pass
            const int32_t w1 = min(p0 + c, BEND[(int32_t)me.f - 1]);
            auto each = [&](auto&& fn) {
                for (int32_t q = w0 + lane; q < w1; q += 32) {
                    if (q == x) continue;
                    const ARec<I, W> oq = AR[q];
                    if ((int32_t)oq.a < (int32_t)me.f && (int32_t)me.a < (int32_t)oq.f && precedes(oq, me)) {
                        const W po = voff[q];
                        fn(po, (W)(po + oq.s));
                    }
                }
            };
            if (policy == MP_FIT_FIRST) {
                o = 0;
                for (;;) {
                    W hit = 0;
                    each([&](W po, W pe) {
                        if (po < o + me.s && o < pe && pe > hit) hit = pe;
                    });
                    hit = warp_max_w(hit);
                    if (hit <= o) break;
                    o = hit;
                }
            } else {
                o = warp_best_fit<W>(me.s, each);
            }
        }
        if (lane == 0) voff[x] = o;
        __syncwarp();
        mx = o + me.s > mx ? o + me.s : mx;
    }
    return mx;
}

// Places the nx large components starting at LST[0, nx) (the 32-bit launch
// defers traces with components above kDeferComp, and with its data in the
// workspace, every trace that needs this tier).  Each is first sorted into
// priority order by the whole CTA.  Components of more than kWalkMin members
// that all live at most kLongLife steps are then placed concurrently, one
// warp walking each (walk_comp).  In the others the long-lived members (if
// any) cut the priority
// order into runs of short-lived ones, which the warps place together from a
// ready queue, each long-lived one then by the whole CTA.  Returns this
// thread's largest end.
template <typename I, typename W, bool kSmem>
__device__ __forceinline__ W large_tier(const ARec<I, W>* AR, W* OFFP, const int32_t* BEND, const uint32_t* SB,
                                     const int32_t* NW, const int32_t* LST, int32_t nx, int32_t n, int32_t* ORD, int32_t* HR, int32_t* CNT, int32_t* QUE, int64_t* bo, int64_t* be,
                                     unsigned char* smem_raw, int32_t policy, int64_t* red, int32_t* s_cnt,
                                     int32_t* s_tail, int32_t* s_fail, int32_t hold) {
    const int warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    W mx = 0;
    W* scratch = nullptr;
    const LongStage<W> st = long_stage<W>(smem_raw, &scratch);
    // 1. every large component sorted into priority order: ORD[p0 + r] is the
    // position of its member of rank r
    for (int32_t qc = 0; qc < nx; ++qc) {
        const int32_t p0 = LST[qc], sz = comp_size(SB, NW, p0, n);
        const int32_t len = (int32_t)pow2_at_least(sz);
        // the sort buffer: with the data in shared memory the cnt and que
        // regions (2n entries, len <= 2n; free until step 3), else the
        // long-lived ranks' buffer (max_tensors rounded up to a power of two);
        // neither overlaps ORD
        int32_t* sortbuf = kSmem ? CNT : HR;
        __syncthreads();  // the thread tier's RP, and the previous component's buffer, are dead
        for (int32_t x = threadIdx.x; x < len; x += blockDim.x) sortbuf[x] = x < sz ? p0 + x : -1;
        __syncthreads();
        block_bitonic_sort(sortbuf, len, [&](int32_t x, int32_t y) {  // sentinels (-1) sort last
            return y < 0 ? x >= 0 : (x >= 0 && precedes(AR[x], AR[y]));
        });
        for (int32_t r = threadIdx.x; r < sz; r += blockDim.x) ORD[p0 + r] = sortbuf[r];
    }
    __syncthreads();
    // 2. components of more than kWalkMin members without long-lived ones.  First the whole CTA gives
    // every member its window and the mask of its predecessors there (W0
    // aliases HR, PM the CNT and QUE words, both free until step 3; W0[p0] = -1
    // marks a component left to step 3); then one warp walks each component,
    // all components at once.
    {
    int32_t* W0 = HR;
    uint64_t* PM = reinterpret_cast<uint64_t*>(CNT);
    for (int32_t qc = 0; qc < nx; ++qc) {
        const int32_t p0 = LST[qc], sz = comp_size(SB, NW, p0, n);
        int32_t any_long = 0, lw = 1;
        for (int32_t k = threadIdx.x; k < sz; k += blockDim.x) {
            const int32_t life = (int32_t)AR[p0 + k].f - (int32_t)AR[p0 + k].a;
            any_long |= life > kLongLife ? 1 : 0;
            if (life <= kLongLife) lw = max(lw, life);
        }
        if (__syncthreads_or(any_long) || sz <= kWalkMin) {
            if (threadIdx.x == 0) W0[p0] = -1;
            continue;
        }
        int64_t lw_max;
        block_excl_max((int64_t)lw, red, &lw_max);
        const int32_t lwc = (int32_t)lw_max;
        for (int32_t x = p0 + threadIdx.x; x < p0 + sz; x += blockDim.x) {
            const ARec<I, W> me = AR[x];
            const int32_t w0 = max(p0, (int32_t)me.a >= lwc ? BEND[(int32_t)me.a - lwc] : 0);
            const int32_t w1 = min(p0 + sz, BEND[(int32_t)me.f - 1]);
            uint64_t pm = 0;
            if (w1 - w0 <= kMaskBits) {
                for (int32_t q = w0; q < w1; ++q) {
                    if (q == x) continue;
                    const ARec<I, W> o = AR[q];
                    if ((int32_t)o.a < (int32_t)me.f && (int32_t)me.a < (int32_t)o.f && precedes(o, me))
                        pm |= 1ull << (q - w0);
                }
            }
            W0[x] = w0 | (w1 - w0 <= kMaskBits ? 0 : kUnmasked);
            PM[x] = pm;
        }
    }
    __syncthreads();
    for (int32_t qc = warp; qc < nx; qc += nwarps) {  // a warp per component
        const int32_t p0 = LST[qc];
        if (W0[p0] < 0) continue;
        const W e = walk_comp<I, W>(AR, OFFP, BEND, ORD + p0, W0, PM, p0, comp_size(SB, NW, p0, n), policy);
        mx = max(mx, e);
    }
    __syncthreads();
    }
    // 3. the other components, one after the other: their long-lived members
    // (if any) cut the priority order into runs of short-lived ones, which the
    // warps place together, each long-lived one then by the whole CTA
    for (int32_t qc = 0; qc < nx; ++qc) {
        const int32_t p0 = LST[qc];
        const int32_t sz = comp_size(SB, NW, p0, n);
        const int32_t* ord = ORD + p0;
        __syncthreads();
        int32_t nl = 0, lw = 1;
        for (int32_t r0 = 0; r0 < sz; r0 += blockDim.x) {
            const int32_t r = r0 + threadIdx.x;
            ARec<I, W> rx;
            int32_t flag = 0;
            if (r < sz) {
                rx = AR[ord[r]];
                const int32_t life = (int32_t)rx.f - (int32_t)rx.a;
                flag = life > kLongLife ? 1 : 0;
                if (!flag) lw = max(lw, life);
            }
            int32_t tot;
            const int32_t at = nl + block_excl_scan<int32_t>(flag, reinterpret_cast<int32_t*>(red), &tot);
            if (flag) {
                HR[at] = r;
                if (!kSmem && at < kLongStage) {
                    st.s[at] = rx.s;
                    st.a[at] = rx.a;
                    st.f[at] = rx.f;
                    st.id[at] = rx.id;
                }
            }
            nl += tot;
        }
        if (nl == 0 && sz > kWalkMin) continue;  // walked in step 2 (nl: a block total, uniform)
        __syncthreads();
        int64_t lw_max;
        block_excl_max((int64_t)lw, red, &lw_max);
        Comp<I, W> cp;
        cp.AR = AR;
        cp.OFFP = OFFP;
        cp.BEND = BEND;
        cp.ord = ord;
        cp.hr = HR;
        cp.p0 = p0;
        cp.c = sz;
        cp.nl = nl;
        cp.lw = (int32_t)lw_max;
        cp.st = st;
        cp.staged = !kSmem && nl <= kLongStage;
        cp.hold = hold;
        for (int32_t k = 0; k <= nl; ++k) {
            const int32_t r0 = k == 0 ? 0 : HR[k - 1] + 1, r1 = k < nl ? HR[k] : sz;
            if (r1 > r0) {  // the short-lived run between two long-lived members
                const W e = place_run<I, W>(cp, r0, r1, k, CNT, QUE,
                                            kSmem ? nullptr : scratch + (size_t)warp * kPredBuf * 2, policy, s_cnt,
                                            s_tail, s_fail);
                mx = max(mx, e);
                __syncthreads();
            }
            if (k < nl) {
                const W o = place_heavy<I, W, kSmem>(cp, k, policy, CNT, scratch,
                                                     kSmem ? 0 : (int32_t)(kScratchBytes / (2 * sizeof(W))), bo, be,
                                                     red, s_cnt);
                if (threadIdx.x == 0) {
                    int32_t q;
                    mx = max(mx, (W)(o + cp.long_rec(k, q).s));
                }
            }
        }
        __syncthreads();
    }

    return mx;
}

// Test builds (MP_TEST_HOOKS) can name one member, by trace and alloc-order
// position, that the CTA tier never queues, so that a run starves and its
// bounded waits run out; in every other build no member is held.
#ifdef MP_TEST_HOOKS
__device__ int32_t g_test_hold[2] = {-1, -1};
__device__ __forceinline__ int32_t test_hold_position(int b) { return b == g_test_hold[0] ? g_test_hold[1] : -1; }
#else
__device__ __forceinline__ int32_t test_hold_position(int) { return -1; }
#endif

// ------------------------------------------------------------- the kernel

// The whole path for trace b, by the whole CTA.
template <typename I, typename W, bool kSmem, bool kFused>
__device__ __forceinline__ void plan_trace(const int b, const mp_batch& bt, const PlanOut& out,
                                           unsigned char* __restrict__ ws, size_t data_stride, size_t buf_offset,
                                           size_t buf_stride) {
    constexpr bool kWide = sizeof(W) == 8;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ int32_t s_cnt, s_tail, s_bin[kBins], s_base[kBins + 1], s_bad, s_fail, s_big;
    __shared__ int32_t s_mbase[kBinWarp + 1];  // the thread tier's members, by size class
    __shared__ uint32_t s_magic[kBinWarp];     // ceil(2^32 / c) of each thread-tier class
    __shared__ unsigned long long s_hi, s_lo, s_max, s_key, s_lbmax;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int32_t policy = out.policy;
    int32_t* __restrict__ status = out.status;
    const bool want_profile = kFused && out.profile != nullptr;
    const TraceView tv = load_trace(bt, b, want_profile);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const PlanLayout<I, W> L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps, kFused);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * data_stride;
    ARec<I, W>* AR = reinterpret_cast<ARec<I, W>*>(base + L.arec);
    W* OFFP = reinterpret_cast<W*>(base + L.offp);
    W* D = reinterpret_cast<W*>(base + L.dprof);  // fused: before the records exist
    int32_t* BEND = reinterpret_cast<int32_t*>(base + L.bend);
    uint32_t* SB = reinterpret_cast<uint32_t*>(base + L.sb);
    int32_t* WT = reinterpret_cast<int32_t*>(base + L.wt);
    int32_t* LST = reinterpret_cast<int32_t*>(base + L.lst);
    uint16_t* RP = reinterpret_cast<uint16_t*>(base + L.rp);
    // CTA tier workspace: a long-lived member's predecessors (offsets, ends),
    // then (data in the workspace) a large component's priority order and
    // long-lived ranks
    const size_t cap2 = (size_t)pow2_at_least(bt.max_tensors > 0 ? bt.max_tensors : 1);
    int64_t* bo = reinterpret_cast<int64_t*>(ws + buf_offset + (size_t)b * buf_stride);
    int64_t* be = bo + cap2;
    int32_t* ORD = kSmem ? reinterpret_cast<int32_t*>(base + L.ord) : reinterpret_cast<int32_t*>(be + cap2);
    int32_t* HR = kSmem ? reinterpret_cast<int32_t*>(base + L.rp) : ORD + cap2;
    int32_t* CNT = kSmem ? reinterpret_cast<int32_t*>(base + L.cnt) : HR + cap2;
    int32_t* QUE = kSmem ? reinterpret_cast<int32_t*>(base + L.que) : CNT + cap2;

    // ---- clear the histogram (and the difference array)
    for (int t = threadIdx.x; t < T; t += blockDim.x) BEND[t] = 0;
    const int32_t dlen = want_profile ? (int32_t)dpadded<W>((size_t)T) : 0;
    for (int32_t t = threadIdx.x; t < dlen; t += blockDim.x) D[t] = 0;
    if (threadIdx.x < kBins) s_bin[threadIdx.x] = 0;
    if (threadIdx.x == 0) {
        s_bad = 0;
        s_fail = 0;
        s_big = 0;
        s_hi = s_lo = s_max = s_lbmax = 0;
        s_key = ~0ull;
    }
    __syncthreads();

    // ---- load, check, alloc-step histogram, profile differences.  The first
    // kCached * blockDim tensors stay in registers for the scatter below.
    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    const bool vec = ((reinterpret_cast<uintptr_t>(Ag) | reinterpret_cast<uintptr_t>(Fg) |
                       reinterpret_cast<uintptr_t>(Sg)) & 15) == 0;
    auto cached_index = [&](int j) -> int32_t {
        return vec ? 4 * (int32_t)threadIdx.x + j : (int32_t)threadIdx.x + j * (int32_t)blockDim.x;
    };
    int32_t ca[kCached], cf[kCached];
    int64_t cs[kCached];
    bool ok = true;
    uint64_t sum = 0;
    auto take = [&](int32_t a, int32_t f, int64_t s) {
        if (!tensor_ok(a, f, s, T)) {
            ok = false;
            return;
        }
        sum = sat_add(sum, (uint64_t)s);
        atomicAdd(BEND + a, 1);
        if (want_profile) {
            d_add(D + dpos<W>(a), s);
            if (f < T) d_add(D + dpos<W>(f), -s);
        }
    };
    if (vec && 4 * (int32_t)threadIdx.x + 3 < n) {
        const int4 a = __ldg(reinterpret_cast<const int4*>(Ag) + threadIdx.x);
        const int4 f = __ldg(reinterpret_cast<const int4*>(Fg) + threadIdx.x);
        const longlong2 s01 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * threadIdx.x);
        const longlong2 s23 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * threadIdx.x + 1);
        ca[0] = a.x, ca[1] = a.y, ca[2] = a.z, ca[3] = a.w;
        cf[0] = f.x, cf[1] = f.y, cf[2] = f.z, cf[3] = f.w;
        cs[0] = s01.x, cs[1] = s01.y, cs[2] = s23.x, cs[3] = s23.y;
    } else {
#pragma unroll
        for (int j = 0; j < kCached; ++j) {
            const int32_t k = cached_index(j);
            if (k < n) {
                ca[j] = __ldg(Ag + k);
                cf[j] = __ldg(Fg + k);
                cs[j] = __ldg(Sg + k);
            }
        }
    }
#pragma unroll
    for (int j = 0; j < kCached; ++j)
        if (cached_index(j) < n) take(ca[j], cf[j], cs[j]);
    const int32_t nc = min(n, kCached * (int32_t)blockDim.x);
    for (int32_t k = nc + threadIdx.x; k < n; k += blockDim.x) take(__ldg(Ag + k), __ldg(Fg + k), __ldg(Sg + k));
    block_add_size_sum(sum, &s_hi, &s_lo);
    if (!ok) s_bad = 1;
    __syncthreads();
    if (!kWide && !s_bad && (s_hi != 0 || s_lo > 0xffffffffull)) {  // sizes sum to 2^32 or more
        if (threadIdx.x == 0) status[b] = kDeferred;
        return;
    }
    if (s_bad || size_sum_overflows(s_hi, s_lo)) {
        if (threadIdx.x == 0) {
            status[b] = s_bad ? MP_EINVAL : MP_EOVERFLOW;
            if (kFused && out.verdict) out.verdict[b] = 0;
            if (kFused && out.conflict) out.conflict[2 * b] = out.conflict[2 * b + 1] = -1;
        }
        return;
    }

    // ---- scan the histogram into bucket starts
    block_excl_scan_array<int32_t, 8>(BEND, T, reinterpret_cast<int32_t*>(red));

    // ---- live profile (fused): scan the difference array, write it out
    if (want_profile) {
        int64_t* pout = out.profile + tv.plo;
        const bool vec_out = (reinterpret_cast<uintptr_t>(pout) & 15) == 0;
        constexpr int kRun = ProfGeom<W>::kLane;  // steps per lane and tile
        constexpr int kVec = 16 / sizeof(W);      // words per 16-byte read
        W carry = 0, lmax = 0;
        for (int32_t base_t = 0; base_t < T; base_t += (int32_t)blockDim.x * kRun) {
            const int32_t my = base_t + (int32_t)threadIdx.x * kRun;
            const W* run = D + dpos<W>(my);
            W v[kRun];
            if (my + kRun <= T) {
#pragma unroll
                for (int k = 0; k < kRun; k += kVec) {
                    if constexpr (kWide) {
                        const longlong2 q = *reinterpret_cast<const longlong2*>(run + k);
                        v[k] = (W)q.x;
                        v[k + 1] = (W)q.y;
                    } else {
                        const uint4 q = *reinterpret_cast<const uint4*>(run + k);
                        v[k] = (W)q.x;
                        v[k + 1] = (W)q.y;
                        v[k + 2] = (W)q.z;
                        v[k + 3] = (W)q.w;
                    }
                }
            } else {
#pragma unroll
                for (int k = 0; k < kRun; ++k) v[k] = my + k < T ? run[k] : (W)0;
            }
#pragma unroll
            for (int k = 1; k < kRun; ++k) v[k] += v[k - 1];
            W tot;
            const W pre = block_excl_scan_w<W>(v[kRun - 1], red, &tot) + carry;
#pragma unroll
            for (int k = 0; k < kRun; ++k) {
                v[k] += pre;
                lmax = v[k] > lmax ? v[k] : lmax;
            }
            if (vec_out && my + kRun <= T) {
#pragma unroll
                for (int k = 0; k < kRun; k += 2)
                    *reinterpret_cast<longlong2*>(pout + my + k) = make_longlong2((int64_t)v[k], (int64_t)v[k + 1]);
            } else {
#pragma unroll
                for (int k = 0; k < kRun; ++k)
                    if (my + k < T) pout[my + k] = (int64_t)v[k];
            }
            carry += tot;
        }
        const unsigned long long lm = (unsigned long long)warp_max_w(lmax);
        if (lane == 0 && lm > 0) atomicMax(&s_lbmax, lm);
        __syncthreads();  // the difference array is dead from here on
    }

    // ---- counting sort into alloc-step records; BEND[t] ends as the number
    // of tensors with alloc step <= t
    auto scatter = [&](int32_t k, int32_t a, int32_t f, int64_t s) {
        ARec<I, W> r;
        r.s = (W)s;
        r.a = (I)a;
        r.f = (I)f;
        r.id = (I)k;
        r.pad = 0;
        AR[atomicAdd(BEND + a, 1)] = r;
    };
#pragma unroll
    for (int j = 0; j < kCached; ++j) {
        const int32_t k = cached_index(j);
        if (k < n) scatter(k, ca[j], cf[j], cs[j]);
    }
    for (int32_t k = nc + threadIdx.x; k < n; k += blockDim.x) scatter(k, __ldg(Ag + k), __ldg(Fg + k), __ldg(Sg + k));
    __syncthreads();

    // ---- components: a run starts where no earlier tensor is live any more.
    // Each warp scans a contiguous chunk of positions, 32 at a time.
    const int32_t chunk = (((n + nwarps - 1) / nwarps) + 31) & ~31;
    const int32_t w0 = min(n, warp * chunk), w1 = min(n, w0 + chunk);
    {
        unsigned fm = 0;
        for (int32_t p = w0 + lane; p < w1; p += 32) fm = max(fm, (unsigned)AR[p].f);
        fm = __reduce_max_sync(0xffffffffu, fm);
        if (lane == 0) reinterpret_cast<int32_t*>(red)[warp] = (int32_t)fm;
    }
    __syncthreads();
    {
        int32_t carry = 0;
        for (int k = 0; k < warp; ++k) carry = max(carry, reinterpret_cast<int32_t*>(red)[k]);
        for (int32_t p0 = w0; p0 < w1; p0 += 32) {
            const int32_t p = p0 + lane;
            const bool valid = p < w1;
            int32_t a = 0, f = 0;
            if (valid) {
                a = AR[p].a;
                f = AR[p].f;
            }
            int32_t incl = f;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t u = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl = max(incl, u);
            }
            int32_t excl = __shfl_up_sync(0xffffffffu, incl, 1);
            excl = lane == 0 ? carry : max(carry, excl);
            const unsigned starts = __ballot_sync(0xffffffffu, valid && (p == 0 || excl <= a));
            if (lane == 0) SB[p0 >> 5] = starts;
            carry = max(carry, __shfl_sync(0xffffffffu, incl, 31));
        }
    }
    __syncthreads();
    const int32_t nwords = (n + 31) >> 5;
    const int32_t* NW = nullptr;
    if (nwords > kWordWalk) {  // per-word table of the next component start
        int32_t* nw = WT;
        for (int32_t w = threadIdx.x; w < nwords; w += blockDim.x) {
            const uint32_t m = SB[w];
            nw[w] = m ? -((w << 5) + __ffs(m) - 1) : -n;
        }
        __syncthreads();
        block_scan_max_i32(nw, nwords, true, reinterpret_cast<int32_t*>(red));
        NW = nw;
    }

    // ---- component starts, one thread per tensor: a single tensor is placed
    // at 0; the starts of larger components are counted by size class
    W mx = 0;
    const unsigned lt_mask = (1u << lane) - 1u;
    for (int32_t q0 = 0; q0 < n; q0 += blockDim.x) {
        const int32_t p = q0 + threadIdx.x;
        int bin = -1;
        if (p < n && ((SB[p >> 5] >> (p & 31)) & 1u)) {
            const int32_t c = comp_size(SB, NW, p, n);
            if (c == 1) {
                OFFP[p] = 0;
                mx = max(mx, AR[p].s);
            } else {
                bin = comp_bin(c);
                // the 32-bit launch keeps the CTA tier only with its data in
                // shared memory and components up to kDeferComp
                if (c > (kSmem ? kDeferComp : kWarpComp)) s_big = 1;
            }
        }
        const unsigned grp = __match_any_sync(0xffffffffu, bin);
        if (bin >= 0 && (grp & lt_mask) == 0) atomicAdd(&s_bin[bin], __popc(grp));
    }
    __syncthreads();
    if (warp == 0) {  // class starts (s_bin becomes each class's cursor) and the thread tier's member counts
        const int32_t v = lane < kBins ? s_bin[lane] : 0;
        const int32_t incl = warp_incl_scan(v);
        if (lane < kBins) s_base[lane] = s_bin[lane] = incl - v;
        if (lane == kBins - 1) s_base[kBins] = incl;
        const int32_t mv = lane < kBinWarp ? v * (kThreadComp - lane) : 0;
        const int32_t mincl = warp_incl_scan(mv);
        if (lane <= kBinWarp) s_mbase[lane] = mincl - mv;
        if (lane < kBinWarp) s_magic[lane] = 0xffffffffu / (uint32_t)(kThreadComp - lane) + 1u;
    }
    __syncthreads();
    if constexpr (!kWide) {
        if (s_big) {  // a component for the larger CTAs of the 64-bit launch
            if (threadIdx.x == 0) status[b] = kDeferred;
            return;
        }
    }
    for (int32_t q0 = 0; q0 < n; q0 += blockDim.x) {
        const int32_t p = q0 + threadIdx.x;
        int bin = -1;
        if (p < n && ((SB[p >> 5] >> (p & 31)) & 1u)) {
            const int32_t c = comp_size(SB, NW, p, n);
            if (c > 1) bin = comp_bin(c);
        }
        const unsigned grp = __match_any_sync(0xffffffffu, bin);
        const int leader = __ffs(grp) - 1;
        int32_t at = 0;
        if (bin >= 0 && lane == leader) at = atomicAdd(&s_bin[bin], __popc(grp));
        at = __shfl_sync(0xffffffffu, at, leader);
        if (bin >= 0) LST[at + __popc(grp & lt_mask)] = p;
    }
    __syncthreads();

    // ---- members of the thread tier's components, one thread per member in
    // the size-sorted component list (so a warp's members mostly share one
    // component size): each gets its priority rank and the mask of members
    // that precede it and overlap its lifetime
    {
        int32_t mb[kBinWarp + 1];
#pragma unroll
        for (int k = 0; k <= kBinWarp; ++k) mb[k] = s_mbase[k];
        for (int32_t g = threadIdx.x; g < mb[kBinWarp]; g += blockDim.x) {
            int bin = 0;
            int32_t below = 0;  // members of the classes before bin
#pragma unroll
            for (int k = 1; k < kBinWarp; ++k) {
                if (g >= mb[k]) {
                    bin = k;
                    below = mb[k];
                }
            }
            const int32_t c = kThreadComp - bin;
            const uint32_t r = (uint32_t)(g - below);
            const int32_t k = (int32_t)__umulhi(r, s_magic[bin]);  // r / c (r < 2^28)
            const int32_t p0 = LST[s_base[bin] + k];
            const int32_t p = p0 + ((int32_t)r - k * c);
            const ARec<I, W> me = AR[p];
            constexpr bool kPacked = sizeof(W) == 4 && sizeof(I) == 2;
            const uint64_t me_key = kPacked ? prio_key(me) : 0;
            uint32_t rank = 0, pred = 0;
            for (int32_t j = 0; j < c; ++j) {
                const int32_t q = p0 + j;
                if (q == p) continue;
                const ARec<I, W> o = AR[q];
                const bool first = kPacked ? precedes_key(o, me_key) : precedes(o, me);
                const bool ov = q < p ? (int32_t)o.f > (int32_t)me.a : (int32_t)o.a < (int32_t)me.f;
                rank += first ? 1u : 0u;
                pred |= (first && ov ? 1u : 0u) << j;
            }
            RP[p] = (uint16_t)(rank | (pred << 4));
        }
    }
    __syncthreads();

    // ---- warp tier, then the thread tier (largest first)
    {
        const int32_t wb = s_base[kBinWarp], nwc = s_base[kBinCta] - wb;
        for (int32_t k = warp; k < nwc; k += nwarps) {
            const int32_t p0 = LST[wb + k];
            const W e = place_warp(AR, OFFP, p0, comp_size(SB, NW, p0, n), policy);
            mx = max(mx, e);
        }
        // the largest thread-tier components go to the last warp, which has
        // the fewest warp-tier components
        for (int32_t g = ((nwarps - 1 - warp) << 5) + lane; g < wb; g += blockDim.x) {
            const int32_t p0 = LST[g], c = comp_size(SB, NW, p0, n);
            const W e = place_thread(AR, RP, OFFP, p0, c, policy);
            mx = max(mx, e);
        }
    }

    // ---- large components, the whole CTA each
    if (s_base[kBins] > s_base[kBinCta]) {
        const W e = large_tier<I, W, kSmem>(AR, OFFP, BEND, SB, NW, LST + s_base[kBinCta], s_base[kBins] - s_base[kBinCta],
                                            n, ORD, HR, CNT,
                                            QUE, bo, be, smem_raw, policy, red, &s_cnt, &s_tail, &s_fail,
                                            test_hold_position(b));
        mx = max(mx, e);
    }

    {
        const unsigned long long m = (unsigned long long)warp_max_w(mx);
        if (lane == 0 && m > 0) atomicMax(&s_max, m);
        if (threadIdx.x == 0) s_cnt = 0;
    }
    __syncthreads();

    // ---- validation of the plan just made (fused): every lifetime-overlapping
    // pair once, from its earlier member in alloc order, is checked for address
    // overlap -- an independent pass over the alloc-ordered records
    if (kFused) {
        // a thread per tensor; windows longer than kValWide go to a list (LST,
        // free by now) and a warp each
        for (int32_t p = threadIdx.x; p < n; p += blockDim.x) {
            const ARec<I, W> ri = AR[p];
            const int32_t stop = BEND[ri.f - 1];  // tensors with alloc < free_i
            if (stop <= p + 1) continue;
            if (stop - p - 1 > kValWide) {
                LST[atomicAdd(&s_cnt, 1)] = p;
                continue;
            }
            const W oi = OFFP[p], ei = oi + ri.s;
            for (int32_t q = p + 1; q < stop; ++q) {
                const W oj = OFFP[q];
                if (oi < oj + AR[q].s && oj < ei) {
                    const uint32_t i = (uint32_t)ri.id, j = (uint32_t)AR[q].id;
                    atomicMin(&s_key, ((unsigned long long)(i < j ? i : j) << 32) | (i < j ? j : i));
                }
            }
        }
        __syncthreads();
        const int32_t nwide = s_cnt;
        for (int32_t k = warp; k < nwide; k += nwarps) {
            const int32_t p = LST[k];
            const ARec<I, W> ri = AR[p];
            const int32_t stop = BEND[ri.f - 1];
            const W oi = OFFP[p], ei = oi + ri.s;
            for (int32_t q = p + 1 + lane; q < stop; q += 32) {
                const W oj = OFFP[q];
                if (oi < oj + AR[q].s && oj < ei) {
                    const uint32_t i = (uint32_t)ri.id, j = (uint32_t)AR[q].id;
                    atomicMin(&s_key, ((unsigned long long)(i < j ? i : j) << 32) | (i < j ? j : i));
                }
            }
        }
        __syncthreads();
    }

    // ---- outputs (offsets by tensor id)
    int64_t* __restrict__ offsets = out.offsets + tv.lo;
    for (int32_t p = threadIdx.x; p < n; p += blockDim.x) offsets[(int32_t)AR[p].id] = (int64_t)OFFP[p];
    if (threadIdx.x == 0) {
        out.plan_peak[b] = (int64_t)s_max;
        if (kFused) {
            if (want_profile && out.peak_lb) out.peak_lb[b] = (int64_t)s_lbmax;
            const unsigned long long key = s_key;
            const bool good = key == ~0ull;
            if (out.verdict) out.verdict[b] = good ? 1 : 0;
            if (out.conflict) {
                out.conflict[2 * b] = good ? -1 : (int32_t)(key >> 32);
                out.conflict[2 * b + 1] = good ? -1 : (int32_t)(key & 0xffffffffu);
            }
        }
        status[b] = s_fail ? MP_ETIMEOUT : MP_OK;
    }
}

// 32-bit launch: one CTA per trace.  64-bit launch: a grid no larger than
// what the GPU holds at once walks every trace and takes the ones the 32-bit
// launch deferred (sizes summing to 2^32 or more, or a component the 32-bit
// launch does not place), with larger CTAs for the CTA tier.
template <typename I, typename W, bool kSmem, bool kFused>
__global__ void __launch_bounds__(sizeof(W) == 8 ? kPlanThreadsWide : (kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal),
                                  sizeof(W) == 8 ? 1 : (kSmem ? 9 : 1))
k_plan(mp_batch bt, PlanOut out, unsigned char* __restrict__ ws, size_t data_stride, size_t buf_offset,
       size_t buf_stride) {
    if constexpr (sizeof(W) == 4) {
        plan_trace<I, W, kSmem, kFused>(blockIdx.x, bt, out, ws, data_stride, buf_offset, buf_stride);
        // the 64-bit launch may start now; it waits for this grid to finish
        // (and its writes to land) before it reads anything this grid wrote
        asm volatile("griddepcontrol.launch_dependents;");
    } else {
        asm volatile("griddepcontrol.wait;" ::: "memory");
        // this CTA's traces are blockIdx.x + k * gridDim.x; their statuses are
        // read 32 at a time by one warp
        __shared__ unsigned s_deferred;
        for (int64_t k0 = 0; blockIdx.x + k0 * gridDim.x < bt.n_traces; k0 += 32) {
            if (threadIdx.x < 32) {
                const int64_t b = blockIdx.x + (k0 + threadIdx.x) * gridDim.x;
                const unsigned m = __ballot_sync(0xffffffffu, b < bt.n_traces && out.status[b] == kDeferred);
                if (threadIdx.x == 0) s_deferred = m;
            }
            __syncthreads();
            unsigned m = s_deferred;
            __syncthreads();
            while (m) {
                const int b = (int)(blockIdx.x + (k0 + __ffs(m) - 1) * gridDim.x);
                m &= m - 1;
                plan_trace<I, W, kSmem, kFused>(b, bt, out, ws, data_stride, buf_offset, buf_stride);
                __syncthreads();
            }
        }
    }
}

struct PlanGeometry {
    bool smem, narrow;
    size_t data, data_stride;
};

// 16-bit indices when every id and step fits; shared memory when the trace's
// working set fits under the ceiling, else a workspace slice per trace.
template <typename W>
PlanGeometry plan_geometry(const mp_batch& bt, bool fused) {
    PlanGeometry g;
    g.narrow = bt.max_tensors < 32767 && bt.max_steps <= 32767;
    g.data = g.narrow ? PlanLayout<int16_t, W>(bt.max_tensors, bt.max_steps, fused).total
                      : PlanLayout<int32_t, W>(bt.max_tensors, bt.max_steps, fused).total;
    g.smem = g.data <= kPlanSmemLimit;
    g.data_stride = g.smem ? 0 : g.data;
    return g;
}

// Workspace: the per-trace slices of the launches that keep their data there
// (the two launches run one after the other and share it), then the CTA
// tier's buffers per trace (a long-lived member's predecessors; a large
// component's priority order, long-lived ranks, predecessor counts and
// ready queue), sized for up to max_tensors.
struct PlanWorkspace {
    size_t buf_offset, buf_stride, total;
};
PlanWorkspace plan_workspace(const mp_batch& bt) {
    PlanWorkspace w;
    size_t slices = 0;
    for (bool fused : {false, true}) {
        const PlanGeometry a = plan_geometry<uint32_t>(bt, fused), b = plan_geometry<int64_t>(bt, fused);
        slices = std::max(slices, std::max(a.data_stride, b.data_stride));
    }
    const size_t cap2 = (size_t)pow2_at_least(bt.max_tensors > 0 ? bt.max_tensors : 1);
    w.buf_offset = mul_sat((size_t)bt.n_traces, slices);
    w.buf_stride = align_up(cap2 * 32);
    w.total = bt.n_traces == 0 ? 0 : add_sat(w.buf_offset, mul_sat((size_t)bt.n_traces, w.buf_stride));
    return w;
}

template <typename I, typename W, bool kSmem, bool kFused>
cudaError_t launch_variant(const mp_batch& bt, const PlanGeometry& g, const PlanWorkspace& pw, const PlanOut& out,
                           unsigned char* ws, cudaStream_t stream) {
    const int threads = sizeof(W) == 8 ? kPlanThreadsWide : (kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal);
    const size_t smem = kSmem ? g.data : (sizeof(W) == 8 ? flow_smem_bytes<W>() : 0);
    const void* fn = (const void*)k_plan<I, W, kSmem, kFused>;
    {
        cudaError_t e = set_smem_limit(fn, smem);
        if (e != cudaSuccess) return e;
    }
    int grid = bt.n_traces;
    if (sizeof(W) == 8) {
        int resident = 0;
        cudaError_t e = max_resident_ctas(fn, threads, smem, &resident);
        if (e != cudaSuccess) return e;
        grid = std::max(1, std::min(grid, resident));
    }
    if (sizeof(W) == 4) {
        k_plan<I, W, kSmem, kFused><<<(unsigned)grid, threads, smem, stream>>>(bt, out, ws, g.data_stride,
                                                                               pw.buf_offset, pw.buf_stride);
        return cudaGetLastError();
    }
    // the 64-bit launch depends on the 32-bit one programmatically: its CTAs
    // may be scheduled while the first grid drains, and wait in-kernel
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_plan<I, W, kSmem, kFused>, bt, out, ws, g.data_stride, pw.buf_offset,
                              pw.buf_stride);
}

template <typename W, bool kFused>
cudaError_t launch_width(const mp_batch& bt, const PlanOut& out, unsigned char* ws, cudaStream_t stream) {
    const PlanGeometry g = plan_geometry<W>(bt, kFused);
    const PlanWorkspace pw = plan_workspace(bt);
    if (g.narrow)
        return g.smem ? launch_variant<int16_t, W, true, kFused>(bt, g, pw, out, ws, stream)
                      : launch_variant<int16_t, W, false, kFused>(bt, g, pw, out, ws, stream);
    return g.smem ? launch_variant<int32_t, W, true, kFused>(bt, g, pw, out, ws, stream)
                  : launch_variant<int32_t, W, false, kFused>(bt, g, pw, out, ws, stream);
}

template <bool kFused>
cudaError_t launch_any(const mp_batch& bt, const PlanOut& out, void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    cudaError_t e = launch_width<uint32_t, kFused>(bt, out, ws, stream);
    if (e != cudaSuccess) return e;
    return launch_width<int64_t, kFused>(bt, out, ws, stream);
}

}  // namespace

// One workspace size serves both the planner and the fused entry point;
// batches of large traces take the grid-wide dataflow (grid.cu).
size_t plan_workspace_bytes(const mp_batch& bt) {
    return grid_path(bt) ? grid_workspace_bytes(bt) : plan_workspace(bt).total;
}

cudaError_t launch_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                        int32_t* status, void* workspace, cudaStream_t stream) {
    if (grid_path(bt)) return launch_grid_plan(bt, policy, offsets, plan_peak, status, workspace, -1, stream);
    const PlanOut out{policy, offsets, plan_peak, status, nullptr, nullptr, nullptr, nullptr};
    return launch_any<false>(bt, out, workspace, stream);
}

cudaError_t launch_plan_fused(const mp_batch& bt, int32_t policy, int64_t* profile, int64_t* peak_lb,
                              int64_t* offsets, int64_t* plan_peak, int32_t* verdict, int32_t* conflict,
                              int32_t* status, void* workspace, cudaStream_t stream) {
    if (grid_path(bt))
        return launch_grid_fused(bt, policy, profile, peak_lb, offsets, plan_peak, verdict, conflict, status,
                                 workspace, stream);
    const PlanOut out{policy, offsets, plan_peak, status, profile, peak_lb, verdict, conflict};
    return launch_any<true>(bt, out, workspace, stream);
}

}  // namespace mp

#ifdef MP_TEST_HOOKS
// Test builds only: greedy_by_size as mp_plan_greedy_by_size, except that the
// member at alloc-order position hold_pos of trace hold_trace is never queued
// (the grid-wide planner for batches of a few large traces, the CTA tier's
// ready queue otherwise), so the planner's bounded waits run out and that
// trace reports MP_ETIMEOUT while the others are planned as usual.
extern "C" __attribute__((visibility("default"))) mp_status mp_test_plan_hold(
    const mp_batch* batch, mp_fit_policy policy, int64_t* offsets, int64_t* plan_peak, int32_t* trace_status,
    void* workspace, size_t workspace_bytes, int32_t hold_trace, int32_t hold_pos, void* stream) {
    static const int32_t none[2] = {-1, -1};
    static int32_t held[2];
    if (batch == nullptr || workspace_bytes < mp::plan_workspace_bytes(*batch)) return MP_EINVAL;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (mp::grid_path(*batch)) {
        const int64_t slot = (int64_t)hold_trace * batch->max_tensors + hold_pos;
        return mp::launch_grid_plan(*batch, policy, offsets, plan_peak, trace_status, workspace, (int32_t)slot, st) ==
                       cudaSuccess
                   ? MP_OK
                   : MP_ECUDA;
    }
    held[0] = hold_trace;
    held[1] = hold_pos;
    cudaError_t e = cudaMemcpyToSymbol(mp::g_test_hold, held, sizeof(held));
    if (e == cudaSuccess) e = mp::launch_plan(*batch, policy, offsets, plan_peak, trace_status, workspace, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    const cudaError_t e2 = cudaMemcpyToSymbol(mp::g_test_hold, none, sizeof(none));
    return e == cudaSuccess && e2 == cudaSuccess ? MP_OK : MP_ECUDA;
}
#endif
