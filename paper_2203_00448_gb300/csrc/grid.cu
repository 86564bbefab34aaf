// grid.cu -- greedy_by_size for batches of large traces, spread over the
// whole GPU (Sec. 2.3's strategy, Sec. 3.2's default; the fused variant also
// builds the live profile and validates the plan, Eq. 2.1).
//
// The sequential definition places tensors one by one in priority order
// (size descending, alloc step ascending, id ascending).  The offset of
// tensor i depends only on its predecessors P_i: the tensors that overlap it
// in lifetime and come first in priority.  So i can be placed as soon as
// every member of P_i is, and the result is bit-identical to the sequential
// one whatever the order in which independent tensors are placed.  Here the
// dependency graph of every trace of the batch is executed as one dataflow by
// a persistent grid that covers the GPU:
//
//   k_grid_prep    one CTA per trace: checks, the exact size sum, the alloc-
//                  step histogram, the live profile (fused), a counting sort
//                  into alloc-ordered records, the list of long-lived
//                  tensors, and the trace's dataflow state;
//   k_grid_flow    one cooperative launch, every CTA resident: first each
//                  warp counts the predecessors of its share of the tensors
//                  (a tensor whose count reaches zero is queued), then the
//                  CTAs take ready tensors from two global queues -- a
//                  short-lived tensor with at most kWarpPairs predecessors is
//                  placed by one warp, any other (a long-lived one has many
//                  candidates) by the whole CTA -- gather the predecessors'
//                  offsets, run the FIRST or BEST gap search, publish the
//                  offset, and decrement the counts of the tensors that follow
//                  it in priority and overlap it, queueing those that reach
//                  zero;
//   k_grid_finish  a warp per 32 tensors: offsets back by tensor id, the plan
//                  peak, and (fused) every lifetime-overlapping pair checked
//                  for address overlap;
//   k_grid_final   one thread per trace: peaks, verdicts, statuses.
//
// Candidates.  A short-lived tensor (life at most kGridLong steps) overlaps
// tensor x only if it is allocated in (a_x - lw, f_x), lw being the longest
// short life of the trace: a window of the alloc-ordered records bounded by
// two bucket ends.  Long-lived tensors are listed apart in alloc order, and
// those overlapping x are among the ones allocated before f_x.  Predecessor
// and successor enumerations use the same candidate sets and tests, so every
// count is decremented exactly as often as it was incremented.
//
// Counts are signed: a tensor's count starts at zero, its own enumeration adds
// |P_i| and every placed predecessor subtracts one, in any order; the value
// is zero again exactly once, after all of them, and whoever makes it zero
// queues the tensor.  No grid-wide barrier separates counting from placing.
//
// Waits.  A worker (a warp, or a CTA for CTA items) takes the next slot of its
// queue and waits for it to be filled; placing a tensor waits for nothing.  A
// worker holds at most one slot, and the lowest-ranked unplaced tensor of a
// trace is always queued, so while tensors remain some worker is placing one
// and every taken slot is filled in the end.  The wait is still bounded: after
// kGridSpinCycles (about a second) in which nothing is queued or placed
// anywhere, the worker raises a flag, every worker leaves, and the traces
// left incomplete report MP_ETIMEOUT.
#include <algorithm>

#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int kGridThreads = 512;             // flow CTA: 16 warps
constexpr int kGridWarps = kGridThreads / 32;
constexpr int kPrepThreads = 512;
constexpr int kFinishThreads = 256;
constexpr int32_t kGridLong = 32;             // lives above this many steps: long-lived, placed by a CTA
// Flow CTA shared memory: a region for the item being placed, then a cache of
// the batch's long-lived records.  A CTA item uses the region for up to
// kLongPredPairs predecessor pairs and kLongSuccs successor slots; a warp item
// uses its warp's 1/16 of it for up to kWarpSortPairs pairs (kWarpPairs
// predecessors, padded for the sort) and kWarpSuccs successor slots.
constexpr size_t kRegionBytes = 176 * 1024;
constexpr int32_t kLongCache = 2400;          // long-lived records cached per CTA (20 bytes each)
constexpr size_t kCacheBytes = (size_t)kLongCache * 20;
constexpr size_t kGridSmem = kRegionBytes + kCacheBytes;
constexpr int32_t kLongPredPairs = 9216;
constexpr int32_t kLongSuccs = (int32_t)((kRegionBytes - (size_t)kLongPredPairs * 16) / 4);
constexpr int32_t kRegionPairs = kLongPredPairs;  // CTA-item pairs beyond this go to the overflow buffer
constexpr int32_t kWarpBytes = (int32_t)(kRegionBytes / 16);
constexpr int32_t kWarpSortPairs = 512;
constexpr int32_t kWarpPairs = 448;  // predecessors a warp holds while it places a short tensor
constexpr int32_t kWarpSuccs = (kWarpBytes - kWarpSortPairs * 16) / 4;
static_assert(kLongSuccs >= 1024 && kWarpSuccs >= 512, "successor lists");
constexpr int kMaxLongCtas = 32;              // CTAs that place CTA items (and own an overflow buffer)
constexpr int32_t kGridValWide = 64;          // validation windows longer than this: a warp each
#ifdef MP_TEST_GRID_SPIN_CYCLES
constexpr long long kGridSpinCycles = MP_TEST_GRID_SPIN_CYCLES;
#else
constexpr long long kGridSpinCycles = 1ll << 31;
#endif

// Queues and counters shared by the whole grid.
struct GridCtl {
    int32_t head_s, tail_s;  // warp items: next slot to take, next slot to fill
    int32_t head_l, tail_l;  // CTA items
    int32_t total;           // tensors of the traces that passed their checks
    int32_t placed;          // tensors placed so far
    int32_t fail;            // a CTA gave up waiting
    int32_t pad;
};

// Per-trace state.
struct TraceInfo {
    int64_t lo;               // first tensor of the trace in the batch arrays
    unsigned long long peak;  // largest offset + size
    unsigned long long key;   // smallest conflicting (min id, max id), packed; ~0 if none
    int32_t n, T, lw, nlong;  // tensors, steps, longest short life, long-lived tensors
    int32_t ok;               // 1 once the trace passed its checks
    int32_t incomplete;       // a tensor was left unplaced
};

// A tensor in alloc-step order (16 bytes: one vector load).
struct GRec {
    int64_t s;
    int32_t a, f;
};

struct GridWs {
    GridCtl* ctl;
    TraceInfo* ti;
    int32_t* bend;   // [B][max_steps]: bucket ends by alloc step
    GRec* rec;       // [B][max_tensors]: alloc-ordered records
    int32_t* rid;    // tensor id of each record
    int64_t* off;    // offset of each record (-1 until placed)
    int32_t* cnt;    // signed predecessor counts
    int32_t* cls;    // 1: a CTA item (long-lived, or more predecessors than a warp's buffer)
    int32_t* qs;     // queue of ready warp items (slot ids, -1 = not filled)
    int32_t* ql;     // queue of ready CTA items
    int32_t* ll;     // [B][max_tensors]: positions of the long-lived records, ascending
    int64_t* ovf;    // per long-capable CTA: pairs beyond the shared region
    int64_t ovf_pairs;
    int32_t M;       // max_tensors: the slot stride of a trace
    int32_t TS;      // max_steps: the bucket stride of a trace
    int64_t hold;    // test hook: the slot that is never queued (-1: none)
};

struct GridOut {
    int32_t policy;
    int64_t* offsets;
    int64_t* plan_peak;
    int32_t* status;
    int64_t* profile;
    int64_t* peak_lb;
    int32_t* verdict;
    int32_t* conflict;
};

// The long-lived records of the batch, trace after trace in long-list order,
// in a CTA's shared memory (when they fit): size, alloc and free step, and
// alloc-order position.  base[b] is where trace b's start (32 traces at most).
struct LongCache {
    int64_t* s;
    int32_t* a;
    int32_t* f;
    int32_t* q;
    const int32_t* base;  // null: no cache, read the long list from global memory
    const int32_t* lw;    // per trace: the longest short life (always set)
    const int32_t* nl;    // per trace: the number of long-lived records (always set)
};

// ---------------------------------------------------------------- memory order

// Values other CTAs write during the flow are read and written with
// gpu-scope relaxed accesses (never a stale L1 line) and ordered by fences.
__device__ __forceinline__ int32_t ld_rlx(const int32_t* p) {
    int32_t v;
    asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_rlx(int64_t* p, int64_t v) {
    asm volatile("st.relaxed.gpu.global.s64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ void st_rlx(int32_t* p, int32_t v) {
    asm volatile("st.relaxed.gpu.global.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// ---------------------------------------------------------------- helpers

__device__ __forceinline__ bool is_long(const GRec& r) { return r.f - r.a > kGridLong; }
__device__ __forceinline__ bool overlaps(const GRec& x, const GRec& y) { return x.a < y.f && y.a < x.f; }

__device__ __forceinline__ int64_t warp_max64(int64_t v) {
    const unsigned full = 0xffffffffu;
    const unsigned hi = __reduce_max_sync(full, (unsigned)((uint64_t)v >> 32));
    const unsigned lo = __reduce_max_sync(full, (unsigned)((uint64_t)v >> 32) == hi ? (unsigned)v : 0u);
    return (int64_t)(((uint64_t)hi << 32) | lo);
}
__device__ __forceinline__ int64_t warp_min64(int64_t v) {
    const unsigned full = 0xffffffffu;
    const unsigned hi = __reduce_min_sync(full, (unsigned)((uint64_t)v >> 32));
    const unsigned lo = __reduce_min_sync(full, (unsigned)((uint64_t)v >> 32) == hi ? (unsigned)v : ~0u);
    return (int64_t)(((uint64_t)hi << 32) | lo);
}

// The trace of slot g and its view.
struct Node {
    int64_t g, base;  // slot, first slot of its trace
    int32_t b, p;     // trace, alloc-order position
    GRec r;
    int32_t id;
};

__device__ __forceinline__ Node load_node(const GridWs& w, int64_t g) {
    Node x;
    x.g = g;
    x.b = (int32_t)(g / w.M);
    x.p = (int32_t)(g - (int64_t)x.b * w.M);
    x.base = (int64_t)x.b * w.M;
    const int4 v = __ldg(reinterpret_cast<const int4*>(w.rec + g));
    x.r.s = (int64_t)(((uint64_t)(uint32_t)v.y << 32) | (uint32_t)v.x);
    x.r.a = v.z;
    x.r.f = v.w;
    x.id = __ldg(w.rid + g);
    return x;
}

__device__ __forceinline__ GRec load_rec(const GridWs& w, int64_t g) {
    const int4 v = __ldg(reinterpret_cast<const int4*>(w.rec + g));
    GRec r;
    r.s = (int64_t)(((uint64_t)(uint32_t)v.y << 32) | (uint32_t)v.x);
    r.a = v.z;
    r.f = v.w;
    return r;
}

// The candidate sets of x: alloc-order positions [w0, w1) (short-lived
// members only) and the long-lived list entries [0, nlong) allocated before f_x.
struct Cands {
    int32_t w0, w1, nlong;
};
__device__ __forceinline__ Cands cands_of(const GridWs& w, int32_t lw, int32_t nlong, const Node& x) {
    const int32_t* bend = w.bend + (int64_t)x.b * w.TS;
    Cands c;
    c.w0 = x.r.a >= lw ? __ldg(bend + (x.r.a - lw)) : 0;
    c.w1 = __ldg(bend + (x.r.f - 1));
    c.nlong = nlong;
    return c;
}

// A candidate of x: its slot and record.
struct Cand {
    int64_t slot;
    GRec r;
};

// Loads candidate k of x's sets -- window positions first (short-lived
// records only), then long-list entries (from the CTA's cache when there is
// one) -- and returns whether it overlaps x in lifetime (x itself and
// long-lived records met in the window do not).
__device__ __forceinline__ bool fetch_cand(const GridWs& w, const LongCache& lc, const Node& x, const Cands& c,
                                           int32_t k, Cand* cd) {
    const int32_t nwin = c.w1 - c.w0;
    int32_t q;
    if (k < nwin) {
        q = c.w0 + k;
    } else if (k < nwin + c.nlong) {
        if (lc.base) {
            const int32_t i = lc.base[x.b] + (k - nwin);
            q = lc.q[i];
            cd->slot = x.base + q;
            cd->r.s = lc.s[i];
            cd->r.a = lc.a[i];
            cd->r.f = lc.f[i];
            return q != x.p && overlaps(cd->r, x.r);
        }
        q = __ldg(w.ll + x.base + (k - nwin));
    } else {
        cd->r.a = INT32_MAX;  // past the sets
        return false;
    }
    cd->slot = x.base + q;
    cd->r = load_rec(w, cd->slot);
    if (q == x.p || (k < nwin && is_long(cd->r))) return false;
    return overlaps(cd->r, x.r);
}

// An overlapping candidate precedes x in priority (else x precedes it).
__device__ __forceinline__ bool cand_precedes(const GridWs& w, const Node& x, const Cand& cd) {
    const GRec& o = cd.r;
    if (o.s != x.r.s) return o.s > x.r.s;
    if (o.a != x.r.a) return o.a < x.r.a;
    return __ldg(w.rid + cd.slot) < x.id;
}

// Offsets other CTAs published: read through L2 (never a stale L1 line),
// after the acquiring fence that follows a queue entry.
__device__ __forceinline__ int64_t off_of(const GridWs& w, int64_t slot) { return __ldcg(w.off + slot); }

// Queues a tensor whose last predecessor is placed (not the held one of a
// test), in the queue of its class (set before its count was added).
__device__ __forceinline__ void push(const GridWs& w, int64_t slot) {
    if (slot == w.hold) return;
    __threadfence();  // every predecessor's offset, and the class, before the queue entry
    const bool cta = __ldcg(w.cls + slot) != 0;
    const int32_t at = atomicAdd(cta ? &w.ctl->tail_l : &w.ctl->tail_s, 1);
    st_rlx((cta ? w.ql : w.qs) + at, (int32_t)slot);
}

// ---------------------------------------------------------------- prep

template <bool kFused>
__global__ void __launch_bounds__(kPrepThreads) k_grid_prep(mp_batch bt, GridOut out, GridWs w) {
    __shared__ int64_t red[72];
    __shared__ unsigned long long s_hi, s_lo;
    __shared__ int s_bad, s_lw, s_nlong;
    const int b = blockIdx.x;
    const int tid = threadIdx.x, nthr = blockDim.x;
    const bool want_profile = kFused && out.profile != nullptr;
    TraceInfo* ti = w.ti + b;
    const TraceView tv = load_trace(bt, b, want_profile);
    auto fail = [&](int32_t st) {
        if (tid == 0) {
            out.status[b] = st;
            ti->ok = 0;
            ti->n = 0;
            if (kFused && out.verdict) out.verdict[b] = 0;
            if (kFused && out.conflict) out.conflict[2 * b] = out.conflict[2 * b + 1] = -1;
        }
    };
    if (tv.st != MP_OK) {
        fail(tv.st);
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    int32_t* bend = w.bend + (int64_t)b * w.TS;
    int64_t* prof = want_profile ? out.profile + tv.plo : nullptr;
    for (int32_t t = tid; t < T; t += nthr) {
        bend[t] = 0;
        if (want_profile) prof[t] = 0;
    }
    if (tid == 0) {
        s_hi = s_lo = 0;
        s_bad = 0;
        s_lw = 1;
        s_nlong = 0;
    }
    __syncthreads();
    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    bool bad = false;
    uint64_t sum = 0;
    for (int32_t k = tid; k < n; k += nthr) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t s = __ldg(Sg + k);
        if (!tensor_ok(a, f, s, T)) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        atomicAdd(bend + a, 1);
        if (want_profile) {
            atomicAdd(reinterpret_cast<unsigned long long*>(prof + a), (unsigned long long)s);
            if (f < T) atomicAdd(reinterpret_cast<unsigned long long*>(prof + f), (unsigned long long)(-s));
        }
    }
    block_add_size_sum(sum, &s_hi, &s_lo);
    if (bad) s_bad = 1;
    __syncthreads();
    if (s_bad || size_sum_overflows(s_hi, s_lo)) {
        fail(s_bad ? MP_EINVAL : MP_EOVERFLOW);
        return;
    }
    if (want_profile) {  // prefix sums of the differences are the profile
        const int64_t mx = block_incl_scan_max_i64<8>(prof, T, 0, red);
        if (tid == 0 && out.peak_lb) out.peak_lb[b] = mx;
    }
    block_excl_scan_array<int32_t, 8>(bend, T, reinterpret_cast<int32_t*>(red));
    const int64_t base = (int64_t)b * w.M;
    int32_t lw = 1;
    for (int32_t k = tid; k < n; k += nthr) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t s = __ldg(Sg + k);
        const int32_t pos = atomicAdd(bend + a, 1);
        *reinterpret_cast<int4*>(w.rec + base + pos) =
            make_int4((int32_t)(uint32_t)(uint64_t)s, (int32_t)(uint32_t)((uint64_t)s >> 32), a, f);
        w.rid[base + pos] = k;
        w.off[base + pos] = -1;
        w.cnt[base + pos] = 0;
        if (f - a <= kGridLong) lw = max(lw, f - a);
    }
    atomicMax(&s_lw, lw);
    __syncthreads();  // bend now holds the bucket ends; the records are in place
    // the long-lived records in alloc order
    int32_t nlong = 0;
    for (int32_t p0 = 0; p0 < n; p0 += nthr) {
        const int32_t p = p0 + tid;
        int32_t flag = 0;
        if (p < n) {
            const int4 v = *reinterpret_cast<const int4*>(w.rec + base + p);
            flag = v.w - v.z > kGridLong ? 1 : 0;
        }
        int32_t tot;
        const int32_t at = nlong + block_excl_scan<int32_t>(flag, reinterpret_cast<int32_t*>(red), &tot);
        if (flag) w.ll[base + at] = p;
        nlong += tot;
    }
    if (tid == 0) {
        ti->lo = tv.lo;
        ti->peak = 0;
        ti->key = ~0ull;
        ti->n = n;
        ti->T = T;
        ti->lw = s_lw;
        ti->nlong = nlong;
        ti->incomplete = 0;
        ti->ok = 1;
        atomicAdd(&w.ctl->total, n);
    }
}

// ---------------------------------------------------------------- flow

constexpr int kU = 2;  // candidates per lane whose loads are in flight together

// Gap search of a warp over predecessor pairs supplied by each(fn), which
// calls fn(off, end) for every pair held by the calling lane: FIRST jumps to
// the largest conflicting end until nothing conflicts; BEST walks the free
// holes below the top.
template <typename Each>
__device__ int64_t warp_fit(int64_t s, int32_t policy, Each&& each) {
    if (policy == MP_FIT_FIRST) {
        int64_t o = 0;
        for (;;) {
            int64_t hit = 0;
            each([&](int64_t po, int64_t pe) {
                if (po < o + s && o < pe && pe > hit) hit = pe;
            });
            hit = warp_max64(hit);
            if (hit <= o) return o;
            o = hit;
        }
    }
    int64_t top = 0;
    each([&](int64_t, int64_t pe) { top = pe > top ? pe : top; });
    top = warp_max64(top);
    int64_t c = 0, best_len = INT64_MAX, best = top;
    while (c < top) {
        for (;;) {  // move c off every predecessor covering it
            int64_t cov = 0;
            each([&](int64_t po, int64_t pe) {
                if (po <= c && c < pe && pe > cov) cov = pe;
            });
            cov = warp_max64(cov);
            if (cov <= c) break;
            c = cov;
        }
        if (c >= top) break;
        int64_t ns = INT64_MAX;  // c is uncovered below the top: the next start above it
        each([&](int64_t po, int64_t) {
            if (po > c && po < ns) ns = po;
        });
        ns = warp_min64(ns);
        const int64_t len = ns - c;
        if (len >= s && len < best_len) {
            best_len = len;
            best = c;
        }
        c = ns;
    }
    return best;
}

// Gap search of a warp over np <= kWarpSortPairs pairs in buf: a bitonic sort
// by offset, then one scan in which the gap before pair k is its offset minus
// the largest end before it (FIRST: the lowest gap that fits; BEST: the
// smallest, the lowest on ties; none: the largest end).
__device__ int64_t warp_sorted_fit(int64_t s, int32_t policy, int64_t* buf, int32_t np) {
    const int lane = threadIdx.x & 31;
    const unsigned full = 0xffffffffu;
    int32_t plen = 1;
    while (plen < np) plen <<= 1;
    for (int32_t k = np + lane; k < plen; k += 32) buf[2 * k] = buf[2 * k + 1] = INT64_MAX;
    __syncwarp();
    for (int32_t kk = 2; kk <= plen; kk <<= 1) {
        for (int32_t j = kk >> 1; j > 0; j >>= 1) {
            for (int32_t t = lane; t < (plen >> 1); t += 32) {
                const int32_t lo = 2 * t - (t & (j - 1)), hi = lo + j;
                const bool up = (lo & kk) == 0;
                const int64_t xo = buf[2 * lo], yo = buf[2 * hi];
                if (up ? yo < xo : xo < yo) {
                    const int64_t xe = buf[2 * lo + 1];
                    buf[2 * lo] = yo;
                    buf[2 * hi] = xo;
                    buf[2 * lo + 1] = buf[2 * hi + 1];
                    buf[2 * hi + 1] = xe;
                }
            }
            __syncwarp();
        }
    }
    const int32_t chunk = (np + 31) / 32;
    const int32_t k0 = min(np, lane * chunk), k1 = min(np, k0 + chunk);
    int64_t local = 0;
    for (int32_t k = k0; k < k1; ++k) local = max(local, buf[2 * k + 1]);
    int64_t incl = local;  // inclusive prefix max of the lanes' chunk maxima
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t u = __shfl_up_sync(full, incl, o);
        if (lane >= o) incl = u > incl ? u : incl;
    }
    const int64_t top = __shfl_sync(full, incl, 31);
    int64_t prev = __shfl_up_sync(full, incl, 1);
    if (lane == 0) prev = 0;
    int64_t key = INT64_MAX, val = INT64_MAX;
    for (int32_t k = k0; k < k1; ++k) {
        const int64_t gl = buf[2 * k] - prev;
        if (gl >= s) {
            const int64_t kx = policy == MP_FIT_FIRST ? prev : gl;  // prev grows with k
            if (kx < key || (kx == key && prev < val)) {
                key = kx;
                val = prev;
            }
        }
        prev = max(prev, buf[2 * k + 1]);
    }
    warp_min_pair(key, val);
    return key == INT64_MAX ? top : val;
}

// Visits x's candidates with one warp, kU per lane with their loads in
// flight together: fn(hit, cand) on every lane in warp-uniform rounds, hit
// meaning the candidate overlaps x.  The long list (ascending alloc steps)
// stops after a round in which every candidate starts at or after f_x.
template <typename Fn>
__device__ __forceinline__ void warp_visit(const GridWs& w, const LongCache& lc, const Node& x, const Cands& c,
                                           Fn&& fn) {
    const int lane = threadIdx.x & 31;
    const int32_t nwin = c.w1 - c.w0, ncand = nwin + c.nlong;
    for (int32_t k0 = 0; k0 < ncand; k0 += 32 * kU) {
        Cand cd[kU];
        bool hit[kU];
        bool past = true;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int32_t k = k0 + u * 32 + lane;
            hit[u] = fetch_cand(w, lc, x, c, k, &cd[u]);
            past &= k < nwin ? false : cd[u].r.a >= x.r.f;
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) fn(hit[u], cd[u]);
        if (k0 + 32 * kU > nwin && __all_sync(0xffffffffu, past)) break;
    }
}

// Drops the count of a successor of a placed tensor; returns true if it
// became ready.  The caller either queues it or, as a continuation, places it
// next itself.
__device__ __forceinline__ bool drop(const GridWs& w, int64_t slot) { return atomicSub(w.cnt + slot, 1) == 1; }

// The class of a tensor that became ready (read after the acquiring fence).
__device__ __forceinline__ bool cta_item(const GridWs& w, int64_t slot) {
    __threadfence();
    return __ldcg(w.cls + slot) != 0;
}

// A short-lived tensor with at most kWarpPairs predecessors, placed by one
// warp.  buf: the warp's share of the region -- kWarpSortPairs (offset, end)
// pairs, then kWarpSuccs successor slots.  One pass over the candidates
// gathers the predecessors and lists the successors; the gap search runs on
// the gathered pairs (BEST with many of them sorts them first); after the
// offset is published the successors' counts drop.  Returns a successor that
// became ready and is a warp item, for this warp to place next (-1 if none);
// the other ready ones are queued.
__device__ int64_t place_short(const GridWs& w, const LongCache& lc, int64_t g, int32_t policy, int64_t* buf) {
    const int lane = threadIdx.x & 31;
    const unsigned full = 0xffffffffu, lt = (1u << lane) - 1u;
    const Node x = load_node(w, g);
    const Cands c = cands_of(w, lc.lw[x.b], lc.nl[x.b], x);
    int32_t* sbuf = reinterpret_cast<int32_t*>(buf + 2 * kWarpSortPairs);
    // the predecessors' (slot, size), then all their offsets at once: one
    // round trip to L2 instead of one per round of candidates
    int32_t np = 0, ns = 0;
    warp_visit(w, lc, x, c, [&](bool hit, const Cand& cd) {
        const bool pred = hit && cand_precedes(w, x, cd);
        const unsigned pb = __ballot_sync(full, pred), sb = __ballot_sync(full, hit && !pred);
        if (pred) {
            const int32_t at = np + __popc(pb & lt);
            if (at < kWarpPairs) {
                buf[2 * at] = cd.slot;
                buf[2 * at + 1] = cd.r.s;
            }
        } else if (hit) {
            const int32_t at = ns + __popc(sb & lt);
            if (at < kWarpSuccs) sbuf[at] = (int32_t)cd.slot;
        }
        np += __popc(pb);
        ns += __popc(sb);
    });
    __syncwarp();
    if (np <= kWarpPairs) {
        for (int32_t k0 = 0; k0 < np; k0 += 32 * 4) {
            int64_t po[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int32_t k = k0 + u * 32 + lane;
                po[u] = k < np ? off_of(w, buf[2 * k]) : 0;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int32_t k = k0 + u * 32 + lane;
                if (k < np) {
                    buf[2 * k + 1] += po[u];
                    buf[2 * k] = po[u];
                }
            }
        }
    }
    __syncwarp();
    int64_t o;
    if (np > kWarpPairs) {  // not expected (such tensors are CTA items): enumerate them again on every pass
        o = warp_fit(x.r.s, policy, [&](auto&& fn) {
            warp_visit(w, lc, x, c, [&](bool hit, const Cand& cd) {
                if (hit && cand_precedes(w, x, cd)) {
                    const int64_t po = off_of(w, cd.slot);
                    fn(po, po + cd.r.s);
                }
            });
        });
    } else if (policy == MP_FIT_BEST && np > 32) {
        o = warp_sorted_fit(x.r.s, policy, buf, np);
    } else {
        o = warp_fit(x.r.s, policy, [&](auto&& fn) {
            for (int32_t k = lane; k < np; k += 32) fn(buf[2 * k], buf[2 * k + 1]);
        });
    }
    if (lane == 0) st_rlx(w.off + g, o);
    __syncwarp();
    __threadfence();  // the offset before any successor's count drops
    if (lane == 0) atomicAdd(&w.ctl->placed, 1);
    int64_t next = -1;
    if (ns <= kWarpSuccs) {
        for (int32_t k0 = 0; k0 < ns; k0 += 32) {
            const int32_t k = k0 + lane;
            const int64_t slot = k < ns ? sbuf[k] : -1;
            const bool ready = slot >= 0 && drop(w, slot);
            const bool warp_item = ready && !cta_item(w, slot);
            const unsigned keep = __ballot_sync(full, warp_item && slot != w.hold);
            const bool mine = next < 0 && keep && lane == __ffs(keep) - 1;
            if (mine) next = slot;
            next = __shfl_sync(full, next, keep ? __ffs(keep) - 1 : 0);
            if (ready && !mine) push(w, slot);
        }
    } else {
        warp_visit(w, lc, x, c, [&](bool hit, const Cand& cd) {
            if (hit && !cand_precedes(w, x, cd) && drop(w, cd.slot)) push(w, cd.slot);
        });
    }
    __syncwarp();
    return next;
}

// Exclusive prefix max (identity 0) of one value per thread; the block max in *total.
__device__ __forceinline__ int64_t cta_excl_max(int64_t v, int64_t* red, int64_t* total) {
    const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int64_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl = u > incl ? u : incl;
    }
    if (lane == 31) red[wp] = incl;
    __syncthreads();
    if (wp == 0) {
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
    const int64_t wex = red[wp];
    const int64_t r = lane == 0 ? wex : (up > wex ? up : wex);
    *total = red[32];
    __syncthreads();
    return r;
}

constexpr int32_t kJumpCap = 128;  // FIRST jumps (no merge sort) at most this often before it sorts records
constexpr int kRegJump = 6;        // predecessor pairs per thread held in registers for the jumps
constexpr int kKeyIdxBits = 13;    // the merge sort's keys: offset << 13 | pair index
constexpr int32_t kMergeMaxPairs = 1 << kKeyIdxBits;

// Ascending bitonic network over a thread's E keys (all indices compile-time).
template <int E>
__device__ __forceinline__ void sort_regs(uint64_t (&k)[E]) {
#pragma unroll
    for (int kk = 2; kk <= E; kk <<= 1) {
#pragma unroll
        for (int j = kk >> 1; j > 0; j >>= 1) {
#pragma unroll
            for (int i = 0; i < E; ++i) {
                const int l = i ^ j;
                if (l > i) {
                    const uint64_t a = k[i], b = k[l];
                    const uint64_t lo = a < b ? a : b, hi = a < b ? b : a;
                    const bool up = (i & kk) == 0;
                    k[i] = up ? lo : hi;
                    k[l] = up ? hi : lo;
                }
            }
        }
    }
}

// The merge sort's buffer: one 8-byte word of padding after every 16, so that
// lanes reading or writing words E apart (E <= 16) fall in distinct banks.
__device__ __forceinline__ int32_t mpad(int32_t i) { return i + (i >> 4); }

// The sorted gap search of a CTA item over its P <= E * blockDim predecessor
// pairs (offset, end) in the region, every offset below 2^(63 - kKeyIdxBits),
// by a merge sort of 64-bit keys (offset << kKeyIdxBits | pair index).  The
// keys are read in E chunks of blockDim pairs; each chunk's ends are then
// packed at the region's start (8 bytes per pair: they only overwrite pairs of
// earlier chunks, read before the chunk's barrier).  Each thread sorts its E
// keys in registers; then log2(blockDim) rounds merge runs of doubling length
// through a padded buffer behind the ends, each thread finding where its E
// outputs start by a merge-path search.  A final scan over the sorted keys
// exposes every gap as in the record sort.
template <int E>
__device__ int64_t merge_sort_fit(int64_t* region, int32_t P, int64_t s, int32_t policy, int64_t* red) {
    const int32_t t = (int32_t)threadIdx.x, nt = (int32_t)blockDim.x;
    const int32_t plen = E * nt;
    int64_t* ends = region;  // [0, P) once packed
    uint64_t* buf = reinterpret_cast<uint64_t*>(region + kMergeMaxPairs);
    uint64_t k[E];
#pragma unroll
    for (int c = 0; c < E; ++c) {
        const int32_t idx = c * nt + t;
        int64_t en = 0;
        k[c] = ~0ull;  // padding sorts last
        if (idx < P) {
            k[c] = ((uint64_t)region[2 * idx] << kKeyIdxBits) | (uint64_t)idx;
            en = region[2 * idx + 1];
        }
        __syncthreads();
        if (idx < P) ends[idx] = en;
    }
    sort_regs<E>(k);
    for (int32_t L = E; L < plen; L <<= 1) {
#pragma unroll
        for (int e = 0; e < E; ++e) buf[mpad(t * E + e)] = k[e];
        __syncthreads();
        const int32_t d = (t * E) & (2 * L - 1);  // my first output within my merged run
        const int32_t a0 = t * E - d, b0 = a0 + L;
        int32_t lo = max(0, d - L), hi = min(d, L);
        while (lo < hi) {  // how many of my run's first d outputs come from A (B first on ties)
            const int32_t mid = (lo + hi) >> 1;
            if (buf[mpad(a0 + mid)] < buf[mpad(b0 + d - 1 - mid)]) lo = mid + 1;
            else hi = mid;
        }
        int32_t i = lo, j = d - lo;
        uint64_t a = i < L ? buf[mpad(a0 + i)] : ~0ull, b = j < L ? buf[mpad(b0 + j)] : ~0ull;
#pragma unroll
        for (int e = 0; e < E; ++e) {
            if (a < b) {
                k[e] = a;
                ++i;
                a = i < L ? buf[mpad(a0 + i)] : ~0ull;
            } else {
                k[e] = b;
                ++j;
                b = j < L ? buf[mpad(b0 + j)] : ~0ull;
            }
        }
        __syncthreads();
    }
    // thread t holds sorted positions [t E, t E + E): the gap before position
    // p is its offset minus the largest end before it
    int64_t local = 0;
#pragma unroll
    for (int e = 0; e < E; ++e)
        if (t * E + e < P) local = max(local, ends[k[e] & (kMergeMaxPairs - 1)]);
    int64_t top;
    int64_t prev = cta_excl_max(local, red, &top);
    int64_t key = INT64_MAX, val = INT64_MAX;
#pragma unroll
    for (int e = 0; e < E; ++e) {
        if (t * E + e >= P) break;
        const int64_t off = (int64_t)(k[e] >> kKeyIdxBits);
        const int64_t gl = off - prev;
        if (gl >= s) {
            const int64_t kx = policy == MP_FIT_FIRST ? prev : gl;  // prev grows with the position
            if (kx < key || (kx == key && prev < val)) {
                key = kx;
                val = prev;
            }
        }
        prev = max(prev, ends[k[e] & (kMergeMaxPairs - 1)]);
    }
    block_min_pair(key, val, red);
    return key == INT64_MAX ? top : val;
}

// Shared state of a CTA item.
struct LongShared {
    int32_t np, ns;
};

// A tensor placed by the whole CTA (long-lived, or more predecessors than a
// warp holds).  One pass over the candidates puts the predecessors' pairs in
// the region (then in this CTA's overflow buffer, ovf) and lists the
// successors after them (if too many, they are enumerated again).  Up to
// kMergeMaxPairs pairs with offsets below 2^(63 - kKeyIdxBits) are merge
// sorted by offset (merge_sort_fit), and one scan exposes every gap (FIRST:
// the lowest that fits; BEST: the smallest, the lowest on ties).  Otherwise
// FIRST jumps to the largest conflicting end until nothing conflicts (pairs
// held in registers, one block reduction per jump); if that takes more than
// kJumpCap jumps, or for BEST, the (offset, end) records are sorted in memory
// and scanned the same way.  Successors that become ready are queued, CTA
// items too: an idle long CTA starts one while this one still drops the
// others (keeping it for this CTA measured slower).
__device__ void place_long(const GridWs& w, const LongCache& lc, int64_t g, int32_t policy, int64_t* region,
                           int64_t* ovf, int64_t* red, LongShared* sh) {
    const Node x = load_node(w, g);
    const Cands c = cands_of(w, lc.lw[x.b], lc.nl[x.b], x);
    const int32_t ncand = (c.w1 - c.w0) + c.nlong;
    const int64_t s = x.r.s;
    int32_t* succ = reinterpret_cast<int32_t*>(region + 2 * kLongPredPairs);
    if (threadIdx.x == 0) {
        sh->np = 0;
        sh->ns = 0;
    }
    __syncthreads();
    auto pair_at = [&](int32_t k) -> int64_t* { return k < kRegionPairs ? region + 2 * k : ovf + 2 * (k - kRegionPairs); };
    const int32_t stride = (int32_t)blockDim.x;
    for (int32_t k0 = threadIdx.x; k0 < ncand; k0 += stride * kU) {
        Cand cd[kU];
        bool hit[kU], pred[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) hit[u] = fetch_cand(w, lc, x, c, k0 + u * stride, &cd[u]);
#pragma unroll
        for (int u = 0; u < kU; ++u) pred[u] = hit[u] && cand_precedes(w, x, cd[u]);
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            if (pred[u]) {  // (slot, size) for now; the offsets are loaded below, all at once
                int64_t* q = pair_at(atomicAdd(&sh->np, 1));
                q[0] = cd[u].slot;
                q[1] = cd[u].r.s;
            } else if (hit[u]) {
                const int32_t at = atomicAdd(&sh->ns, 1);
                if (at < kLongSuccs) succ[at] = (int32_t)cd[u].slot;
            }
        }
    }
    __syncthreads();
    const int32_t P = sh->np, S = sh->ns;
    // the predecessors' offsets: every thread's loads in flight together; the
    // first kRegJump * blockDim pairs also stay in registers for the jumps
    int64_t ro[kRegJump], re[kRegJump];
    uint64_t obits = 0;  // the or of this thread's offsets
#pragma unroll
    for (int j = 0; j < kRegJump; ++j) {
        const int32_t k = (int32_t)threadIdx.x + j * stride;
        ro[j] = k < P ? off_of(w, pair_at(k)[0]) : 0;
        obits |= (uint64_t)ro[j];
    }
#pragma unroll
    for (int j = 0; j < kRegJump; ++j) {
        const int32_t k = (int32_t)threadIdx.x + j * stride;
        re[j] = 0;  // an empty [0, 0) pads: it never conflicts
        if (k < P) {
            int64_t* q = pair_at(k);
            re[j] = ro[j] + q[1];
            q[0] = ro[j];
            q[1] = re[j];
        }
    }
    for (int32_t k0 = (int32_t)threadIdx.x + kRegJump * stride; k0 < P; k0 += 4 * stride) {
        int64_t po[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int32_t k = k0 + u * stride;
            po[u] = k < P ? off_of(w, pair_at(k)[0]) : 0;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int32_t k = k0 + u * stride;
            if (k < P) {
                int64_t* q = pair_at(k);
                q[1] += po[u];
                q[0] = po[u];
                obits |= (uint64_t)po[u];
            }
        }
    }
    // whether some offset is too wide for the merge sort's keys
    const bool wide_keys = __syncthreads_or((obits >> (63 - kKeyIdxBits)) != 0);
    int64_t o = 0;
    const int32_t nt = (int32_t)blockDim.x;
    const bool merge = !wide_keys && P <= kMergeMaxPairs && P <= 16 * nt;
    bool sorted = !merge && policy == MP_FIT_BEST;
    if (merge) {
        o = P <= nt       ? merge_sort_fit<1>(region, P, s, policy, red)
            : P <= 2 * nt ? merge_sort_fit<2>(region, P, s, policy, red)
            : P <= 4 * nt ? merge_sort_fit<4>(region, P, s, policy, red)
            : P <= 8 * nt ? merge_sort_fit<8>(region, P, s, policy, red)
                          : merge_sort_fit<16>(region, P, s, policy, red);
    } else if (!sorted) {  // one barrier per jump: the warps' maxima alternate between two buffers
        const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5;
        for (int32_t jumps = 0;; ++jumps) {
            if (jumps == kJumpCap) {
                sorted = true;
                break;
            }
            int64_t nx = 0;
#pragma unroll
            for (int j = 0; j < kRegJump; ++j)
                if (ro[j] < o + s && o < re[j] && re[j] > nx) nx = re[j];
            for (int32_t k = (int32_t)threadIdx.x + kRegJump * stride; k < P; k += stride) {
                const int64_t* q = pair_at(k);
                const int64_t qo = q[0], qe = q[1];
                if (qo < o + s && o < qe && qe > nx) nx = qe;
            }
            nx = warp_max64(nx);
            int64_t* rb = red + (jumps & 1) * 32;
            if (lane == 0) rb[wp] = nx;
            __syncthreads();
            int64_t m = 0;
#pragma unroll
            for (int k = 0; k < kGridWarps; ++k) m = max(m, rb[k]);
            if (m <= o) break;
            o = m;
        }
        __syncthreads();  // every read of the maxima done before red is used again
    }
    if (sorted) {
        int32_t plen = 1;
        while (plen < P) plen <<= 1;
        // sort by offset: in the region's pair part if it holds plen pairs, else
        // all of them in the overflow buffer (a power of two at least
        // max_tensors): ovf[0, P - r) already holds the pairs past the region's
        // r = min(P, kRegionPairs), and the region's go behind them
        int64_t* arr = region;
        if (plen > kRegionPairs) {
            const int32_t r = min(P, kRegionPairs);
            for (int32_t k = threadIdx.x; k < r; k += blockDim.x) {
                ovf[2 * (P - r + k)] = region[2 * k];
                ovf[2 * (P - r + k) + 1] = region[2 * k + 1];
            }
            arr = ovf;
        }
        for (int32_t k = P + threadIdx.x; k < plen; k += blockDim.x) {
            arr[2 * k] = INT64_MAX;
            arr[2 * k + 1] = INT64_MAX;
        }
        __syncthreads();
        for (int32_t kk = 2; kk <= plen; kk <<= 1) {
            for (int32_t j = kk >> 1; j > 0; j >>= 1) {
                for (int32_t t = threadIdx.x; t < (plen >> 1); t += blockDim.x) {
                    const int32_t lo = 2 * t - (t & (j - 1)), hi = lo + j;
                    const bool up = (lo & kk) == 0;
                    const int64_t xo = arr[2 * lo], yo = arr[2 * hi];
                    if (up ? yo < xo : xo < yo) {
                        const int64_t xe = arr[2 * lo + 1];
                        arr[2 * lo] = yo;
                        arr[2 * hi] = xo;
                        arr[2 * lo + 1] = arr[2 * hi + 1];
                        arr[2 * hi + 1] = xe;
                    }
                }
                __syncthreads();
            }
        }
        // the gap before pair k is its offset minus the largest end before it
        const int32_t chunk = (P + blockDim.x - 1) / blockDim.x;
        const int32_t k0 = min(P, (int32_t)threadIdx.x * chunk), k1 = min(P, k0 + chunk);
        int64_t local = 0;
        for (int32_t k = k0; k < k1; ++k) local = max(local, arr[2 * k + 1]);
        int64_t top;
        int64_t prev = cta_excl_max(local, red, &top);
        int64_t key = INT64_MAX, val = INT64_MAX;
        for (int32_t k = k0; k < k1; ++k) {
            const int64_t gl = arr[2 * k] - prev;
            if (gl >= s) {
                const int64_t kx = policy == MP_FIT_FIRST ? prev : gl;  // prev grows with k
                if (kx < key || (kx == key && prev < val)) {
                    key = kx;
                    val = prev;
                }
            }
            prev = max(prev, arr[2 * k + 1]);
        }
        block_min_pair(key, val, red);
        o = key == INT64_MAX ? top : val;
    }
    if (threadIdx.x == 0) st_rlx(w.off + g, o);
    __syncthreads();
    __threadfence();
    if (threadIdx.x == 0) atomicAdd(&w.ctl->placed, 1);
    auto ready = [&](int64_t slot) {
        if (drop(w, slot)) push(w, slot);
    };
    if (S <= kLongSuccs) {  // the drops of a thread's successors in flight together
        for (int32_t k0 = threadIdx.x; k0 < S; k0 += 4 * stride) {
            int32_t old4[4];
            int64_t sl[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int32_t k = k0 + u * stride;
                sl[u] = k < S ? succ[k] : -1;
                old4[u] = sl[u] >= 0 ? atomicSub(w.cnt + sl[u], 1) : 0;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                if (old4[u] != 1) continue;
                const int64_t slot = sl[u];
                push(w, slot);
            }
        }
    } else {
        for (int32_t k0 = threadIdx.x; k0 < ncand; k0 += stride * kU) {
            Cand cd[kU];
            bool sc[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) sc[u] = fetch_cand(w, lc, x, c, k0 + u * stride, &cd[u]);
#pragma unroll
            for (int u = 0; u < kU; ++u)
                if (sc[u] && !cand_precedes(w, x, cd[u])) ready(cd[u].slot);
        }
    }
    __syncthreads();  // every successor dropped before the region is reused
}

// Waits (bounded) until queue slot h (of the queue whose fill count is *tail)
// is filled and returns its entry, or returns -1 once every tensor is placed,
// another worker gave up, or nothing was queued or placed anywhere for
// kGridSpinCycles (then it raises the flag).  Only the slot is polled often,
// at a rate set by its distance from the queue's fill point; the shared
// counters are read every eighth poll, so idle workers load the L2 little.
__device__ int32_t take_slot(const GridWs& w, const int32_t* queue, const int32_t* tail, int32_t h,
                             int32_t total) {
    GridCtl* ctl = w.ctl;
    long long idle_since = clock64();
    int32_t seen = -1, dist = 0;
    for (int32_t polls = 0;; ++polls) {
        const int32_t v = ld_rlx(queue + h);
        if (v >= 0) return v;
        if ((polls & 7) == 0) {
            if (ld_rlx(&ctl->fail)) return -1;
            const int32_t placed = ld_rlx(&ctl->placed);
            if (placed >= total) return -1;
            const int32_t t = ld_rlx(tail);
            dist = h - t;
            const int32_t act = placed + ld_rlx(&ctl->tail_s) + ld_rlx(&ctl->tail_l);
            if (act != seen) {
                seen = act;
                idle_since = clock64();
            } else if (clock64() - idle_since > kGridSpinCycles) {
                atomicExch(&ctl->fail, 1);
                return -1;
            }
        }
        __nanosleep(dist <= 0 ? 32 : dist <= 4 ? 128 : dist <= 64 ? 512 : 2048);
    }
}

// The persistent grid.  Each CTA first copies the batch's long-lived records
// into its shared-memory cache (if they fit), then all warps count
// predecessors; then the first long_ctas CTAs place CTA items (thread 0 takes
// the next long-queue slot for the whole CTA) and every warp of the others
// places warp items (each takes the next short-queue slot for itself).  A
// warp that makes a warp item ready places it next instead of queueing it; a
// CTA queues every successor it makes ready.  A worker waits only for the entry of the slot it took and
// never holds one entry while waiting for another; the lowest-ranked unplaced
// tensor of a trace is always queued or being placed, so a taken slot is
// always filled in the end.  With w.hold >= 0 (tests only) the tensor of that
// slot is never queued, so the flow starves and the wait runs out.
__global__ void __launch_bounds__(kGridThreads, 1)
k_grid_flow(mp_batch bt, int32_t policy, GridWs w, int32_t long_ctas) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ int32_t s_long, s_cbase[kGridMaxTraces + 1], s_lw[kGridMaxTraces], s_nl[kGridMaxTraces];
    __shared__ LongShared s_sh;
    int64_t* region = reinterpret_cast<int64_t*>(smem_raw);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t M = w.M;
    const int64_t slots = (int64_t)bt.n_traces * M;
    GridCtl* ctl = w.ctl;

    // the long-lived cache: trace b's records at [s_cbase[b], s_cbase[b + 1])
    LongCache lc;
    {
        unsigned char* cache = smem_raw + kRegionBytes;
        lc.s = reinterpret_cast<int64_t*>(cache);
        lc.a = reinterpret_cast<int32_t*>(cache + (size_t)kLongCache * 8);
        lc.f = lc.a + kLongCache;
        lc.q = lc.f + kLongCache;
        lc.base = nullptr;
        lc.lw = s_lw;
        lc.nl = s_nl;
        if (threadIdx.x < bt.n_traces) {
            const TraceInfo* tb = w.ti + threadIdx.x;
            s_lw[threadIdx.x] = tb->ok ? tb->lw : 1;
            s_nl[threadIdx.x] = tb->ok ? tb->nlong : 0;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int32_t at = 0;
            for (int32_t b = 0; b < bt.n_traces; ++b) {
                s_cbase[b] = at;
                at += s_nl[b];
            }
            s_cbase[bt.n_traces] = at;
        }
        __syncthreads();
        if (s_cbase[bt.n_traces] <= kLongCache) {
            for (int32_t b = 0; b < bt.n_traces; ++b) {
                const int32_t nl = s_cbase[b + 1] - s_cbase[b];
                for (int32_t k = threadIdx.x; k < nl; k += blockDim.x) {
                    const int32_t q = __ldg(w.ll + (int64_t)b * M + k);
                    const GRec r = load_rec(w, (int64_t)b * M + q);
                    const int32_t i = s_cbase[b] + k;
                    lc.s[i] = r.s;
                    lc.a[i] = r.a;
                    lc.f[i] = r.f;
                    lc.q[i] = q;
                }
            }
            lc.base = s_cbase;
        }
        __syncthreads();
    }

    // counts: a warp per tensor; the class is set before the count is added
    {
        const int64_t gw = (int64_t)blockIdx.x * kGridWarps + warp, nw = (int64_t)gridDim.x * kGridWarps;
        for (int64_t g = gw; g < slots; g += nw) {
            const int32_t b = (int32_t)(g / M), p = (int32_t)(g - (int64_t)b * M);
            const TraceInfo* tip = w.ti + b;
            if (!tip->ok || p >= tip->n) continue;
            const Node x = load_node(w, g);
            const Cands c = cands_of(w, lc.lw[b], lc.nl[b], x);
            int32_t np = 0;
            warp_visit(w, lc, x, c, [&](bool hit, const Cand& cd) {
                np += __popc(__ballot_sync(0xffffffffu, hit && cand_precedes(w, x, cd)));
            });
            if (lane == 0) {
                st_rlx(w.cls + g, (is_long(x.r) || np > kWarpPairs) ? 1 : 0);
                __threadfence();
                if (atomicAdd(w.cnt + g, np) + np == 0) push(w, g);
            }
        }
    }

    const int32_t total = ctl->total;
    if ((int32_t)blockIdx.x < long_ctas) {
        int64_t* ovf = w.ovf_pairs > 0 ? w.ovf + (int64_t)blockIdx.x * 2 * w.ovf_pairs : nullptr;
        for (;;) {
            if (threadIdx.x == 0) {
                const int32_t h = atomicAdd(&ctl->head_l, 1);
                s_long = h < total ? take_slot(w, w.ql, &ctl->tail_l, h, total) : -1;
                __threadfence();  // the predecessors' offsets after the entry
            }
            __syncthreads();
            const int64_t item = s_long;
            __syncthreads();
            if (item < 0) break;
            __threadfence();
            place_long(w, lc, item, policy, region, ovf, red, &s_sh);
        }
    } else {
        int64_t* buf = region + (int64_t)warp * (kWarpBytes / 8);
        int64_t next = -1;
        for (;;) {
            if (next < 0) {
                int32_t v = -1;
                if (lane == 0) {
                    const int32_t h = atomicAdd(&ctl->head_s, 1);
                    v = h < total ? take_slot(w, w.qs, &ctl->tail_s, h, total) : -1;
                    __threadfence();
                }
                next = __shfl_sync(0xffffffffu, v, 0);
                if (next < 0) break;
            }
            __threadfence();
            next = place_short(w, lc, next, policy, buf);
        }
    }
}

// ---------------------------------------------------------------- finish

template <bool kFused>
__global__ void __launch_bounds__(kFinishThreads) k_grid_finish(mp_batch bt, GridOut out, GridWs w) {
    const int lane = threadIdx.x & 31;
    const unsigned full = 0xffffffffu;
    const int64_t M = w.M;
    const int64_t slots = (int64_t)bt.n_traces * M;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t c0 = gw * 32; c0 < slots; c0 += nw * 32) {
        const int64_t g = c0 + lane;
        int32_t b = -1, p = 0;
        bool valid = false;
        TraceInfo* tip = nullptr;
        if (g < slots) {
            b = (int32_t)(g / M);
            p = (int32_t)(g - (int64_t)b * M);
            tip = w.ti + b;
            valid = tip->ok && p < tip->n;
        }
        int64_t end = 0;
        GRec r{};
        int32_t id = 0;
        bool wide = false;
        int32_t stop = 0;
        if (valid) {
            r = load_rec(w, g);
            id = w.rid[g];
            const int64_t o = w.off[g];
            if (o < 0) {
                tip->incomplete = 1;
            } else {
                out.offsets[tip->lo + id] = o;
                end = o + r.s;
                if (kFused) {
                    stop = w.bend[(int64_t)b * w.TS + r.f - 1];
                    if (stop - p - 1 > kGridValWide) {
                        wide = true;
                    } else {
                        for (int32_t q = p + 1; q < stop; ++q) {
                            const int64_t gq = (int64_t)b * M + q;
                            const int64_t oq = w.off[gq];
                            if (oq >= 0 && o < oq + load_rec(w, gq).s && oq < end) {
                                const uint32_t i = (uint32_t)id, j = (uint32_t)w.rid[gq];
                                atomicMin(&tip->key, ((unsigned long long)(i < j ? i : j) << 32) | (i < j ? j : i));
                            }
                        }
                    }
                }
            }
        }
        // the plan peak: one atomic per trace present in these 32 slots (the
        // lanes of one trace reduce together; ends are below 2^63)
        const unsigned same = __match_any_sync(full, b);
        const unsigned mhi = __reduce_max_sync(same, (unsigned)((uint64_t)end >> 32));
        const unsigned mlo = __reduce_max_sync(same, (unsigned)((uint64_t)end >> 32) == mhi ? (unsigned)end : 0u);
        const unsigned long long m = ((unsigned long long)mhi << 32) | mlo;
        if (valid && (same & ((1u << lane) - 1u)) == 0 && m > 0) atomicMax(&tip->peak, m);
        if (kFused) {  // windows too long for one lane: the whole warp each
            unsigned wm = __ballot_sync(full, wide);
            while (wm) {
                const int src = __ffs(wm) - 1;
                wm &= wm - 1;
                const int32_t pb = __shfl_sync(full, b, src), pp = __shfl_sync(full, p, src);
                const int32_t pstop = __shfl_sync(full, stop, src), pid = __shfl_sync(full, id, src);
                const int64_t po = __shfl_sync(full, end - r.s, src), pe = __shfl_sync(full, end, src);
                for (int32_t q = pp + 1 + lane; q < pstop; q += 32) {
                    const int64_t gq = (int64_t)pb * M + q;
                    const int64_t oq = w.off[gq];
                    if (oq >= 0 && po < oq + load_rec(w, gq).s && oq < pe) {
                        const uint32_t i = (uint32_t)pid, j = (uint32_t)w.rid[gq];
                        atomicMin(&w.ti[pb].key, ((unsigned long long)(i < j ? i : j) << 32) | (i < j ? j : i));
                    }
                }
            }
        }
    }
}

template <bool kFused>
__global__ void k_grid_final(mp_batch bt, GridOut out, GridWs w) {
    const int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= bt.n_traces) return;
    const TraceInfo ti = w.ti[b];
    if (!ti.ok) return;  // its status was written by the prep kernel
    out.plan_peak[b] = (int64_t)ti.peak;
    out.status[b] = ti.incomplete ? MP_ETIMEOUT : MP_OK;
    if (kFused) {
        const bool good = ti.key == ~0ull;
        if (out.verdict) out.verdict[b] = good ? 1 : 0;
        if (out.conflict) {
            out.conflict[2 * b] = good ? -1 : (int32_t)(ti.key >> 32);
            out.conflict[2 * b + 1] = good ? -1 : (int32_t)(ti.key & 0xffffffffu);
        }
    }
}

// ---------------------------------------------------------------- host

struct GridLayout {
    size_t ctl, ti, bend, rec, rid, off, cnt, cls, qs, ql, ll, ovf, total;
    int64_t ovf_pairs;
};

int64_t pow2_ceil(int64_t x) {
    int64_t p = 1;
    while (p < x) p <<= 1;
    return p;
}

GridLayout grid_layout(const mp_batch& bt) {
    GridLayout L;
    const size_t B = (size_t)bt.n_traces, M = (size_t)std::max(bt.max_tensors, 1), TS = (size_t)bt.max_steps;
    const size_t slots = mul_sat(B, M);
    size_t at = 0;
    auto take = [&](size_t bytes) {
        const size_t here = at;
        at = bytes > SIZE_MAX - kAlign ? SIZE_MAX : add_sat(at, align_up(bytes));
        return here;
    };
    L.ctl = take(sizeof(GridCtl));
    L.ti = take(mul_sat(B, sizeof(TraceInfo)));
    L.bend = take(mul_sat(mul_sat(B, TS), 4));
    L.rec = take(mul_sat(slots, sizeof(GRec)));
    L.rid = take(mul_sat(slots, 4));
    L.off = take(mul_sat(slots, 8));
    L.cnt = take(mul_sat(slots, 4));
    L.cls = take(mul_sat(slots, 4));
    L.qs = take(mul_sat(slots, 4));
    L.ql = take(mul_sat(slots, 4));
    L.ll = take(mul_sat(slots, 4));
    // a long-lived tensor has fewer than max_tensors predecessors; BEST sorts a
    // power of two of pairs
    L.ovf_pairs = pow2_ceil((int64_t)M) > kRegionPairs ? pow2_ceil((int64_t)M) : 0;
    L.ovf = take(mul_sat((size_t)kMaxLongCtas, mul_sat((size_t)L.ovf_pairs, 16)));
    L.total = at;
    return L;
}

GridWs grid_ws(const mp_batch& bt, const GridLayout& L, unsigned char* ws) {
    GridWs w;
    w.ctl = reinterpret_cast<GridCtl*>(ws + L.ctl);
    w.ti = reinterpret_cast<TraceInfo*>(ws + L.ti);
    w.bend = reinterpret_cast<int32_t*>(ws + L.bend);
    w.rec = reinterpret_cast<GRec*>(ws + L.rec);
    w.rid = reinterpret_cast<int32_t*>(ws + L.rid);
    w.off = reinterpret_cast<int64_t*>(ws + L.off);
    w.cnt = reinterpret_cast<int32_t*>(ws + L.cnt);
    w.cls = reinterpret_cast<int32_t*>(ws + L.cls);
    w.qs = reinterpret_cast<int32_t*>(ws + L.qs);
    w.ql = reinterpret_cast<int32_t*>(ws + L.ql);
    w.ll = reinterpret_cast<int32_t*>(ws + L.ll);
    w.ovf = reinterpret_cast<int64_t*>(ws + L.ovf);
    w.ovf_pairs = L.ovf_pairs;
    w.M = std::max(bt.max_tensors, 1);
    w.TS = bt.max_steps;
    w.hold = -1;
    return w;
}

template <bool kFused>
cudaError_t launch_grid_impl(const mp_batch& bt, const GridOut& out, void* workspace, int32_t hold,
                             cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const GridLayout L = grid_layout(bt);
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    GridWs w = grid_ws(bt, L, ws);
    w.hold = hold;
    cudaError_t e = cudaMemsetAsync(ws + L.ctl, 0, sizeof(GridCtl), stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(ws + L.qs, 0xff, L.ll - L.qs, stream);  // both queues: -1
    if (e != cudaSuccess) return e;
    k_grid_prep<kFused><<<(unsigned)bt.n_traces, kPrepThreads, 0, stream>>>(bt, out, w);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;

    const void* flow = (const void*)k_grid_flow;
    e = set_smem_limit(flow, kGridSmem);
    if (e != cudaSuccess) return e;
    int resident = 0;
    e = max_resident_ctas(flow, kGridThreads, kGridSmem, &resident);
    if (e != cudaSuccess) return e;
    const int grid = resident;
    if (grid < 2) return cudaErrorInvalidConfiguration;  // both kinds of worker need a CTA
    // a quarter of the CTAs (at most kMaxLongCtas) place CTA items, the rest warp items
    int32_t long_ctas = std::max(1, std::min(grid / 4, kMaxLongCtas));
    int32_t policy = out.policy;
    mp_batch bt_arg = bt;
    GridWs w_arg = w;
    void* args[] = {&bt_arg, &policy, &w_arg, &long_ctas};
    e = cudaLaunchCooperativeKernel(flow, dim3((unsigned)grid), dim3(kGridThreads), args, kGridSmem, stream);
    if (e != cudaSuccess) return e;

    int sms = 0, dev = 0;
    e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int64_t warps_needed = ((int64_t)bt.n_traces * w.M + 31) / 32;
    const int64_t blocks = std::min<int64_t>((warps_needed + (kFinishThreads / 32) - 1) / (kFinishThreads / 32),
                                             (int64_t)sms * 8);
    k_grid_finish<kFused><<<(unsigned)std::max<int64_t>(blocks, 1), kFinishThreads, 0, stream>>>(bt, out, w);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_grid_final<kFused><<<(unsigned)((bt.n_traces + 255) / 256), 256, 0, stream>>>(bt, out, w);
    return cudaGetLastError();
}

}  // namespace

bool grid_path(const mp_batch& bt) {
    return bt.max_tensors > kGridMinTensors && bt.n_traces <= kGridMaxTraces &&
           (int64_t)bt.n_traces * (int64_t)bt.max_tensors <= INT32_MAX;
}

size_t grid_workspace_bytes(const mp_batch& bt) { return bt.n_traces == 0 ? 0 : grid_layout(bt).total; }

cudaError_t launch_grid_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                             int32_t* status, void* workspace, int32_t hold, cudaStream_t stream) {
    const GridOut out{policy, offsets, plan_peak, status, nullptr, nullptr, nullptr, nullptr};
    return launch_grid_impl<false>(bt, out, workspace, hold, stream);
}

cudaError_t launch_grid_fused(const mp_batch& bt, int32_t policy, int64_t* profile, int64_t* peak_lb,
                              int64_t* offsets, int64_t* plan_peak, int32_t* verdict, int32_t* conflict,
                              int32_t* status, void* workspace, cudaStream_t stream) {
    const GridOut out{policy, offsets, plan_peak, status, profile, peak_lb, verdict, conflict};
    return launch_grid_impl<true>(bt, out, workspace, -1, stream);
}

}  // namespace mp
