// plan.cu -- stage 2: greedy_by_size offset assignment (Sec. 2.3; the default
// strategy of Sec. 3.2).
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
//   - at most kThreadComp tensors: one thread, entirely in registers (a
//     sorting network into priority order, then placement one by one);
//   - at most kWarpComp tensors: one warp, a tensor per lane; each lane counts
//     the members that precede it (its priority rank), then the warp places
//     rank 0, 1, ... in turn, every placed lane testing its own tensor as a
//     predecessor, with single-instruction warp reductions;
//   - larger: the whole CTA bitonic-sorts the component into priority order,
//     then places it tensor by tensor with a CTA-wide gather of the
//     overlapping placed tensors and a CTA-wide gap search.
// Batches of short-lived traces split into hundreds of tiny components per
// trace, so nearly all work runs thread- or warp-parallel with no per-tensor
// barrier.
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
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int32_t kThreadComp = 4;  // components up to this size: one thread (registers)
constexpr int32_t kWarpComp = 32;   // ... up to this size: one warp (a tensor per lane); else the CTA
constexpr int32_t kCandMax = 64;    // CTA tier: up to this many predecessors, test all candidates
constexpr int64_t kNone = INT64_MAX;

__host__ __device__ constexpr size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

__host__ __device__ inline int64_t pow2_at_least(int64_t x) {
    int64_t p = 1;
    while (p < x) p <<= 1;
    return p;
}

// A tensor in alloc-step order, and in priority order (with its offset).
template <typename I>
struct ARec {
    int64_t s;
    I a, f, id, pad;
};
template <typename I>
struct SRec {
    int64_t s, off;
    I a, f, id, pad;
};

template <typename I>
struct PlanLayout {
    size_t arec, offid, bend, cst, lst, xl, dprof, total;
    __host__ __device__ PlanLayout(int64_t n, int64_t T, bool fused) {
        arec = 0;
        offid = arec + align16((size_t)n * sizeof(ARec<I>));
        bend = offid + align16((size_t)n * 8);
        cst = bend + align16((size_t)T * 4);
        lst = cst + align16((size_t)(n + 1) * 4);
        xl = lst + align16((size_t)n * sizeof(I));
        dprof = xl + align16((size_t)n * sizeof(I));
        total = align_up(dprof + (fused ? align16(prof_padded((size_t)T) * 8) : 0));
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

// ------------------------------------------------------------- gap search

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

// ------------------------------------------------------------- one thread

// Places the component AR[p0, p0 + c), c <= kThreadComp, in registers; writes
// offsets by id and returns the largest end.
template <typename I>
__device__ int64_t place_thread(const ARec<I>* AR, int32_t p0, int32_t c, int32_t policy, int64_t* OFFID) {
    int64_t s[kThreadComp], off[kThreadComp];
    int32_t a[kThreadComp], f[kThreadComp], id[kThreadComp];
#pragma unroll
    for (int k = 0; k < kThreadComp; ++k) {
        if (k < c) {
            const ARec<I> r = AR[p0 + k];
            s[k] = r.s;
            a[k] = r.a;
            f[k] = r.f;
            id[k] = r.id;
        } else {  // sentinel: after every real tensor
            s[k] = -1;
            a[k] = f[k] = 0;
            id[k] = INT32_MAX;
        }
        off[k] = 0;
    }
    auto cx = [&](int x, int y) {  // order x before y by priority
        const bool swap = s[y] != s[x] ? s[y] > s[x] : (a[y] != a[x] ? a[y] < a[x] : id[y] < id[x]);
        if (swap) {
            int64_t t64 = s[x]; s[x] = s[y]; s[y] = t64;
            int32_t t = a[x]; a[x] = a[y]; a[y] = t;
            t = f[x]; f[x] = f[y]; f[y] = t;
            t = id[x]; id[x] = id[y]; id[y] = t;
        }
    };
    cx(0, 1); cx(2, 3); cx(0, 2); cx(1, 3); cx(1, 2);  // sorting network for four
    int64_t mx = 0;
#pragma unroll
    for (int r = 0; r < kThreadComp; ++r) {
        if (r >= c) break;
        auto each = [&](auto&& fn) {
#pragma unroll
            for (int q = 0; q < kThreadComp; ++q)
                if (q < r && a[q] < f[r] && a[r] < f[q]) fn(off[q], off[q] + s[q]);
        };
        if (policy == MP_FIT_FIRST) {
            off[r] = fit_first_scan(s[r], each);
        } else {
            int64_t top = 0;
            each([&](int64_t, int64_t pe) { top = pe > top ? pe : top; });
            off[r] = fit_best_scan(s[r], top, each);
        }
        OFFID[id[r]] = off[r];
        mx = off[r] + s[r] > mx ? off[r] + s[r] : mx;
    }
    return mx;
}

// ------------------------------------------------------------- one warp

// Warp max / min of non-negative int64 values by two 32-bit reductions
// (high words first, then the low words of the lanes holding the top high word).
__device__ __forceinline__ int64_t warp_max_nonneg(int64_t v) {
    const unsigned hi = __reduce_max_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32));
    const unsigned lo = __reduce_max_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32) == hi ? (unsigned)v : 0u);
    return (int64_t)(((uint64_t)hi << 32) | lo);
}
__device__ __forceinline__ int64_t warp_min_nonneg(int64_t v) {
    const unsigned hi = __reduce_min_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32));
    const unsigned lo = __reduce_min_sync(0xffffffffu, (unsigned)((uint64_t)v >> 32) == hi ? (unsigned)v : ~0u);
    return (int64_t)(((uint64_t)hi << 32) | lo);
}

// Places the component AR[p0, p0 + c), c <= 32, with one warp (a tensor per
// lane); every lane must call it.  Writes offsets by id; returns the largest end.
template <typename I>
__device__ int64_t place_warp(const ARec<I>* AR, int32_t p0, int32_t c, int32_t policy, int64_t* OFFID) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    const bool act = lane < c;
    ARec<I> me;
    if (act) me = AR[p0 + lane];
    const int64_t s = act ? me.s : 0;
    const int32_t a = act ? (int32_t)me.a : 0, f = act ? (int32_t)me.f : 0, id = act ? (int32_t)me.id : -1;
    int rank = 0;  // members that precede this one
    for (int l = 0; l < c; ++l) {
        const int64_t sl = __shfl_sync(full, s, l);
        const int32_t al = __shfl_sync(full, a, l), il = __shfl_sync(full, id, l);
        if (act && l != lane) rank += (sl != s ? sl > s : (al != a ? al < a : il < id)) ? 1 : 0;
    }
    int64_t off = 0, end = 0;
    bool placed = false;
    for (int r = 0; r < c; ++r) {
        const int src = __ffs(__ballot_sync(full, act && rank == r)) - 1;
        const int32_t ai = __shfl_sync(full, a, src), fi = __shfl_sync(full, f, src);
        const int64_t si = __shfl_sync(full, s, src);
        const bool pred = placed && a < fi && ai < f;  // placed: ranks below r
        int64_t o = 0;
        if (policy == MP_FIT_FIRST) {
            for (;;) {
                const int64_t mx = warp_max_nonneg((pred && off < o + si && o < end) ? end : 0);
                if (mx <= o) break;
                o = mx;
            }
        } else {
            const int64_t top = warp_max_nonneg(pred ? end : 0);
            int64_t cc = 0, best_len = kNone;
            o = top;
            while (cc < top) {
                for (;;) {  // move cc off any predecessor that covers it
                    const int64_t mx = warp_max_nonneg((pred && off <= cc && cc < end) ? end : 0);
                    if (mx <= cc) break;
                    cc = mx;
                }
                if (cc >= top) break;
                const int64_t ns = warp_min_nonneg((pred && off > cc) ? off : kNone);
                const int64_t len = ns - cc;
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
    if (act) OFFID[id] = off;
    return warp_max_nonneg(act ? end : 0);
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

struct CtaScratch {
    int64_t* red;  // >= 64 slots
    int32_t* cnt;
    unsigned long long* top;
};

// Places the priority-ordered records R[0, c) of one component with the whole
// CTA.  bo/be: workspace buffers of at least pow2_at_least(c) entries each.
template <typename I>
__device__ void place_large(SRec<I>* R, int32_t c, int32_t policy, int64_t* bo, int64_t* be, const CtaScratch& sc) {
    for (int32_t r = 0; r < c; ++r) {
        const int64_t s = R[r].s;
        const int32_t ai = R[r].a, fi = R[r].f;
        if (threadIdx.x == 0) {
            *sc.cnt = 0;
            *sc.top = 0;
        }
        __syncthreads();
        for (int32_t x = threadIdx.x; x < r; x += blockDim.x) {  // placed, lifetime-overlapping
            if (R[x].a < fi && ai < R[x].f) {
                const int64_t o = R[x].off, e = o + R[x].s;
                const int32_t pos = atomicAdd(sc.cnt, 1);
                bo[pos] = o;
                be[pos] = e;
                atomicMax(sc.top, (unsigned long long)e);
            }
        }
        __syncthreads();
        const int32_t P = *sc.cnt;
        const int64_t top = (int64_t)*sc.top;
        int64_t key = kNone, val = kNone;
        if (P <= kCandMax) {
            for (int32_t k = threadIdx.x; k <= P; k += blockDim.x) {
                const int64_t cand = k == 0 ? 0 : be[k - 1];
                if (policy == MP_FIT_FIRST) {
                    bool ok = true;
                    for (int32_t x = 0; x < P && ok; ++x) ok = !(bo[x] < cand + s && cand < be[x]);
                    if (ok && cand < key) key = val = cand;
                } else if (cand < top) {
                    int64_t next = INT64_MAX;
                    bool covered = false;
                    for (int32_t x = 0; x < P && !covered; ++x) {
                        covered = bo[x] <= cand && cand < be[x];
                        if (bo[x] >= cand && bo[x] < next) next = bo[x];
                    }
                    const int64_t gl = next - cand;
                    if (!covered && gl >= s && (gl < key || (gl == key && cand < val))) {
                        key = gl;
                        val = cand;
                    }
                }
            }
            block_min_pair(key, val, sc.red);
        } else if (policy == MP_FIT_FIRST) {
            int64_t o = 0;
            for (;;) {
                int64_t next = o;
                for (int32_t x = threadIdx.x; x < P; x += blockDim.x)
                    if (bo[x] < o + s && o < be[x] && be[x] > next) next = be[x];
                next = block_max_i64(next, sc.red);
                if (next == o) break;
                o = next;
            }
            key = val = o;
        } else {
            // Sort predecessors by offset, then gap_k = off_(k) - max end of those before k.
            const int32_t plen = (int32_t)pow2_at_least(P);
            for (int32_t x = P + threadIdx.x; x < plen; x += blockDim.x) {
                bo[x] = INT64_MAX;
                be[x] = INT64_MAX;
            }
            __syncthreads();
            for (int32_t k = 2; k <= plen; k <<= 1) {
                for (int32_t j = k >> 1; j > 0; j >>= 1) {
                    for (int32_t t = threadIdx.x; t < (plen >> 1); t += blockDim.x) {
                        const int32_t lo = 2 * t - (t & (j - 1)), hi = lo + j;
                        const bool up = (lo & k) == 0;
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
            const int32_t chunk = (P + blockDim.x - 1) / blockDim.x;
            const int32_t k0 = min(P, (int32_t)threadIdx.x * chunk), k1 = min(P, k0 + chunk);
            int64_t local = 0;
            for (int32_t k = k0; k < k1; ++k) local = be[k] > local ? be[k] : local;
            int64_t total;
            int64_t prev = block_excl_max(local, sc.red, &total);
            for (int32_t k = k0; k < k1; ++k) {
                const int64_t gl = bo[k] - prev;
                if (gl >= s && (gl < key || (gl == key && prev < val))) {
                    key = gl;
                    val = prev;
                }
                prev = be[k] > prev ? be[k] : prev;
            }
            block_min_pair(key, val, sc.red);
        }
        if (threadIdx.x == 0) R[r].off = (policy == MP_FIT_FIRST) ? key : (key == kNone ? top : val);
        __syncthreads();
    }
}

template <typename I, bool kSmem, bool kFused>
__global__ void __launch_bounds__(kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal)
k_plan(mp_batch bt, PlanOut out, unsigned char* __restrict__ ws, size_t data_stride, size_t buf_offset,
       size_t buf_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ int32_t s_cnt, s_nt, s_nw, s_nx, s_bad;
    __shared__ unsigned long long s_top, s_hi, s_lo, s_max, s_key, s_lbmax;
    const int b = blockIdx.x;
    const int32_t policy = out.policy;
    int32_t* __restrict__ status = out.status;
    const bool want_profile = kFused && out.profile != nullptr;
    const TraceView tv = load_trace(bt, b, want_profile);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const PlanLayout<I> L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps, kFused);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * data_stride;
    ARec<I>* AR = reinterpret_cast<ARec<I>*>(base + L.arec);
    int64_t* OFFID = reinterpret_cast<int64_t*>(base + L.offid);
    int32_t* BEND = reinterpret_cast<int32_t*>(base + L.bend);
    int32_t* CST = reinterpret_cast<int32_t*>(base + L.cst);
    I* LST = reinterpret_cast<I*>(base + L.lst);  // thread-tier components from the front, warp-tier from the back
    I* XL = reinterpret_cast<I*>(base + L.xl);    // CTA-tier components
    // CTA tier workspace: predecessor offsets / ends, then the priority-ordered records
    const size_t cap2 = (size_t)pow2_at_least(bt.max_tensors > 0 ? bt.max_tensors : 1);
    int64_t* bo = reinterpret_cast<int64_t*>(ws + buf_offset + (size_t)b * buf_stride);
    int64_t* be = bo + cap2;
    SRec<I>* SR = reinterpret_cast<SRec<I>*>(be + cap2);

    // ---- load, check, alloc-step histogram
    for (int t = threadIdx.x; t < T; t += blockDim.x) BEND[t] = 0;
    if (threadIdx.x == 0) {
        s_nt = s_nw = s_nx = 0;
        s_bad = 0;
        s_hi = s_lo = s_max = s_lbmax = 0;
        s_key = ~0ull;
    }
    __syncthreads();
    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    bool ok = true;
    uint64_t sum = 0;
    auto take = [&](int32_t a, int32_t f, int64_t s) {
        if (!tensor_ok(a, f, s, T)) {
            ok = false;
            return;
        }
        sum = sat_add(sum, (uint64_t)s);
        atomicAdd(BEND + a, 1);
    };
    int k0 = 0;
    if (((reinterpret_cast<uintptr_t>(Ag) | reinterpret_cast<uintptr_t>(Fg) | reinterpret_cast<uintptr_t>(Sg)) &
         15) == 0) {
        const int n4 = n >> 2;
        for (int q = threadIdx.x; q < n4; q += blockDim.x) {
            const int4 a = __ldg(reinterpret_cast<const int4*>(Ag) + q);
            const int4 f = __ldg(reinterpret_cast<const int4*>(Fg) + q);
            const longlong2 s01 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * q);
            const longlong2 s23 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * q + 1);
            take(a.x, f.x, s01.x);
            take(a.y, f.y, s01.y);
            take(a.z, f.z, s23.x);
            take(a.w, f.w, s23.y);
        }
        k0 = n4 << 2;
    }
    for (int k = k0 + threadIdx.x; k < n; k += blockDim.x) take(__ldg(Ag + k), __ldg(Fg + k), __ldg(Sg + k));
    block_add_size_sum(sum, &s_hi, &s_lo);
    if (!ok) s_bad = 1;
    __syncthreads();
    if (s_bad || size_sum_overflows(s_hi, s_lo)) {
        if (threadIdx.x == 0) {
            status[b] = s_bad ? MP_EINVAL : MP_EOVERFLOW;
            if (kFused && out.verdict) out.verdict[b] = 0;
            if (kFused && out.conflict) out.conflict[2 * b] = out.conflict[2 * b + 1] = -1;
        }
        return;
    }

    // ---- counting sort into alloc-step records (second read hits the cache)
    block_excl_scan_array<int32_t, 8>(BEND, T, reinterpret_cast<int32_t*>(red));
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k);
        ARec<I> r;
        r.s = __ldg(Sg + k);
        r.a = (I)a;
        r.f = (I)__ldg(Fg + k);
        r.id = (I)k;
        r.pad = 0;
        AR[atomicAdd(BEND + a, 1)] = r;
    }
    __syncthreads();

    // ---- live profile from the records (fused): difference array, scan, write
    if (want_profile) {
        int64_t* D = reinterpret_cast<int64_t*>(base + L.dprof);
        const int64_t dlen = (int64_t)prof_padded((size_t)T);
        for (int64_t t = threadIdx.x; t < dlen; t += blockDim.x) D[t] = 0;
        __syncthreads();
        for (int p = threadIdx.x; p < n; p += blockDim.x) {
            const ARec<I> r = AR[p];
            atomic_add_u64_split(D + prof_pos(r.a), (uint64_t)r.s);
            if (r.f < T) atomic_add_u64_split(D + prof_pos(r.f), (uint64_t)(-r.s));
        }
        __syncthreads();
        int64_t* pout = out.profile + tv.plo;
        const bool vec_out = (reinterpret_cast<uintptr_t>(pout) & 15) == 0;
        int64_t carry = 0, lmax = 0;
        for (int64_t base_t = 0; base_t < T; base_t += (int64_t)blockDim.x * kProfRun) {
            const int64_t my = base_t + (int64_t)threadIdx.x * kProfRun;
            const int64_t* run = D + prof_pos(my);
            int64_t v[kProfRun];
#pragma unroll
            for (int k = 0; k < kProfRun; k += 2) {
                if (my + kProfRun <= T) {
                    const longlong2 q = *reinterpret_cast<const longlong2*>(run + k);
                    v[k] = q.x;
                    v[k + 1] = q.y;
                } else {
                    v[k] = my + k < T ? run[k] : 0;
                    v[k + 1] = my + k + 1 < T ? run[k + 1] : 0;
                }
            }
#pragma unroll
            for (int k = 1; k < kProfRun; ++k) v[k] += v[k - 1];
            int64_t tot;
            const int64_t pre = block_excl_scan<int64_t>(v[kProfRun - 1], red, &tot) + carry;
#pragma unroll
            for (int k = 0; k < kProfRun; ++k) {
                v[k] += pre;
                lmax = v[k] > lmax ? v[k] : lmax;
            }
            if (vec_out && my + kProfRun <= T) {
#pragma unroll
                for (int k = 0; k < kProfRun; k += 2)
                    *reinterpret_cast<longlong2*>(pout + my + k) = make_longlong2(v[k], v[k + 1]);
            } else {
#pragma unroll
                for (int k = 0; k < kProfRun; ++k)
                    if (my + k < T) pout[my + k] = v[k];
            }
            carry += tot;
        }
        lmax = warp_max_i64(lmax);
        if ((threadIdx.x & 31) == 0 && lmax > 0) atomicMax(&s_lbmax, (unsigned long long)lmax);
    }

    // ---- components: a run starts where no earlier tensor is live any more
    const int32_t chunk = (n + blockDim.x - 1) / blockDim.x;
    const int32_t q0 = min(n, (int32_t)threadIdx.x * chunk), q1 = min(n, q0 + chunk);
    int64_t fmax = 0;
    for (int32_t p = q0; p < q1; ++p) fmax = max(fmax, (int64_t)AR[p].f);
    int64_t ftot;
    const int64_t run0 = block_excl_max(fmax, red, &ftot);
    int32_t starts = 0;
    {
        int64_t run = run0;
        for (int32_t p = q0; p < q1; ++p) {
            starts += (p == 0 || run <= AR[p].a) ? 1 : 0;
            run = max(run, (int64_t)AR[p].f);
        }
    }
    int32_t ncomp;
    const int32_t first = block_excl_scan<int32_t>(starts, reinterpret_cast<int32_t*>(red), &ncomp);
    {
        int64_t run = run0;
        int32_t idx = first;
        for (int32_t p = q0; p < q1; ++p) {
            if (p == 0 || run <= AR[p].a) CST[idx++] = p;
            run = max(run, (int64_t)AR[p].f);
        }
    }
    if (threadIdx.x == 0) CST[ncomp] = n;
    __syncthreads();
    for (int32_t c = threadIdx.x; c < ncomp; c += blockDim.x) {
        const int32_t sz = CST[c + 1] - CST[c];
        if (sz <= kThreadComp) LST[atomicAdd(&s_nt, 1)] = (I)c;
        else if (sz <= kWarpComp) LST[n - 1 - atomicAdd(&s_nw, 1)] = (I)c;
        else XL[atomicAdd(&s_nx, 1)] = (I)c;
    }
    __syncthreads();

    // ---- small and medium components: warps take the medium ones, then
    // every thread the small ones
    int64_t mx = 0;
    {
        const int32_t nw = s_nw, nt = s_nt, nwarps = blockDim.x >> 5;
        for (int32_t k = threadIdx.x >> 5; k < nw; k += nwarps) {
            const int32_t c = LST[n - 1 - k], p0 = CST[c];
            const int64_t e = place_warp(AR, p0, CST[c + 1] - p0, policy, OFFID);
            mx = e > mx ? e : mx;
        }
        for (int32_t k = threadIdx.x; k < nt; k += blockDim.x) {
            const int32_t c = LST[k], p0 = CST[c];
            const int64_t e = place_thread(AR, p0, CST[c + 1] - p0, policy, OFFID);
            mx = e > mx ? e : mx;
        }
    }

    // ---- large components, the whole CTA each
    const int32_t nx = s_nx;
    const CtaScratch sc{red, &s_cnt, &s_top};
    for (int32_t q = 0; q < nx; ++q) {
        const int32_t c = XL[q], p0 = CST[c], sz = CST[c + 1] - p0;
        const int32_t len = (int32_t)pow2_at_least(sz);
        int32_t* idx = reinterpret_cast<int32_t*>(bo);  // the index list lives in bo while sorting
        for (int32_t x = threadIdx.x; x < len; x += blockDim.x) idx[x] = x < sz ? p0 + x : -1;
        __syncthreads();
        block_bitonic_sort(idx, len, [&](int32_t x, int32_t y) {  // sentinels (-1) sort last
            return y < 0 ? x >= 0 : (x >= 0 && precedes(AR[x], AR[y]));
        });
        for (int32_t x = threadIdx.x; x < sz; x += blockDim.x) {
            const ARec<I> me = AR[idx[x]];
            SRec<I> out;
            out.s = me.s;
            out.off = 0;
            out.a = me.a;
            out.f = me.f;
            out.id = me.id;
            out.pad = 0;
            SR[x] = out;
        }
        __syncthreads();
        place_large(SR, sz, policy, bo, be, sc);
        for (int32_t x = threadIdx.x; x < sz; x += blockDim.x) {
            const int64_t o = SR[x].off;
            OFFID[SR[x].id] = o;
            mx = o + SR[x].s > mx ? o + SR[x].s : mx;
        }
        __syncthreads();
    }

    mx = warp_max_i64(mx);
    if ((threadIdx.x & 31) == 0 && mx > 0) atomicMax(&s_max, (unsigned long long)mx);
    __syncthreads();

    // ---- validation of the plan just made (fused): every lifetime-overlapping
    // pair once, from its earlier member in alloc order, is checked for address
    // overlap -- an independent pass over the alloc-ordered records
    if (kFused) {
        for (int p = threadIdx.x; p < n; p += blockDim.x) {
            const ARec<I> ri = AR[p];
            const int32_t stop = BEND[ri.f - 1];  // tensors with alloc < free_i
            if (stop <= p + 1) continue;
            const int64_t oi = OFFID[ri.id], ei = oi + ri.s;
            for (int q = p + 1; q < stop; ++q) {
                const ARec<I> rj = AR[q];
                const int64_t oj = OFFID[rj.id];
                if (oi < oj + rj.s && oj < ei) {
                    const uint32_t i = (uint32_t)ri.id, j = (uint32_t)rj.id;
                    atomicMin(&s_key, ((unsigned long long)(i < j ? i : j) << 32) | (i < j ? j : i));
                }
            }
        }
        __syncthreads();
    }

    // ---- outputs
    for (int k = threadIdx.x; k < n; k += blockDim.x) out.offsets[tv.lo + k] = OFFID[k];
    if (threadIdx.x == 0) {
        out.plan_peak[b] = (int64_t)s_max;
        if (kFused) {
            if (want_profile && out.peak_lb) out.peak_lb[b] = (int64_t)s_lbmax;
            const unsigned long long key = s_key;
            const bool ok = key == ~0ull;
            if (out.verdict) out.verdict[b] = ok ? 1 : 0;
            if (out.conflict) {
                out.conflict[2 * b] = ok ? -1 : (int32_t)(key >> 32);
                out.conflict[2 * b + 1] = ok ? -1 : (int32_t)(key & 0xffffffffu);
            }
        }
        status[b] = MP_OK;
    }
}

struct PlanGeometry {
    bool smem, narrow;
    size_t data, data_stride, buf_offset, buf_stride, workspace;
};

// 16-bit indices when every id and step fits; shared memory when the trace's
// working set fits under the ceiling, else a workspace slice per trace.  The
// workspace always holds the CTA tier's buffers (predecessor offsets / ends,
// the index list of a large component, and its records in priority order),
// sized for up to max_tensors.
PlanGeometry plan_geometry(const mp_batch& bt, bool fused) {
    PlanGeometry g;
    g.narrow = bt.max_tensors < 32767 && bt.max_steps <= 32767;
    g.data = g.narrow ? PlanLayout<int16_t>(bt.max_tensors, bt.max_steps, fused).total
                      : PlanLayout<int32_t>(bt.max_tensors, bt.max_steps, fused).total;
    g.smem = g.data <= kPlanSmemLimit;
    g.data_stride = g.smem ? 0 : g.data;
    g.buf_offset = (size_t)bt.n_traces * g.data_stride;
    const size_t cap2 = (size_t)pow2_at_least(bt.max_tensors > 0 ? bt.max_tensors : 1);
    g.buf_stride = align_up(cap2 * 16 + (size_t)bt.max_tensors * (g.narrow ? sizeof(SRec<int16_t>) : sizeof(SRec<int32_t>)));
    g.workspace = bt.n_traces == 0 ? 0 : g.buf_offset + (size_t)bt.n_traces * g.buf_stride;
    return g;
}

template <typename I, bool kSmem, bool kFused>
cudaError_t launch_variant(const mp_batch& bt, const PlanGeometry& g, const PlanOut& out, unsigned char* ws,
                           cudaStream_t stream) {
    const size_t smem = kSmem ? g.data : 0;
    if (kSmem) {
        cudaError_t e = set_smem_limit((const void*)k_plan<I, kSmem, kFused>, smem);
        if (e != cudaSuccess) return e;
    }
    k_plan<I, kSmem, kFused>
        <<<(unsigned)bt.n_traces, kSmem ? kPlanThreadsSmem : kPlanThreadsGlobal, smem, stream>>>(
            bt, out, ws, g.data_stride, g.buf_offset, g.buf_stride);
    return cudaGetLastError();
}

template <bool kFused>
cudaError_t launch_any(const mp_batch& bt, const PlanOut& out, void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const PlanGeometry g = plan_geometry(bt, kFused);
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    if (g.narrow)
        return g.smem ? launch_variant<int16_t, true, kFused>(bt, g, out, ws, stream)
                      : launch_variant<int16_t, false, kFused>(bt, g, out, ws, stream);
    return g.smem ? launch_variant<int32_t, true, kFused>(bt, g, out, ws, stream)
                  : launch_variant<int32_t, false, kFused>(bt, g, out, ws, stream);
}

}  // namespace

// One workspace size serves both the planner and the fused entry point.
size_t plan_workspace_bytes(const mp_batch& bt) {
    const size_t a = plan_geometry(bt, false).workspace, b = plan_geometry(bt, true).workspace;
    return a > b ? a : b;
}

cudaError_t launch_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                        int32_t* status, void* workspace, cudaStream_t stream) {
    const PlanOut out{policy, offsets, plan_peak, status, nullptr, nullptr, nullptr, nullptr};
    return launch_any<false>(bt, out, workspace, stream);
}

cudaError_t launch_plan_fused(const mp_batch& bt, int32_t policy, int64_t* profile, int64_t* peak_lb,
                              int64_t* offsets, int64_t* plan_peak, int32_t* verdict, int32_t* conflict,
                              int32_t* status, void* workspace, cudaStream_t stream) {
    const PlanOut out{policy, offsets, plan_peak, status, profile, peak_lb, verdict, conflict};
    return launch_any<true>(bt, out, workspace, stream);
}

}  // namespace mp
