// breadth.cu -- greedy by breadth, the strategy of Pisarchyk et al. that
// Sec. 6 discusses: operators are taken by breadth (the sizes of their input
// and output tensors) descending, and each assigns offsets to its tensors not
// yet placed, largest first, by greedy_by_size's gap search.  A trace has one
// operator per step and no consumer lists, so the operator at step t is read
// as producing the tensors allocated at t and using for the last time the
// tensors freed at t + 1: its breadth is the bytes of both (a tensor of one
// step counts once), and a tensor is placed by the wider of its producer and
// its last user.  The order is therefore: that breadth descending, that
// operator's step (the earlier on ties), then size descending, alloc step
// ascending, id ascending.
//
// GPU form: one CTA per trace, in two kernels.  k_breadth_comp places every
// trace whose working set fits in shared memory by lifetime components (see
// its comment below): a thread, a warp or the whole CTA per component.  The
// traces it leaves (a large component that outgrows its scratch) and batches
// that do not fit go to k_breadth: the breadths (two integer atomics per
// tensor, order-independent), each tensor's wider operator, an in-place
// odd-even merge sort of the ids by that order, then placement tensor by
// tensor: all warps gather the placed tensors whose lifetimes overlap the
// next one (one shared counter update per warp) and warp 0 runs the gap
// search with warp reductions.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int32_t kBDeferred = -2;  // status of a trace left by k_breadth_comp to k_breadth

// Per-trace working set: the breadth of the operator at each step; per tensor
// (by id) its operator's breadth and step, (alloc, free), size and offset; the priority order; the
// gathered predecessors' offsets and ends.
struct BreadthLayout {
    size_t prof, km, kt, ord, af, sz, off, pb, pe, total;
    __host__ __device__ BreadthLayout(int64_t n, int64_t T) {
        prof = 0;
        km = prof + align_up((size_t)T * 8);
        kt = km + align_up((size_t)n * 8);
        ord = kt + align_up((size_t)n * 4);
        af = ord + align_up((size_t)n * 4);
        sz = af + align_up((size_t)n * 8);
        off = sz + align_up((size_t)n * 8);
        pb = off + align_up((size_t)n * 8);
        pe = pb + align_up((size_t)n * 8);
        total = pe + align_up((size_t)n * 8);
    }
};

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

// Gap search by one warp over P predecessors (pb / pe), each lane taking every
// 32nd: FIRST jumps to the largest end among the conflicting ones until none
// conflicts; BEST walks the free holes below the top and keeps the smallest
// that fits (the lowest on ties), else the top.  Every lane returns the offset.
__device__ int64_t warp_gap_search(int32_t policy, int64_t s, const int64_t* pb, const int64_t* pe, int32_t P) {
    const int lane = threadIdx.x & 31;
    int64_t o = 0;
    if (policy == MP_FIT_FIRST) {
        for (;;) {
            int64_t next = 0;
            for (int32_t k = lane; k < P; k += 32)
                if (pb[k] < o + s && o < pe[k] && pe[k] > next) next = pe[k];
            next = warp_max_nonneg(next);
            if (next <= o) return o;
            o = next;
        }
    }
    int64_t top = 0;
    for (int32_t k = lane; k < P; k += 32) top = pe[k] > top ? pe[k] : top;
    top = warp_max_nonneg(top);
    int64_t c = 0, best_len = INT64_MAX;
    o = top;
    while (c < top) {
        for (;;) {  // move c off any predecessor that covers it
            int64_t next = 0;
            for (int32_t k = lane; k < P; k += 32)
                if (pb[k] <= c && c < pe[k] && pe[k] > next) next = pe[k];
            next = warp_max_nonneg(next);
            if (next <= c) break;
            c = next;
        }
        if (c >= top) break;
        int64_t ns = INT64_MAX;
        for (int32_t k = lane; k < P; k += 32)
            if (pb[k] > c && pb[k] < ns) ns = pb[k];
        ns = warp_min_nonneg(ns);
        const int64_t len = ns - c;
        if (len >= s && len < best_len) {
            best_len = len;
            o = c;
        }
        c = ns;
    }
    return o;
}

// Odd-even merge sort (Batcher) of keys[0, n) in place by `before`, for any n
// (a comparator whose upper index falls past n would only meet padding that
// sorts last).  Every thread of the block must call it.
template <typename Before>
__device__ void block_sort_ids(int32_t* keys, int32_t n, Before&& before) {
    for (int32_t lp = 0; (1 << lp) < n; ++lp) {
        const int32_t p = 1 << lp;
        for (int32_t lk = lp; lk >= 0; --lk) {
            const int32_t k = 1 << lk, j0 = k == p ? 0 : k;
            const int32_t umax = ((n >> (lk + 1)) + 1) << lk;
            for (int32_t u = threadIdx.x; u < umax; u += blockDim.x) {
                const int32_t m = j0 + ((u >> lk) << (lk + 1)) + (u & (k - 1));
                if (m + k < n && (m >> (lp + 1)) == ((m + k) >> (lp + 1))) {
                    const int32_t x = keys[m], y = keys[m + k];
                    if (before(y, x)) {
                        keys[m] = y;
                        keys[m + k] = x;
                    }
                }
            }
            __syncthreads();
        }
    }
}

template <bool kSmem>
__global__ void __launch_bounds__(kBreadthThreads)
k_breadth(mp_batch bt, int32_t policy, int64_t* __restrict__ offsets, int64_t* __restrict__ plan_peak,
          int32_t* __restrict__ status, unsigned char* __restrict__ ws, size_t ws_stride, bool deferred_only) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ int32_t s_cnt, s_bad;
    __shared__ unsigned long long s_hi, s_lo;
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned lt = (1u << lane) - 1u;
    if (deferred_only && status[b] != kBDeferred) return;  // placed by k_breadth_comp
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) {
            status[b] = tv.st;
            plan_peak[b] = 0;
        }
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const BreadthLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * ws_stride;
    int64_t* PROF = reinterpret_cast<int64_t*>(base + L.prof);
    int64_t* KM = reinterpret_cast<int64_t*>(base + L.km);
    int32_t* KT = reinterpret_cast<int32_t*>(base + L.kt);
    int32_t* ORD = reinterpret_cast<int32_t*>(base + L.ord);
    int2* AF = reinterpret_cast<int2*>(base + L.af);
    int64_t* SZ = reinterpret_cast<int64_t*>(base + L.sz);
    int64_t* OFF = reinterpret_cast<int64_t*>(base + L.off);
    int64_t* PB = reinterpret_cast<int64_t*>(base + L.pb);
    int64_t* PE = reinterpret_cast<int64_t*>(base + L.pe);

    for (int t = threadIdx.x; t < T; t += blockDim.x) PROF[t] = 0;
    if (threadIdx.x == 0) {
        s_bad = 0;
        s_hi = s_lo = 0;
    }
    __syncthreads();
    bool bad = false;
    uint64_t sum = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(bt.alloc_step + tv.lo + k), f = __ldg(bt.free_step + tv.lo + k);
        const int64_t s = __ldg(bt.size_bytes + tv.lo + k);
        if (!tensor_ok(a, f, s, T)) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        AF[k] = make_int2(a, f);
        SZ[k] = s;
        ORD[k] = k;
        // outputs of the operator at a, inputs of the operator at f - 1 (a
        // tensor counts for two operators at most: the sums stay below 2^64)
        atomic_add_u64_split(PROF + a, (uint64_t)s);
        if (f - 1 != a) atomic_add_u64_split(PROF + (f - 1), (uint64_t)s);
    }
    block_add_size_sum(sum, &s_hi, &s_lo);
    if (bad) s_bad = 1;
    __syncthreads();
    if (s_bad || size_sum_overflows(s_hi, s_lo)) {
        if (threadIdx.x == 0) {
            status[b] = s_bad ? MP_EINVAL : MP_EOVERFLOW;
            plan_peak[b] = 0;
        }
        return;
    }
    // PROF[t] (as uint64): the breadth of the operator at step t.  Each
    // tensor's operator: the wider of its producer and its last user, the
    // earlier one on ties
    const uint64_t* BR = reinterpret_cast<const uint64_t*>(PROF);
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int2 af = AF[k];
        uint64_t m = BR[af.x];
        int32_t tm = af.x;
        if (BR[af.y - 1] > m) {
            m = BR[af.y - 1];
            tm = af.y - 1;
        }
        KM[k] = (int64_t)m;
        KT[k] = tm;
    }
    __syncthreads();
    block_sort_ids(ORD, n, [&](int32_t x, int32_t y) {
        if (KM[x] != KM[y]) return (uint64_t)KM[x] > (uint64_t)KM[y];
        if (KT[x] != KT[y]) return KT[x] < KT[y];
        if (SZ[x] != SZ[y]) return SZ[x] > SZ[y];
        if (AF[x].x != AF[y].x) return AF[x].x < AF[y].x;
        return x < y;
    });

    // placement in that order
    for (int32_t r = 0; r < n; ++r) {
        if (threadIdx.x == 0) s_cnt = 0;
        __syncthreads();  // the previous offset is written, the counter reset
        const int32_t i = ORD[r];
        const int2 me = AF[i];
        for (int32_t x0 = warp * 32; x0 < r; x0 += blockDim.x) {
            const int32_t x = x0 + lane;
            bool ov = false;
            int32_t j = 0;
            if (x < r) {
                j = ORD[x];
                const int2 o = AF[j];
                ov = o.x < me.y && me.x < o.y;
            }
            const unsigned m = __ballot_sync(0xffffffffu, ov);
            if (m == 0) continue;
            const int leader = __ffs(m) - 1;
            int32_t at = 0;
            if (lane == leader) at = atomicAdd(&s_cnt, __popc(m));
            at = __shfl_sync(0xffffffffu, at, leader) + __popc(m & lt);
            if (ov) {
                PB[at] = OFF[j];
                PE[at] = OFF[j] + SZ[j];
            }
        }
        __syncthreads();  // the predecessors are gathered
        if (warp == 0) {
            const int64_t o = warp_gap_search(policy, SZ[i], PB, PE, s_cnt);
            if (lane == 0) OFF[i] = o;
        }
    }
    __syncthreads();
    int64_t mx = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        offsets[tv.lo + k] = OFF[k];
        mx = OFF[k] + SZ[k] > mx ? OFF[k] + SZ[k] : mx;
    }
    mx = block_max_i64(mx, red);
    if (threadIdx.x == 0) {
        plan_peak[b] = mx;
        status[b] = MP_OK;
    }
}

bool breadth_fits_smem(const mp_batch& bt) {
    return BreadthLayout(bt.max_tensors, bt.max_steps).total <= kSmemCeiling;
}

// ------------------------------------------------------------- components
// Lifetime components are independent under any placement order (a tensor's
// offset depends only on placed tensors whose lifetimes overlap its own), so
// traces are placed by k_breadth_comp: one CTA per trace counting-sorts the
// tensors by alloc step into records carrying their order keys, finds the
// components (a run starts where no earlier tensor is still live), and places
// each component in the breadth order -- one thread for up to kBThreadComp
// members, one warp (a member per lane) for up to kBWarpComp, the whole CTA
// beyond.  Traces with more than kBBigComps such large components or one too
// large for the CTA tier's scratch, and batches whose working set does not
// fit in shared memory, are left to k_breadth (status kBDeferred in between).

// Exclusive prefix maximum (identity 0) of one non-negative value per thread
// over the block; ends with a barrier.  red: >= 33 slots.
__device__ int32_t block_excl_max_i32(int32_t v, int32_t* red) {
    const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int32_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl = max(incl, u);
    }
    if (lane == 31) red[wp] = incl;
    __syncthreads();
    if (wp == 0) {
        const int32_t x = lane < nw ? red[lane] : 0;
        int32_t xi = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t u = __shfl_up_sync(0xffffffffu, xi, o);
            if (lane >= o) xi = max(xi, u);
        }
        const int32_t ex = __shfl_up_sync(0xffffffffu, xi, 1);
        if (lane < nw) red[lane] = lane == 0 ? 0 : ex;
    }
    __syncthreads();
    const int32_t up = __shfl_up_sync(0xffffffffu, incl, 1);
    const int32_t r = lane == 0 ? red[wp] : max(up, red[wp]);
    __syncthreads();
    return r;
}
constexpr int32_t kBThreadComp = 8;
constexpr int32_t kBWarpComp = 32;
constexpr int32_t kBBigComps = 64;  // components of more than kBWarpComp members a trace may have here

// A tensor in alloc-step order with the keys of the breadth order.
struct BRec {
    uint64_t m;    // breadth of its wider operator
    int64_t s;     // size
    int32_t a, f;  // lifetime [a, f)
    int32_t t;     // that operator's step
    int32_t id;    // tensor id in the trace
};

// x comes before y: breadth descending, operator step, size descending, alloc
// step, id.
__device__ __forceinline__ bool b_before(const BRec& x, const BRec& y) {
    if (x.m != y.m) return x.m > y.m;
    if (x.t != y.t) return x.t < y.t;
    if (x.s != y.s) return x.s > y.s;
    if (x.a != y.a) return x.a < y.a;
    return x.id < y.id;
}

struct BCompLayout {
    size_t br, bend, rec, off, rk, sb, lst, byr, total;
    __host__ __device__ BCompLayout(int64_t n, int64_t T) {
        br = 0;
        bend = br + align16b((size_t)T * 8);
        rec = bend + align16b((size_t)T * 4);
        off = rec + align16b((size_t)n * sizeof(BRec));
        rk = off + align16b((size_t)n * 8);
        sb = rk + align16b((size_t)n * 4);
        lst = sb + align16b((size_t)((n + 31) / 32) * 4);
        byr = lst + align16b((size_t)n * 4);
        total = byr + align16b((size_t)n);
    }
    __host__ __device__ static size_t align16b(size_t x) { return (x + 15) / 16 * 16; }
};

// The CTA tier's scratch (the per-step arrays, 12 bytes a step) holds a
// component of c members: its order and the gathered (offset, end) pairs.
__device__ __forceinline__ bool big_fits(int32_t c, int32_t T) {
    return BCompLayout::align16b((size_t)c * 4) + (size_t)c * 16 <=
           BCompLayout::align16b((size_t)T * 8) + BCompLayout::align16b((size_t)T * 4);
}

// One thread places a component of c <= kBThreadComp members at positions
// [p0, p0 + c), whose ranks in the breadth order and predecessor masks (the
// earlier-ranked members whose lifetimes overlap, as bits of the member
// index) were computed per member (RK[p] = mask << 8 | rank; BYR[p0 + r]: the
// member of rank r).  Each member in rank order: FIRST jumps to the largest
// conflicting end; BEST walks the free holes below the top in address order
// (the smallest that fits, the lowest on ties, else the top).
__device__ void place_comp_thread(const BRec* __restrict__ R, int64_t* __restrict__ OFF,
                                  const int32_t* __restrict__ RK, const uint8_t* __restrict__ BYR, int32_t p0,
                                  int32_t c, int32_t policy) {
    for (int32_t r = 0; r < c; ++r) {
        const int32_t i = BYR[p0 + r];
        const int64_t s = R[p0 + i].s;
        const uint32_t mask = (uint32_t)RK[p0 + i] >> 8;
        int64_t o = 0;
        if (mask != 0) {
            if (policy == MP_FIT_FIRST) {
                for (;;) {
                    int64_t nx = 0;
                    for (uint32_t m = mask; m; m &= m - 1) {
                        const int32_t j = p0 + __ffs(m) - 1;
                        const int64_t oj = OFF[j], ej = oj + R[j].s;
                        if (oj < o + s && o < ej && ej > nx) nx = ej;
                    }
                    if (nx <= o) break;
                    o = nx;
                }
            } else {
                int64_t top = 0;
                for (uint32_t m = mask; m; m &= m - 1) {
                    const int32_t j = p0 + __ffs(m) - 1;
                    top = max(top, OFF[j] + R[j].s);
                }
                int64_t cc = 0, best = -1, best_gap = 0;
                for (;;) {
                    for (;;) {  // move cc past every member that covers it
                        int64_t nx = cc;
                        for (uint32_t m = mask; m; m &= m - 1) {
                            const int32_t j = p0 + __ffs(m) - 1;
                            const int64_t oj = OFF[j], ej = oj + R[j].s;
                            if (oj <= cc && cc < ej) nx = max(nx, ej);
                        }
                        if (nx == cc) break;
                        cc = nx;
                    }
                    if (cc >= top) break;
                    int64_t ns = INT64_MAX;
                    for (uint32_t m = mask; m; m &= m - 1) {
                        const int32_t j = p0 + __ffs(m) - 1;
                        if (OFF[j] > cc) ns = min(ns, OFF[j]);
                    }
                    const int64_t gap = ns - cc;
                    if (gap >= s && (best < 0 || gap < best_gap)) {
                        best = cc;
                        best_gap = gap;
                    }
                    cc = ns;
                }
                o = best >= 0 ? best : top;
            }
        }
        OFF[p0 + i] = o;
    }
}

// One warp places a component of kBThreadComp < c <= kBWarpComp members, a
// member per lane: each lane counts the members before it, then the lanes
// place rank 0, 1, ... in turn with warp reductions over the earlier-ranked
// members that overlap the placed one (the same FIRST and BEST as above).
__device__ void place_comp_warp(const BRec* __restrict__ R, int64_t* __restrict__ OFF, int32_t p0, int32_t c,
                                int32_t policy) {
    const unsigned full = 0xffffffffu;
    const int lane = threadIdx.x & 31;
    const bool act = lane < c;
    BRec me{};
    if (act) me = R[p0 + lane];
    int32_t rank = 0;
    for (int32_t j = 0; j < c; ++j) {
        const BRec o = R[p0 + j];
        if (act && j != lane && b_before(o, me)) ++rank;
    }
    int64_t myoff = 0;
    for (int32_t r = 0; r < c; ++r) {
        const int L = __ffs(__ballot_sync(full, act && rank == r)) - 1;
        const int32_t La = __shfl_sync(full, me.a, L), Lf = __shfl_sync(full, me.f, L);
        const int64_t Ls = __shfl_sync(full, me.s, L);
        const bool pred = act && rank < r && me.a < Lf && La < me.f;
        const int64_t pe = myoff + me.s;
        int64_t o = 0;
        if (policy == MP_FIT_FIRST) {
            for (;;) {
                const int64_t nx = warp_max_nonneg(pred && myoff < o + Ls && o < pe ? pe : 0);
                if (nx <= o) break;
                o = nx;
            }
        } else {
            const int64_t top = warp_max_nonneg(pred ? pe : 0);
            int64_t cc = 0, best = -1, best_gap = 0;
            for (;;) {
                for (;;) {
                    const int64_t nx = warp_max_nonneg(pred && myoff <= cc && cc < pe ? pe : cc);
                    if (nx == cc) break;
                    cc = nx;
                }
                if (cc >= top) break;
                const int64_t ns = warp_min_nonneg(pred && myoff > cc ? myoff : INT64_MAX);
                const int64_t gap = ns - cc;
                if (gap >= Ls && (best < 0 || gap < best_gap)) {
                    best = cc;
                    best_gap = gap;
                }
                cc = ns;
            }
            o = best >= 0 ? best : top;
        }
        if (lane == L) myoff = o;
    }
    if (act) OFF[p0 + lane] = myoff;
}

__global__ void __launch_bounds__(kBreadthThreads)
k_breadth_comp(mp_batch bt, int32_t policy, int64_t* __restrict__ offsets, int64_t* __restrict__ plan_peak,
               int32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ int32_t s_bad, s_defer, s_nt, s_nw, s_nb, s_cnt, s_bin[kBThreadComp - 1], s_base[kBThreadComp];
    __shared__ int32_t s_mbase[kBThreadComp];    // the thread tier's members, by size class
    __shared__ uint32_t s_magic[kBThreadComp - 1];  // ceil(2^32 / c) of each size class
    __shared__ int32_t s_big[kBBigComps];
    __shared__ unsigned long long s_hi, s_lo;
    const int b = blockIdx.x;
    const int tid = threadIdx.x, nthr = blockDim.x, warp = tid >> 5, nwarps = nthr >> 5;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (tid == 0) {
            status[b] = tv.st;
            plan_peak[b] = 0;
        }
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const BCompLayout L(n, T);
    uint64_t* BR = reinterpret_cast<uint64_t*>(smem_raw + L.br);
    int32_t* BEND = reinterpret_cast<int32_t*>(smem_raw + L.bend);
    BRec* R = reinterpret_cast<BRec*>(smem_raw + L.rec);
    int64_t* OFF = reinterpret_cast<int64_t*>(smem_raw + L.off);
    int32_t* RK = reinterpret_cast<int32_t*>(smem_raw + L.rk);
    uint32_t* SB = reinterpret_cast<uint32_t*>(smem_raw + L.sb);
    int32_t* LST = reinterpret_cast<int32_t*>(smem_raw + L.lst);
    uint8_t* BYR = reinterpret_cast<uint8_t*>(smem_raw + L.byr);
    const int32_t* Ag = bt.alloc_step + tv.lo;
    const int32_t* Fg = bt.free_step + tv.lo;
    const int64_t* Sg = bt.size_bytes + tv.lo;
    const int32_t nwords = (n + 31) >> 5;
    for (int32_t t = tid; t < T; t += nthr) {
        BR[t] = 0;
        BEND[t] = 0;
    }
    for (int32_t w = tid; w < nwords; w += nthr) SB[w] = 0;
    if (tid == 0) {
        s_bad = s_defer = s_nt = s_nw = s_nb = 0;
        s_hi = s_lo = 0;
    }
    if (tid < kBThreadComp - 1) s_bin[tid] = 0;
    __syncthreads();
    // checks, operator breadths (as in k_breadth) and the alloc-step histogram
    bool bad = false;
    uint64_t sum = 0;
    for (int32_t k = tid; k < n; k += nthr) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t sz = __ldg(Sg + k);
        if (!tensor_ok(a, f, sz, T)) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)sz);
        atomic_add_u64_split(reinterpret_cast<int64_t*>(BR) + a, (uint64_t)sz);
        if (f - 1 != a) atomic_add_u64_split(reinterpret_cast<int64_t*>(BR) + (f - 1), (uint64_t)sz);
        atomicAdd(BEND + a, 1);
    }
    block_add_size_sum(sum, &s_hi, &s_lo);
    if (bad) s_bad = 1;
    __syncthreads();
    if (s_bad || size_sum_overflows(s_hi, s_lo)) {
        if (tid == 0) {
            status[b] = s_bad ? MP_EINVAL : MP_EOVERFLOW;
            plan_peak[b] = 0;
        }
        return;
    }
    block_excl_scan_array<int32_t, 8>(BEND, T, reinterpret_cast<int32_t*>(red));
    // records in alloc-step order, each with its wider operator (the earlier
    // one on ties)
    for (int32_t k = tid; k < n; k += nthr) {
        BRec r;
        r.a = __ldg(Ag + k);
        r.f = __ldg(Fg + k);
        r.s = __ldg(Sg + k);
        r.id = k;
        r.m = BR[r.a];
        r.t = r.a;
        if (BR[r.f - 1] > r.m) {
            r.m = BR[r.f - 1];
            r.t = r.f - 1;
        }
        R[atomicAdd(BEND + r.a, 1)] = r;
    }
    __syncthreads();
    // component starts: position p starts one when every earlier tensor is
    // freed by a_p (prefix maximum of the free steps over contiguous chunks)
    {
        const int32_t chunk = (n + nthr - 1) / nthr;
        const int32_t q0 = min(n, tid * chunk), q1 = min(n, q0 + chunk);
        int32_t local = 0;
        for (int32_t q = q0; q < q1; ++q) local = max(local, R[q].f);
        int32_t run = block_excl_max_i32(local, reinterpret_cast<int32_t*>(red));
        for (int32_t q = q0; q < q1; ++q) {
            if (q == 0 || run <= R[q].a) atomicOr(SB + (q >> 5), 1u << (q & 31));
            run = max(run, R[q].f);
        }
    }
    __syncthreads();
    // every component start finds its size: a single tensor sits at 0; the
    // components are counted by tier and size
    auto size_from = [&](int32_t p0) {  // distance from a start to the next one
        int32_t w = p0 >> 5;
        uint32_t m = SB[w] & ~((2u << (p0 & 31)) - 1u);
        while (m == 0 && ++w < nwords) m = SB[w];
        return (m ? (w << 5) + __ffs(m) - 1 : n) - p0;
    };
    for (int32_t p = tid; p < n; p += nthr) {
        if (!((SB[p >> 5] >> (p & 31)) & 1u)) continue;
        const int32_t c = size_from(p);
        if (c == 1) {
            OFF[p] = 0;
        } else if (c <= kBThreadComp) {
            atomicAdd(&s_bin[kBThreadComp - c], 1);
        } else if (c <= kBWarpComp) {
            LST[n - 1 - atomicAdd(&s_nw, 1)] = p * 64 + c;
        } else {  // the CTA tier, while its scratch holds the component
            const int32_t at = atomicAdd(&s_nb, 1);
            if (at < kBBigComps && big_fits(c, T)) s_big[at] = p;
            else s_defer = 1;
        }
    }
    __syncthreads();
    if (s_defer) {  // too many large components, or one too large: the per-tensor kernel places this trace
        if (tid == 0) status[b] = kBDeferred;
        return;
    }
    if (tid == 0) {  // thread-tier components in descending size: bin starts, then cursors; member counts
        int32_t at = 0, mat = 0;
        for (int32_t k = 0; k < kBThreadComp - 1; ++k) {
            s_base[k] = at;
            s_mbase[k] = mat;
            s_magic[k] = 0xffffffffu / (uint32_t)(kBThreadComp - k) + 1u;
            at += s_bin[k];
            mat += s_bin[k] * (kBThreadComp - k);
            s_bin[k] = s_base[k];
        }
        s_nt = at;
        s_mbase[kBThreadComp - 1] = mat;
    }
    __syncthreads();
    for (int32_t p = tid; p < n; p += nthr) {
        if (!((SB[p >> 5] >> (p & 31)) & 1u)) continue;
        const int32_t c = size_from(p);
        if (c >= 2 && c <= kBThreadComp) LST[atomicAdd(&s_bin[kBThreadComp - c], 1)] = p * 64 + c;
    }
    __syncthreads();
    // members of the thread tier's components, one thread per member in the
    // size-sorted component list (so a warp's members mostly share one
    // component size): each gets its rank in the breadth order and the mask
    // of the earlier-ranked members that overlap its lifetime
    {
        int32_t mb[kBThreadComp];
#pragma unroll
        for (int k = 0; k < kBThreadComp; ++k) mb[k] = s_mbase[k];
        for (int32_t g = tid; g < mb[kBThreadComp - 1]; g += nthr) {
            int bin = 0;
            int32_t below = 0;  // members of the classes before bin
#pragma unroll
            for (int k = 1; k < kBThreadComp - 1; ++k) {
                if (g >= mb[k]) {
                    bin = k;
                    below = mb[k];
                }
            }
            const int32_t c = kBThreadComp - bin;
            const uint32_t r = (uint32_t)(g - below);
            const int32_t k = (int32_t)__umulhi(r, s_magic[bin]);  // r / c (r < 2^28)
            const int32_t p0 = LST[s_base[bin] + k] >> 6;
            const int32_t p = p0 + ((int32_t)r - k * c);
            const BRec me = R[p];
            uint32_t rank = 0, mask = 0;
            for (int32_t j = 0; j < c; ++j) {
                if (p0 + j == p) continue;
                const BRec o = R[p0 + j];
                if (b_before(o, me)) {
                    ++rank;
                    if (o.a < me.f && me.a < o.f) mask |= 1u << j;
                }
            }
            RK[p] = (int32_t)(mask << 8 | rank);
            BYR[p0 + rank] = (uint8_t)(p - p0);
        }
    }
    __syncthreads();
    for (int32_t i = warp; i < s_nw; i += nwarps) {
        const int32_t v = LST[n - 1 - i];
        place_comp_warp(R, OFF, v >> 6, v & 63, policy);
    }
    // the largest thread-tier components go to the last warp, which has the
    // fewest warp-tier components
    for (int32_t g = ((nwarps - 1 - warp) << 5) + (tid & 31); g < s_nt; g += nthr) {
        const int32_t v = LST[g];
        place_comp_thread(R, OFF, RK, BYR, v >> 6, v & 63, policy);
    }
    // components of more than kBWarpComp members: the whole CTA, one member at
    // a time in the breadth order (the per-step arrays, done with, are the
    // scratch: the order, then the gathered predecessors' offsets and ends)
    const int32_t nbig = min(s_nb, kBBigComps);
    for (int32_t k = 0; k < nbig; ++k) {
        __syncthreads();  // the previous component's scratch reads are done
        const int32_t p0 = s_big[k], c = size_from(p0);
        int32_t* ORDC = reinterpret_cast<int32_t*>(smem_raw + L.br);
        int64_t* PB = reinterpret_cast<int64_t*>(smem_raw + L.br + BCompLayout::align16b((size_t)c * 4));
        int64_t* PE = PB + c;
        for (int32_t i = tid; i < c; i += nthr) ORDC[i] = p0 + i;
        __syncthreads();
        block_sort_ids(ORDC, c, [&](int32_t x, int32_t y) { return b_before(R[x], R[y]); });
        const unsigned lt = (1u << (tid & 31)) - 1u;
        for (int32_t r = 0; r < c; ++r) {
            if (tid == 0) s_cnt = 0;
            __syncthreads();  // the previous member's offset is written, the counter reset
            const int32_t i = ORDC[r];
            const BRec me = R[i];
            for (int32_t x0 = warp * 32; x0 < r; x0 += nthr) {
                const int32_t x = x0 + (tid & 31);
                bool ov = false;
                int32_t j = 0;
                if (x < r) {
                    j = ORDC[x];
                    ov = R[j].a < me.f && me.a < R[j].f;
                }
                const unsigned m = __ballot_sync(0xffffffffu, ov);
                if (m == 0) continue;
                const int leader = __ffs(m) - 1;
                int32_t at = 0;
                if ((tid & 31) == leader) at = atomicAdd(&s_cnt, __popc(m));
                at = __shfl_sync(0xffffffffu, at, leader) + __popc(m & lt);
                if (ov) {
                    PB[at] = OFF[j];
                    PE[at] = OFF[j] + R[j].s;
                }
            }
            __syncthreads();  // the predecessors are gathered
            if (warp == 0) {
                const int64_t o = warp_gap_search(policy, me.s, PB, PE, s_cnt);
                if ((tid & 31) == 0) OFF[i] = o;
            }
        }
    }
    __syncthreads();
    int64_t mx = 0;
    for (int32_t p = tid; p < n; p += nthr) {
        const int64_t o = OFF[p];
        offsets[tv.lo + R[p].id] = o;
        mx = max(mx, o + R[p].s);
    }
    mx = block_max_i64(mx, red);
    if (tid == 0) {
        plan_peak[b] = mx;
        status[b] = MP_OK;
    }
}

bool breadth_comp_fits(const mp_batch& bt) {
    return BCompLayout(bt.max_tensors, bt.max_steps).total <= kSmemCeiling;
}

}  // namespace

size_t breadth_workspace_bytes(const mp_batch& bt) {
    if (bt.n_traces == 0 || breadth_fits_smem(bt)) return 0;
    return mul_sat((size_t)bt.n_traces, BreadthLayout(bt.max_tensors, bt.max_steps).total);
}

cudaError_t launch_breadth(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak, int32_t* status,
                           void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const bool comp = breadth_comp_fits(bt);
    if (comp) {
        const size_t cbytes = BCompLayout(bt.max_tensors, bt.max_steps).total;
        cudaError_t e = set_smem_limit((const void*)k_breadth_comp, cbytes);
        if (e != cudaSuccess) return e;
        k_breadth_comp<<<(unsigned)bt.n_traces, kBreadthThreads, cbytes, stream>>>(bt, policy, offsets, plan_peak,
                                                                                  status);
    }
    const size_t bytes = BreadthLayout(bt.max_tensors, bt.max_steps).total;
    if (breadth_fits_smem(bt)) {
        cudaError_t e = set_smem_limit((const void*)k_breadth<true>, bytes);
        if (e != cudaSuccess) return e;
        k_breadth<true><<<(unsigned)bt.n_traces, kBreadthThreads, bytes, stream>>>(bt, policy, offsets, plan_peak,
                                                                                   status, nullptr, 0, comp);
    } else {
        k_breadth<false><<<(unsigned)bt.n_traces, kBreadthThreads, 0, stream>>>(
            bt, policy, offsets, plan_peak, status, static_cast<unsigned char*>(workspace), bytes, comp);
    }
    return cudaGetLastError();
}

}  // namespace mp
