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
// GPU form: one CTA per trace.  The breadths (two integer atomics per
// tensor, order-independent), each tensor's wider operator, an in-place
// odd-even merge sort of the ids by that order, then placement tensor by
// tensor: all warps gather the placed tensors whose lifetimes overlap the
// next one (one shared counter update per warp) and warp 0 runs the gap
// search with warp reductions.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

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
          int32_t* __restrict__ status, unsigned char* __restrict__ ws, size_t ws_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ int32_t s_cnt, s_bad;
    __shared__ unsigned long long s_hi, s_lo;
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned lt = (1u << lane) - 1u;
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

}  // namespace

size_t breadth_workspace_bytes(const mp_batch& bt) {
    if (bt.n_traces == 0 || breadth_fits_smem(bt)) return 0;
    return mul_sat((size_t)bt.n_traces, BreadthLayout(bt.max_tensors, bt.max_steps).total);
}

cudaError_t launch_breadth(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak, int32_t* status,
                           void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const size_t bytes = BreadthLayout(bt.max_tensors, bt.max_steps).total;
    if (breadth_fits_smem(bt)) {
        cudaError_t e = set_smem_limit((const void*)k_breadth<true>, bytes);
        if (e != cudaSuccess) return e;
        k_breadth<true><<<(unsigned)bt.n_traces, kBreadthThreads, bytes, stream>>>(bt, policy, offsets, plan_peak,
                                                                                   status, nullptr, 0);
    } else {
        k_breadth<false><<<(unsigned)bt.n_traces, kBreadthThreads, 0, stream>>>(
            bt, policy, offsets, plan_peak, status, static_cast<unsigned char*>(workspace), bytes);
    }
    return cudaGetLastError();
}

}  // namespace mp
