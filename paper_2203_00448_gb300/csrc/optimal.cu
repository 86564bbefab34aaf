// optimal.cu -- the exact optimum of Eq. 2.1 for traces of at most kOptMax
// tensors, by exhaustive search.  Every order of the tensors is tried, each
// tensor placed in turn at its lowest feasible offset among the lifetime-
// overlapping tensors placed before it, and the smallest resulting total_mem
// is the optimum: taking the tensors of any optimal packing by ascending
// offset, each lands at or below its optimal offset, so some order reaches
// the optimum.  Among equally good orders the first in lexicographic order
// gives the reported offsets.  It measures how far greedy_by_size (Sec. 2.3)
// is from optimal, the comparison of Sec. 3.2's strategy study.
//
// GPU form: the n! orders of a trace are split into chunks of kOptChunk
// ranks; one CTA per (trace, chunk) and a thread per kOptPerThread
// consecutive ranks (unranked once, then advanced by next-permutation, which
// follows the same lexicographic order); each CTA keeps the minimum of
// (total_mem, rank).  A second kernel reduces the chunks of each trace and
// places its winning order again to write the offsets.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int kOptMax = 10;
constexpr int kOptPerThread = 32;
constexpr int64_t kOptChunk = (int64_t)kOptThreads * kOptPerThread;

__host__ __device__ constexpr int64_t factorial(int n) { return n <= 1 ? 1 : n * factorial(n - 1); }

__device__ __forceinline__ int nib(uint64_t x, int k) { return (int)((x >> (4 * k)) & 15u); }
__device__ __forceinline__ uint64_t set_nib(uint64_t x, int k, int v) {
    return (x & ~(15ull << (4 * k))) | ((uint64_t)v << (4 * k));
}

// The permutation of rank k (lexicographic, 0-based) of 0..n-1, 4 bits per slot.
__device__ uint64_t unrank(int64_t k, int n) {
    uint64_t avail = 0, perm = 0;  // the unused values, in increasing order
    for (int v = 0; v < n; ++v) avail = set_nib(avail, v, v);
    int left = n;
    for (int r = 0; r < n; ++r) {
        const int64_t f = factorial(n - 1 - r);
        const int d = (int)(k / f);
        k -= d * f;
        perm = set_nib(perm, r, nib(avail, d));
        for (int j = d; j < left - 1; ++j) avail = set_nib(avail, j, nib(avail, j + 1));
        --left;
    }
    return perm;
}

// The next permutation in lexicographic order; false after the last.
__device__ bool next_perm(uint64_t& perm, int n) {
    int k = n - 2;
    while (k >= 0 && nib(perm, k) >= nib(perm, k + 1)) --k;
    if (k < 0) return false;
    int l = n - 1;
    while (nib(perm, l) <= nib(perm, k)) --l;
    const int t = nib(perm, k);
    perm = set_nib(perm, k, nib(perm, l));
    perm = set_nib(perm, l, t);
    for (int x = k + 1, y = n - 1; x < y; ++x, --y) {
        const int u = nib(perm, x);
        perm = set_nib(perm, x, nib(perm, y));
        perm = set_nib(perm, y, u);
    }
    return true;
}

// One trace of at most kOptMax tensors: sizes and the lifetime-overlap mask
// of every tensor.
struct OptTrace {
    int64_t s[kOptMax];
    uint32_t ov[kOptMax];
};

// Places the tensors in the order perm, each at its lowest feasible offset
// (jumping past conflicting predecessors until none conflicts); returns the
// largest end, and the offsets (by tensor) when off is given.
__device__ int64_t place_order(const OptTrace& tr, int n, uint64_t perm, int64_t* off) {
    int64_t o_r[kOptMax], e_r[kOptMax];
    int id_r[kOptMax];
    int64_t peak = 0;
#pragma unroll
    for (int r = 0; r < kOptMax; ++r) {
        if (r >= n) break;
        const int i = nib(perm, r);
        id_r[r] = i;
        const int64_t s = tr.s[i];
        const uint32_t ov = tr.ov[i];
        int64_t o = 0;
        for (;;) {
            int64_t next = o;
#pragma unroll
            for (int q = 0; q < kOptMax; ++q)
                if (q < r && ((ov >> id_r[q]) & 1u) && o_r[q] < o + s && o < e_r[q] && e_r[q] > next) next = e_r[q];
            if (next == o) break;
            o = next;
        }
        o_r[r] = o;
        e_r[r] = o + s;
        peak = e_r[r] > peak ? e_r[r] : peak;
        if (off) off[i] = o;
    }
    return peak;
}

// Loads trace b into tr and checks it; MP_OK, or the trace's status (more
// than kOptMax tensors: MP_EINVAL).
__device__ int32_t load_opt_trace(const mp_batch& bt, int b, OptTrace& tr, int& n, int64_t& lo) {
    const TraceView tv = load_trace(bt, b, false);
    lo = tv.lo;
    n = 0;
    if (tv.st != MP_OK) return tv.st;
    if (tv.n > kOptMax) return MP_EINVAL;
    n = tv.n;
    int32_t a[kOptMax], f[kOptMax];
    uint64_t sum = 0;
    bool bad = false;
    for (int i = 0; i < n; ++i) {
        a[i] = __ldg(bt.alloc_step + lo + i);
        f[i] = __ldg(bt.free_step + lo + i);
        tr.s[i] = __ldg(bt.size_bytes + lo + i);
        if (!tensor_ok(a[i], f[i], tr.s[i], tv.T)) bad = true;
        else sum = sat_add(sum, (uint64_t)tr.s[i]);
    }
    if (bad) return MP_EINVAL;
    if (sum > (uint64_t)INT64_MAX) return MP_EOVERFLOW;
    for (int i = 0; i < n; ++i) {
        uint32_t m = 0;
        for (int j = 0; j < n; ++j)
            if (j != i && a[i] < f[j] && a[j] < f[i]) m |= 1u << j;
        tr.ov[i] = m;
    }
    return MP_OK;
}

// (total_mem, rank) minimum of chunk c of trace b into best[b * chunks + c].
__global__ void __launch_bounds__(kOptThreads)
k_opt_search(mp_batch bt, int32_t chunks, longlong2* __restrict__ best) {
    __shared__ OptTrace tr;
    __shared__ int s_n, s_st;
    __shared__ int64_t red_k[kOptThreads / 32], red_v[kOptThreads / 32];
    const int b = blockIdx.x / chunks, c = blockIdx.x % chunks;
    if (threadIdx.x == 0) {
        int n;
        int64_t lo;
        s_st = load_opt_trace(bt, b, tr, n, lo);
        s_n = n;
    }
    __syncthreads();
    const int n = s_n;
    int64_t bv = INT64_MAX, bk = INT64_MAX;
    if (s_st == MP_OK && n > 0) {
        const int64_t total = factorial(n);
        const int64_t k0 = (int64_t)c * kOptChunk + (int64_t)threadIdx.x * kOptPerThread;
        if (k0 < total) {
            uint64_t perm = unrank(k0, n);
            const int64_t k1 = min(total, k0 + kOptPerThread);
            for (int64_t k = k0; k < k1; ++k) {
                const int64_t v = place_order(tr, n, perm, nullptr);
                if (v < bv) {  // ranks increase: the first rank keeps a tie
                    bv = v;
                    bk = k;
                }
                next_perm(perm, n);
            }
        }
    }
    // minimum over the block by (value, rank)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t v2 = __shfl_xor_sync(0xffffffffu, bv, o), k2 = __shfl_xor_sync(0xffffffffu, bk, o);
        if (v2 < bv || (v2 == bv && k2 < bk)) {
            bv = v2;
            bk = k2;
        }
    }
    if ((threadIdx.x & 31) == 0) {
        red_v[threadIdx.x >> 5] = bv;
        red_k[threadIdx.x >> 5] = bk;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < kOptThreads / 32; ++w)
            if (red_v[w] < bv || (red_v[w] == bv && red_k[w] < bk)) {
                bv = red_v[w];
                bk = red_k[w];
            }
        best[blockIdx.x] = make_longlong2(bv, bk);
    }
}

// One warp per trace: the best of its chunks, placed again for the offsets.
__global__ void __launch_bounds__(kOptThreads)
k_opt_finish(mp_batch bt, int32_t chunks, const longlong2* __restrict__ best, int64_t* __restrict__ offsets,
             int64_t* __restrict__ opt_peak, int32_t* __restrict__ status) {
    const int lane = threadIdx.x & 31;
    const int b = blockIdx.x * (kOptThreads / 32) + (threadIdx.x >> 5);
    if (b >= bt.n_traces) return;
    int64_t bv = INT64_MAX, bk = INT64_MAX;
    for (int c = lane; c < chunks; c += 32) {
        const longlong2 r = best[(size_t)b * chunks + c];
        if (r.x < bv || (r.x == bv && r.y < bk)) {
            bv = r.x;
            bk = r.y;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t v2 = __shfl_xor_sync(0xffffffffu, bv, o), k2 = __shfl_xor_sync(0xffffffffu, bk, o);
        if (v2 < bv || (v2 == bv && k2 < bk)) {
            bv = v2;
            bk = k2;
        }
    }
    if (lane != 0) return;
    OptTrace tr;
    int n;
    int64_t lo;
    const int32_t st = load_opt_trace(bt, b, tr, n, lo);
    status[b] = st;
    if (st != MP_OK) {
        opt_peak[b] = 0;
        return;
    }
    if (n == 0) {
        opt_peak[b] = 0;
        return;
    }
    int64_t off[kOptMax];
    const int64_t v = place_order(tr, n, unrank(bk, n), off);
    for (int i = 0; i < n; ++i) offsets[lo + i] = off[i];
    opt_peak[b] = v;
}

int32_t opt_chunks(const mp_batch& bt) {
    const int nmax = bt.max_tensors < kOptMax ? (bt.max_tensors > 0 ? bt.max_tensors : 1) : kOptMax;
    return (int32_t)((factorial(nmax) + kOptChunk - 1) / kOptChunk);
}

}  // namespace

size_t optimal_workspace_bytes(const mp_batch& bt) {
    if (bt.n_traces == 0) return 0;
    const size_t need = mul_sat(mul_sat((size_t)bt.n_traces, (size_t)opt_chunks(bt)), sizeof(longlong2));
    return need > SIZE_MAX - kAlign ? SIZE_MAX : align_up(need);
}

cudaError_t launch_optimal(const mp_batch& bt, int64_t* offsets, int64_t* opt_peak, int32_t* status, void* workspace,
                           cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const int32_t chunks = opt_chunks(bt);
    longlong2* best = static_cast<longlong2*>(workspace);
    k_opt_search<<<(unsigned)((int64_t)bt.n_traces * chunks), kOptThreads, 0, stream>>>(bt, chunks, best);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int per_cta = kOptThreads / 32;
    k_opt_finish<<<(unsigned)((bt.n_traces + per_cta - 1) / per_cta), kOptThreads, 0, stream>>>(
        bt, chunks, best, offsets, opt_peak, status);
    return cudaGetLastError();
}

}  // namespace mp
