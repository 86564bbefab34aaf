// common.cuh -- device helpers shared by the memory-planning kernels (sm_103a).
//
// Trace-level argument checks, saturating size sums and block-wide integer
// scans/reductions.  Everything here is integer arithmetic, so every kernel
// built on it is deterministic and bit-exact regardless of launch shape.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "memplan.h"

namespace mp {

constexpr int kWarp = 32;
constexpr uint64_t kSatCap = 0x8000000000000000ull;  // INT64_MAX + 1

// Per-trace view of the CSR metadata, with the checks every stage applies.
struct TraceView {
    int64_t lo;    // first tensor (global index)
    int32_t n;     // tensors in the trace
    int32_t T;     // op steps
    int64_t plo;   // first profile entry (mp_live_profile only)
    int32_t st;    // MP_OK or MP_EINVAL
};

__device__ __forceinline__ TraceView load_trace(const mp_batch& bt, int b, bool need_profile) {
    TraceView v;
    int64_t lo = __ldg(bt.trace_ptr + b), hi = __ldg(bt.trace_ptr + b + 1);
    int32_t T = __ldg(bt.steps + b);
    v.st = MP_OK;
    v.lo = lo;
    v.T = T;
    v.n = 0;
    v.plo = 0;
    if (lo < 0 || hi < lo || hi > bt.n_tensors || hi - lo > (int64_t)bt.max_tensors || T < 0 ||
        T > bt.max_steps) {
        v.st = MP_EINVAL;
        return v;
    }
    v.n = (int32_t)(hi - lo);
    if (need_profile) {
        int64_t plo = __ldg(bt.profile_ptr + b), phi = __ldg(bt.profile_ptr + b + 1);
        if (plo < 0 || phi - plo != (int64_t)T || phi > bt.n_steps) v.st = MP_EINVAL;
        v.plo = plo;
    }
    return v;
}

// One tensor's own validity: 0 <= a < f <= T and s >= 1.
__device__ __forceinline__ bool tensor_ok(int32_t a, int32_t f, int64_t s, int32_t T) {
    return a >= 0 && f > a && f <= T && s > 0;
}

// x + y saturated at 2^63, for x, y <= 2^63 (never wraps a uint64).
__device__ __forceinline__ uint64_t sat_add(uint64_t x, uint64_t y) {
    uint64_t r = x + y;
    return (r < x || r > kSatCap) ? kSatCap : r;
}

// Atomic 64-bit add built from 32-bit shared-memory atomics (64-bit shared
// atomics are several times slower): add the low word, take its carry from
// the value it replaced, and add high word + carry only when that is non-zero.
// Every 64-bit add is split exactly, so once all adds have completed the word
// holds the exact sum modulo 2^64; intermediate states are not meaningful.
__device__ __forceinline__ void atomic_add_u64_split(int64_t* word, uint64_t v) {
    unsigned int* w = reinterpret_cast<unsigned int*>(word);  // little-endian: w[0] low, w[1] high
    const unsigned int lo = (unsigned int)v, hi = (unsigned int)(v >> 32);
    const unsigned int old = atomicAdd(w, lo);
    const unsigned int h = hi + ((unsigned int)(old + lo) < old ? 1u : 0u);
    if (h) atomicAdd(w + 1, h);
}

// Difference arrays of the live profile are scanned kProfRun consecutive steps
// per lane; in shared memory each run is followed by kProfPad int64 of padding
// so that the lanes' 16-byte reads of their runs fall in distinct banks.
constexpr int kProfRun = 16;
constexpr int kProfPad = 2;
__host__ __device__ constexpr int64_t prof_pos(int64_t t) { return t + kProfPad * (t / kProfRun); }
__host__ __device__ constexpr size_t prof_padded(size_t T) {
    return T + kProfPad * ((T + kProfRun - 1) / kProfRun);
}

// ------------------------------------------------------------ warp level

__device__ __forceinline__ uint64_t warp_sat_sum(uint64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = sat_add(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ int64_t warp_max_i64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        int64_t w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

__device__ __forceinline__ int64_t warp_min_i64(int64_t v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        int64_t w = __shfl_xor_sync(0xffffffffu, v, o);
        v = w < v ? w : v;
    }
    return v;
}

// Lexicographic minimum of (key, val) pairs over the warp.
__device__ __forceinline__ void warp_min_pair(int64_t& key, int64_t& val) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        int64_t k2 = __shfl_xor_sync(0xffffffffu, key, o);
        int64_t v2 = __shfl_xor_sync(0xffffffffu, val, o);
        if (k2 < key || (k2 == key && v2 < val)) {
            key = k2;
            val = v2;
        }
    }
}

template <typename V>
__device__ __forceinline__ V warp_incl_scan(V v) {
    const int lane = threadIdx.x & (kWarp - 1);
#pragma unroll
    for (int o = 1; o < kWarp; o <<= 1) {
        V w = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += w;
    }
    return v;
}

// Adds a per-thread size sum (each <= 2^63) into two shared 64-bit counters as
// exact 32-bit halves: one warp-level reduction, then one atomic pair per warp.
// The block total exceeds INT64_MAX iff hi + (lo >> 32) >= 2^31 afterwards.
__device__ __forceinline__ void block_add_size_sum(uint64_t sum, unsigned long long* hi,
                                                   unsigned long long* lo) {
    unsigned long long h = sum >> 32, l = sum & 0xffffffffull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        h += __shfl_xor_sync(0xffffffffu, h, o);
        l += __shfl_xor_sync(0xffffffffu, l, o);
    }
    if ((threadIdx.x & 31) == 0 && (h | l)) {
        atomicAdd(hi, h);
        atomicAdd(lo, l);
    }
}

__device__ __forceinline__ bool size_sum_overflows(unsigned long long hi, unsigned long long lo) {
    return hi + (lo >> 32) >= (1ull << 31);
}

// ------------------------------------------------------------ block level
// All block helpers must be called by every thread of the block; `red` is a
// __shared__ scratch of at least 32 elements of the reduced type.  They end
// with a barrier, so `red` may be reused right after.

__device__ __forceinline__ uint64_t block_sat_sum(uint64_t v, uint64_t* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    v = warp_sat_sum(v);
    if (lane == 0) red[w] = v;
    __syncthreads();
    uint64_t r = 0;
    for (int k = 0; k < nw; ++k) r = sat_add(r, red[k]);
    __syncthreads();
    return r;
}

__device__ __forceinline__ int64_t block_max_i64(int64_t v, int64_t* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    v = warp_max_i64(v);
    if (lane == 0) red[w] = v;
    __syncthreads();
    int64_t r = red[0];
    for (int k = 1; k < nw; ++k) r = red[k] > r ? red[k] : r;
    __syncthreads();
    return r;
}

__device__ __forceinline__ int64_t block_min_i64(int64_t v, int64_t* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    v = warp_min_i64(v);
    if (lane == 0) red[w] = v;
    __syncthreads();
    int64_t r = red[0];
    for (int k = 1; k < nw; ++k) r = red[k] < r ? red[k] : r;
    __syncthreads();
    return r;
}

// Lexicographic min of (key, val); red needs 64 int64 slots.
__device__ __forceinline__ void block_min_pair(int64_t& key, int64_t& val, int64_t* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    warp_min_pair(key, val);
    if (lane == 0) {
        red[w] = key;
        red[32 + w] = val;
    }
    __syncthreads();
    int64_t k = red[0], v = red[32];
    for (int q = 1; q < nw; ++q)
        if (red[q] < k || (red[q] == k && red[32 + q] < v)) {
            k = red[q];
            v = red[32 + q];
        }
    __syncthreads();
    key = k;
    val = v;
}

// Exclusive scan of per-thread values over the block; returns this thread's
// prefix and writes the block total to *total.
template <typename V>
__device__ __forceinline__ V block_excl_scan(V v, V* red, V* total) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
    V incl = warp_incl_scan(v);
    if (lane == 31) red[w] = incl;
    __syncthreads();
    if (w == 0) {
        V x = lane < nw ? red[lane] : V(0);
        V xs = warp_incl_scan(x);
        if (lane < nw) red[lane] = xs - x;  // exclusive prefix of warp totals
        if (lane == nw - 1) red[32] = xs;
    }
    __syncthreads();
    V r = red[w] + incl - v;
    *total = red[32];
    __syncthreads();
    return r;
}

// In-place exclusive scan of x[0..len) (any memory space) by the whole block,
// in tiles of blockDim * ITEMS consecutive elements; returns the total.
// red: >= 33 slots.
template <typename V, int ITEMS>
__device__ V block_excl_scan_array(V* x, int64_t len, V* red) {
    V carry = 0;
    const int64_t tile = (int64_t)blockDim.x * ITEMS;
    for (int64_t base = 0; base < len; base += tile) {
        const int64_t my = base + (int64_t)threadIdx.x * ITEMS;
        V loc[ITEMS];
        V sum = 0;
#pragma unroll
        for (int k = 0; k < ITEMS; ++k) {
            loc[k] = (my + k < len) ? x[my + k] : V(0);
            sum += loc[k];
        }
        V tot;
        V pre = block_excl_scan<V>(sum, red, &tot) + carry;
#pragma unroll
        for (int k = 0; k < ITEMS; ++k) {
            if (my + k < len) x[my + k] = pre;
            pre += loc[k];
        }
        carry += tot;
        __syncthreads();
    }
    return carry;
}

// In-place inclusive scan of x[0..len); returns the block-wide maximum of the
// scanned values (or `init_max` if larger / len == 0).
template <int ITEMS>
__device__ int64_t block_incl_scan_max_i64(int64_t* x, int64_t len, int64_t init_max, int64_t* red) {
    int64_t carry = 0, mx = init_max;
    const int64_t tile = (int64_t)blockDim.x * ITEMS;
    for (int64_t base = 0; base < len; base += tile) {
        const int64_t my = base + (int64_t)threadIdx.x * ITEMS;
        int64_t loc[ITEMS];
        int64_t sum = 0;
#pragma unroll
        for (int k = 0; k < ITEMS; ++k) {
            loc[k] = (my + k < len) ? x[my + k] : 0;
            sum += loc[k];
        }
        int64_t tot;
        int64_t pre = block_excl_scan<int64_t>(sum, red, &tot) + carry;
#pragma unroll
        for (int k = 0; k < ITEMS; ++k) {
            pre += loc[k];
            if (my + k < len) {
                x[my + k] = pre;
                mx = pre > mx ? pre : mx;
            }
        }
        carry += tot;
        __syncthreads();
    }
    return block_max_i64(mx, red);
}

}  // namespace mp
