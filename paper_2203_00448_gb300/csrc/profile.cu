// profile.cu -- stage 1: live-bytes profile and its peak (lower bound on total_mem).
//
// profile[t] = sum of size_i over tensors with alloc_i <= t < free_i.  Its
// maximum bounds every feasible total_mem of Eq. 2.1 from below (the tensors
// live at one step must sit side by side in the slab).
//
// GPU form: one CTA of kProfileThreads per trace.  Each thread loads its
// first kProfCached tensors into registers before anything else (16-byte
// loads when the trace's slices are aligned).  The CTA first reduces the
// exact size sum; then it builds the difference array D (D[a] += s, D[f] -= s
// for f < T) with integer atomics -- order-independent, so exact -- and scans
// it in tiles of kProfileThreads * kProfItems steps, kProfItems consecutive
// steps per thread, writing the profile straight from registers.  Every
// partial sum of D lies between 0 and the size sum, so when that sum is below
// 2^32 the array holds 32-bit words (wrapping differences, exact partial
// sums) with plain 32-bit atomics and a 32-bit scan; otherwise each 64-bit
// add is done as 32-bit adds with an explicit carry, which shared memory
// executes far faster than 64-bit atomics.  In shared memory every
// kProfItems entries are followed by 16 bytes of padding, so that the
// threads' 16-byte reads of their runs fall in distinct banks.  D lives in
// shared memory when T fits, otherwise (64-bit words only) in the trace's own
// slice of the profile output (exactly T entries; the decrement at f = T is
// never needed), scanned in place.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int kProfItems = 8;   // profile steps per thread per tile
constexpr int kProfCached = 4;  // tensors per thread loaded into registers up front

// Position of step t in the difference array of W words: padded by 16 bytes
// after every kProfItems entries in shared memory.
template <bool kSmem, typename W>
__device__ __forceinline__ int32_t dpos(int32_t t) {
    return kSmem ? t + (int32_t)(16 / sizeof(W)) * (t / kProfItems) : t;
}

// Shared memory of one trace: the padded 64-bit array (the 32-bit one is smaller).
__host__ __device__ constexpr size_t padded_steps(size_t T) {
    return T + 2 * ((T + kProfItems - 1) / kProfItems);
}

__device__ __forceinline__ void d_add(uint32_t* d, int64_t v) { atomicAdd(d, (uint32_t)v); }
__device__ __forceinline__ void d_add(int64_t* d, int64_t v) { atomic_add_u64_split(d, (uint64_t)v); }

// Adds one (valid) tensor to the difference array.
template <bool kSmem, typename W>
__device__ __forceinline__ void add_tensor(W* D, int32_t T, int32_t a, int32_t f, int64_t s) {
    d_add(D + dpos<kSmem, W>(a), s);
    if (f < T) d_add(D + dpos<kSmem, W>(f), -s);
}

// The difference array's scan and the profile write; returns the block's
// largest profile value (every thread).
template <bool kSmem, typename W>
__device__ __forceinline__ int64_t scan_and_write(W* D, int64_t* out, int32_t T, int64_t* red,
                                                  unsigned long long* s_max) {
    const int32_t tid = (int32_t)threadIdx.x;
    const bool vec_d = (reinterpret_cast<uintptr_t>(D) & 15) == 0;
    const bool vec_out = (reinterpret_cast<uintptr_t>(out) & 15) == 0;
    constexpr int kVec = 16 / sizeof(W);  // words per 16-byte read
    W carry = 0, mx = 0;
    for (int32_t base = 0; base < T; base += (int32_t)blockDim.x * kProfItems) {
        const int32_t my = base + tid * kProfItems;
        W v[kProfItems];
        const W* run = D + dpos<kSmem, W>(my);
        if (vec_d && my + kProfItems <= T) {
#pragma unroll
            for (int k = 0; k < kProfItems; k += kVec) {
                if constexpr (sizeof(W) == 8) {
                    const longlong2 q = *reinterpret_cast<const longlong2*>(run + k);
                    v[k] = (W)q.x;
                    v[k + 1] = (W)q.y;
                } else {
                    const uint4 q = *reinterpret_cast<const uint4*>(run + k);
                    v[k] = q.x;
                    v[k + 1] = q.y;
                    v[k + 2] = q.z;
                    v[k + 3] = q.w;
                }
            }
        } else {
#pragma unroll
            for (int k = 0; k < kProfItems; ++k) v[k] = my + k < T ? run[k] : (W)0;
        }
#pragma unroll
        for (int k = 1; k < kProfItems; ++k) v[k] += v[k - 1];
        W tot;
        const W pre = block_excl_scan<W>(v[kProfItems - 1], reinterpret_cast<W*>(red), &tot) + carry;
        carry += tot;
#pragma unroll
        for (int k = 0; k < kProfItems; ++k) {
            v[k] += pre;
            mx = v[k] > mx ? v[k] : mx;
        }
        if (vec_out && my + kProfItems <= T) {
#pragma unroll
            for (int k = 0; k < kProfItems; k += 2)
                *reinterpret_cast<longlong2*>(out + my + k) = make_longlong2((int64_t)v[k], (int64_t)v[k + 1]);
        } else {
#pragma unroll
            for (int k = 0; k < kProfItems; ++k)
                if (my + k < T) out[my + k] = (int64_t)v[k];
        }
    }
    unsigned long long m;
    if constexpr (sizeof(W) == 8) {
        m = (unsigned long long)warp_max_i64(mx);
    } else {
        m = __reduce_max_sync(0xffffffffu, mx);
    }
    if ((threadIdx.x & 31) == 0 && m > 0) atomicMax(s_max, m);
    __syncthreads();
    return (int64_t)*s_max;
}

template <bool kSmem>
__global__ void __launch_bounds__(kProfileThreads, kSmem ? 10 : 1)
k_live_profile(mp_batch bt, int64_t* __restrict__ profile, int64_t* __restrict__ peak_lb,
               int32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[40];
    __shared__ unsigned long long s_max;
    __shared__ unsigned int s_sum[3];
    __shared__ int s_bad;
    const int32_t tid = (int32_t)threadIdx.x, nthr = (int32_t)blockDim.x;
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, true);
    if (tv.st != MP_OK) {
        if (tid == 0) status[b] = tv.st;
        return;
    }
    const int32_t T = tv.T, n = tv.n;
    const int32_t* __restrict__ A = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ F = bt.free_step + tv.lo;
    const int64_t* __restrict__ S = bt.size_bytes + tv.lo;
    const bool vec_in = ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(F) |
                          reinterpret_cast<uintptr_t>(S)) & 15) == 0;
    auto cidx = [&](int j) -> int32_t { return vec_in ? 4 * tid + j : tid + j * nthr; };
    int32_t ca[kProfCached], cf[kProfCached];
    int64_t cs[kProfCached];
    if (vec_in && 4 * tid + 3 < n) {
        const int4 a = __ldg(reinterpret_cast<const int4*>(A) + tid);
        const int4 f = __ldg(reinterpret_cast<const int4*>(F) + tid);
        const longlong2 s01 = __ldg(reinterpret_cast<const longlong2*>(S) + 2 * tid);
        const longlong2 s23 = __ldg(reinterpret_cast<const longlong2*>(S) + 2 * tid + 1);
        ca[0] = a.x, ca[1] = a.y, ca[2] = a.z, ca[3] = a.w;
        cf[0] = f.x, cf[1] = f.y, cf[2] = f.z, cf[3] = f.w;
        cs[0] = s01.x, cs[1] = s01.y, cs[2] = s23.x, cs[3] = s23.y;
    } else {
#pragma unroll
        for (int j = 0; j < kProfCached; ++j) {
            const int32_t k = cidx(j);
            ca[j] = cf[j] = 0;
            cs[j] = 0;
            if (k < n) {
                ca[j] = __ldg(A + k);
                cf[j] = __ldg(F + k);
                cs[j] = __ldg(S + k);
            }
        }
    }

    int64_t* out = profile + tv.plo;
    unsigned char* dmem = kSmem ? smem_raw : reinterpret_cast<unsigned char*>(out);
    // Zero the bytes of the 64-bit array (they cover the 32-bit one).
    {
        const int32_t dlen = kSmem ? (int32_t)padded_steps(T) : T;
        int64_t* D = reinterpret_cast<int64_t*>(dmem);
        if ((reinterpret_cast<uintptr_t>(D) & 15) == 0) {
            longlong2* D2 = reinterpret_cast<longlong2*>(D);
            for (int32_t t = tid; t < (dlen >> 1); t += nthr) D2[t] = make_longlong2(0, 0);
            if ((dlen & 1) && tid == 0) D[dlen - 1] = 0;
        } else {
            for (int32_t t = tid; t < dlen; t += nthr) D[t] = 0;
        }
    }
    if (tid == 0) {
        s_max = 0;
        s_bad = 0;
        s_sum[0] = s_sum[1] = s_sum[2] = 0;
    }
    __syncthreads();

    // Validity and the exact size sum (three 21-bit limbs of the per-thread
    // sums saturated at 2^63; a warp reduction of each cannot wrap).
    bool ok = true;
    uint64_t sum = 0;
#pragma unroll
    for (int j = 0; j < kProfCached; ++j) {
        if (cidx(j) < n) {
            ok &= tensor_ok(ca[j], cf[j], cs[j], T);
            sum = sat_add(sum, (uint64_t)cs[j] & ~kSatCap);
        }
    }
    const int32_t nc = min(n, kProfCached * nthr);
    for (int32_t k = nc + tid; k < n; k += nthr) {
        const int64_t sk = __ldg(S + k);
        ok &= tensor_ok(__ldg(A + k), __ldg(F + k), sk, T);
        sum = sat_add(sum, (uint64_t)sk & ~kSatCap);
    }
    {
        const unsigned full = 0xffffffffu;
        const unsigned l0 = __reduce_add_sync(full, (unsigned)(sum & 0x1fffffu));
        const unsigned l1 = __reduce_add_sync(full, (unsigned)((sum >> 21) & 0x1fffffu));
        const unsigned l2 = __reduce_add_sync(full, (unsigned)(sum >> 42));
        const bool bad = !__all_sync(full, ok);
        if ((tid & 31) == 0) {
            if (l0 | l1 | l2) {
                atomicAdd(s_sum, l0);
                atomicAdd(s_sum + 1, l1);
                atomicAdd(s_sum + 2, l2);
            }
            if (bad) s_bad = 1;
        }
    }
    __syncthreads();
    const uint64_t l0 = s_sum[0], l1 = s_sum[1] + (l0 >> 21), l2 = s_sum[2] + (l1 >> 21);
    if (s_bad || l2 >= (1ull << 21)) {  // an invalid tensor, or sizes summing past INT64_MAX
        if (tid == 0) status[b] = s_bad ? MP_EINVAL : MP_EOVERFLOW;
        return;
    }
    const bool narrow = kSmem && l2 == 0 && (l1 >> 11) == 0;  // the size sum is below 2^32

    int64_t peak;
    if (narrow) {
        uint32_t* D = reinterpret_cast<uint32_t*>(dmem);
#pragma unroll
        for (int j = 0; j < kProfCached; ++j)
            if (cidx(j) < n) add_tensor<kSmem, uint32_t>(D, T, ca[j], cf[j], cs[j]);
        for (int32_t k = nc + tid; k < n; k += nthr) add_tensor<kSmem, uint32_t>(D, T, __ldg(A + k), __ldg(F + k), __ldg(S + k));
        __syncthreads();
        peak = scan_and_write<kSmem, uint32_t>(D, out, T, red, &s_max);
    } else {
        int64_t* D = reinterpret_cast<int64_t*>(dmem);
#pragma unroll
        for (int j = 0; j < kProfCached; ++j)
            if (cidx(j) < n) add_tensor<kSmem, int64_t>(D, T, ca[j], cf[j], cs[j]);
        for (int32_t k = nc + tid; k < n; k += nthr) add_tensor<kSmem, int64_t>(D, T, __ldg(A + k), __ldg(F + k), __ldg(S + k));
        __syncthreads();
        peak = scan_and_write<kSmem, int64_t>(D, out, T, red, &s_max);
    }
    if (tid == 0) {
        peak_lb[b] = peak;
        status[b] = MP_OK;
    }
}

}  // namespace

// Per-CTA dynamic shared memory: one padded difference array of max_steps.
size_t profile_smem_bytes(const mp_batch& bt) {
    return padded_steps(bt.max_steps) * sizeof(int64_t);
}

cudaError_t launch_live_profile(const mp_batch& bt, int64_t* profile, int64_t* peak_lb, int32_t* status,
                                cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const size_t smem = profile_smem_bytes(bt);
    dim3 grid((unsigned)bt.n_traces), block(kProfileThreads);
    if (smem <= kProfileSmemLimit) {
        cudaError_t e = set_smem_limit((const void*)k_live_profile<true>, smem);
        if (e != cudaSuccess) return e;
        k_live_profile<true><<<grid, block, smem, stream>>>(bt, profile, peak_lb, status);
    } else {
        k_live_profile<false><<<grid, block, 0, stream>>>(bt, profile, peak_lb, status);
    }
    return cudaGetLastError();
}

}  // namespace mp
