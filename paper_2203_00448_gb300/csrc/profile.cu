// profile.cu -- stage 1: live-bytes profile and its peak (lower bound on total_mem).
//
// profile[t] = sum of size_i over tensors with alloc_i <= t < free_i.  Its
// maximum bounds every feasible total_mem of Eq. 2.1 from below (the tensors
// live at one step must sit side by side in the slab).
//
// GPU form: one warp per trace.  The warp builds the difference array D
// (D[a] += s, D[f] -= s for f < T) with integer atomics -- order-independent,
// so exact; each 64-bit add is done as 32-bit adds with an explicit carry,
// which shared memory executes far faster than 64-bit atomics -- then scans
// it, kScanItems consecutive steps per lane, and writes the profile straight
// from registers.  In shared memory every kScanItems entries are followed by
// 16 bytes of padding, so the lanes' 16-byte reads of their runs fall in
// distinct banks.  D lives in the warp's slice of shared
// memory when T fits, otherwise in the trace's own slice of the profile output
// (which has exactly T entries; the decrement at f = T is never needed).
// Warps are independent (no CTA barrier), so an SM keeps dozens of traces in
// flight and the DRAM round trips of one trace overlap the work of others.
// Tensor arrays are read with 16-byte loads and the profile written with
// 16-byte stores whenever the trace's slices are 16-byte aligned.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

constexpr int kScanItems = kProfRun;  // profile steps per lane per tile

// Position of step t in the (padded, when kSmem) difference array.
template <bool kSmem>
__device__ __forceinline__ int64_t dpos(int64_t t) {
    return kSmem ? prof_pos(t) : t;
}

__host__ __device__ constexpr size_t padded_steps(size_t T) { return prof_padded(T); }

// Adds one tensor to the difference array; returns false if it is invalid.
template <bool kSmem>
__device__ __forceinline__ bool add_tensor(int64_t* D, int32_t T, int32_t a, int32_t f, int64_t s, uint64_t& sum) {
    if (!tensor_ok(a, f, s, T)) return false;
    sum = sat_add(sum, (uint64_t)s);
    atomic_add_u64_split(D + dpos<kSmem>(a), (uint64_t)s);
    if (f < T) atomic_add_u64_split(D + dpos<kSmem>(f), (uint64_t)(-s));
    return true;
}

// Warp-level: true if the saturated per-lane size sums total more than INT64_MAX.
__device__ __forceinline__ bool warp_sum_overflows(uint64_t sum) {
    unsigned long long h = sum >> 32, l = sum & 0xffffffffull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        h += __shfl_xor_sync(0xffffffffu, h, o);
        l += __shfl_xor_sync(0xffffffffu, l, o);
    }
    return h + (l >> 32) >= (1ull << 31);
}

template <bool kSmem>
__global__ void __launch_bounds__(kProfileThreads)
k_live_profile(mp_batch bt, int64_t* __restrict__ profile, int64_t* __restrict__ peak_lb,
               int32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int b = blockIdx.x * (kProfileThreads / 32) + warp;
    if (b >= bt.n_traces) return;
    const TraceView tv = load_trace(bt, b, true);
    if (tv.st != MP_OK) {
        if (lane == 0) status[b] = tv.st;
        return;
    }
    const int32_t T = tv.T, n = tv.n;
    int64_t* out = profile + tv.plo;
    int64_t* D = kSmem ? reinterpret_cast<int64_t*>(smem_raw) + (size_t)warp * padded_steps(bt.max_steps) : out;
    const int64_t dlen = kSmem ? (int64_t)padded_steps(T) : T;
    const bool vec_d = (reinterpret_cast<uintptr_t>(D) & 15) == 0;
    if (vec_d) {
        longlong2* D2 = reinterpret_cast<longlong2*>(D);
        for (int t = lane; t < (dlen >> 1); t += 32) D2[t] = make_longlong2(0, 0);
        if ((dlen & 1) && lane == 0) D[dlen - 1] = 0;
    } else {
        for (int t = lane; t < dlen; t += 32) D[t] = 0;
    }
    __syncwarp();

    const int32_t* __restrict__ A = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ F = bt.free_step + tv.lo;
    const int64_t* __restrict__ S = bt.size_bytes + tv.lo;
    bool ok = true;
    uint64_t sum = 0;
    int k0 = 0;
    const bool vec_in = ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(F) |
                          reinterpret_cast<uintptr_t>(S)) & 15) == 0;
    if (vec_in) {  // four tensors per 16-byte load
        const int n4 = n >> 2;
        const int4* A4 = reinterpret_cast<const int4*>(A);
        const int4* F4 = reinterpret_cast<const int4*>(F);
        const longlong2* S2 = reinterpret_cast<const longlong2*>(S);
#pragma unroll 2
        for (int q = lane; q < n4; q += 32) {
            const int4 a = __ldg(A4 + q), f = __ldg(F4 + q);
            const longlong2 s01 = __ldg(S2 + 2 * q), s23 = __ldg(S2 + 2 * q + 1);
            ok &= add_tensor<kSmem>(D, T, a.x, f.x, s01.x, sum);
            ok &= add_tensor<kSmem>(D, T, a.y, f.y, s01.y, sum);
            ok &= add_tensor<kSmem>(D, T, a.z, f.z, s23.x, sum);
            ok &= add_tensor<kSmem>(D, T, a.w, f.w, s23.y, sum);
        }
        k0 = n4 << 2;
    }
    for (int k = k0 + lane; k < n; k += 32) ok &= add_tensor<kSmem>(D, T, __ldg(A + k), __ldg(F + k), __ldg(S + k), sum);
    const bool bad = !__all_sync(0xffffffffu, ok);
    const bool ovf = warp_sum_overflows(sum);
    if (bad || ovf) {
        if (lane == 0) status[b] = bad ? MP_EINVAL : MP_EOVERFLOW;
        return;
    }
    __syncwarp();

    // Inclusive scan: kScanItems consecutive steps per lane, tiles of 32 lanes.
    const bool vec_out = (reinterpret_cast<uintptr_t>(out) & 15) == 0;
    int64_t carry = 0, mx = 0;
    for (int64_t base = 0; base < T; base += 32 * kScanItems) {
        const int64_t my = base + (int64_t)lane * kScanItems;
        int64_t v[kScanItems];
        const int64_t* run = D + dpos<kSmem>(my);
        if (vec_d && my + kScanItems <= T) {
#pragma unroll
            for (int k = 0; k < kScanItems; k += 2) {
                const longlong2 p = *reinterpret_cast<const longlong2*>(run + k);
                v[k] = p.x;
                v[k + 1] = p.y;
            }
        } else {
#pragma unroll
            for (int k = 0; k < kScanItems; ++k) v[k] = my + k < T ? run[k] : 0;
        }
#pragma unroll
        for (int k = 1; k < kScanItems; ++k) v[k] += v[k - 1];
        const int64_t incl = warp_incl_scan(v[kScanItems - 1]);
        const int64_t pre = incl - v[kScanItems - 1] + carry;
        carry += __shfl_sync(0xffffffffu, incl, 31);
#pragma unroll
        for (int k = 0; k < kScanItems; ++k) {
            v[k] += pre;
            mx = v[k] > mx ? v[k] : mx;
        }
        if (vec_out && my + kScanItems <= T) {
#pragma unroll
            for (int k = 0; k < kScanItems; k += 2)
                *reinterpret_cast<longlong2*>(out + my + k) = make_longlong2(v[k], v[k + 1]);
        } else {
#pragma unroll
            for (int k = 0; k < kScanItems; ++k)
                if (my + k < T) out[my + k] = v[k];
        }
    }
    mx = warp_max_i64(mx);
    if (lane == 0) {
        peak_lb[b] = mx;
        status[b] = MP_OK;
    }
}

}  // namespace

// Per-CTA dynamic shared memory: one difference array of max_steps per warp.
size_t profile_smem_bytes(const mp_batch& bt) {
    return (size_t)(kProfileThreads / 32) * padded_steps(bt.max_steps) * sizeof(int64_t);
}

cudaError_t launch_live_profile(const mp_batch& bt, int64_t* profile, int64_t* peak_lb, int32_t* status,
                                cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const size_t smem = profile_smem_bytes(bt);
    const int per_cta = kProfileThreads / 32;
    dim3 grid((unsigned)((bt.n_traces + per_cta - 1) / per_cta)), block(kProfileThreads);
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
