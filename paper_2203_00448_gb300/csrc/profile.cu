// profile.cu -- stage 1: live-bytes profile and its peak (lower bound on total_mem).
//
// profile[t] = sum of size_i over tensors with alloc_i <= t < free_i.  Its
// maximum bounds every feasible total_mem of Eq. 2.1 from below (the tensors
// live at one step must sit side by side in the slab).
//
// GPU form: one CTA per trace builds the difference array D (D[a] += s,
// D[f] -= s for f < T) with integer atomics -- order-independent, so exact --
// then scans it in place and takes the maximum.  D lives in shared memory when
// T fits, otherwise in the trace's own slice of the profile output, which
// has exactly T entries (the decrement at f = T is never needed).
#include "common.cuh"
#include "launch.h"

namespace mp {

template <bool kSmem>
__global__ void __launch_bounds__(kProfileThreads)
k_live_profile(mp_batch bt, int64_t* __restrict__ profile, int64_t* __restrict__ peak_lb,
               int32_t* __restrict__ status) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[64];
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, true);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t T = tv.T, n = tv.n;
    int64_t* out = profile + tv.plo;
    int64_t* D = kSmem ? reinterpret_cast<int64_t*>(smem_raw) : out;
    for (int t = threadIdx.x; t < T; t += blockDim.x) D[t] = 0;
    __syncthreads();

    const int32_t* __restrict__ A = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ F = bt.free_step + tv.lo;
    const int64_t* __restrict__ S = bt.size_bytes + tv.lo;
    bool bad = false;
    uint64_t sum = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(A + k), f = __ldg(F + k);
        const int64_t s = __ldg(S + k);
        if (!tensor_ok(a, f, s, T)) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        atomicAdd(reinterpret_cast<unsigned long long*>(D + a), (unsigned long long)s);
        if (f < T) atomicAdd(reinterpret_cast<unsigned long long*>(D + f), (unsigned long long)(-s));
    }
    bad = __syncthreads_or(bad);
    sum = block_sat_sum(sum, reinterpret_cast<uint64_t*>(red));
    if (bad || sum > (uint64_t)INT64_MAX) {
        if (threadIdx.x == 0) status[b] = bad ? MP_EINVAL : MP_EOVERFLOW;
        return;
    }
    const int64_t mx = block_incl_scan_max_i64<4>(D, T, 0, red);
    if (kSmem) {
        for (int t = threadIdx.x; t < T; t += blockDim.x) out[t] = D[t];
    }
    if (threadIdx.x == 0) {
        peak_lb[b] = mx;
        status[b] = MP_OK;
    }
}

size_t profile_smem_bytes(const mp_batch& bt) { return (size_t)bt.max_steps * sizeof(int64_t); }

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
