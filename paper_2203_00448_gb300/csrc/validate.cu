// validate.cu -- stage 3: pairwise plan validation (Eq. 2.1's ordering
// constraints), and the plan peak (Eq. 2.1's total_mem).
//
// A plan is valid iff no two tensors with overlapping lifetimes have
// intersecting address ranges.  Enumerating only the lifetime-overlapping
// pairs: sort the tensors of a trace by alloc step (counting sort over the T
// steps); for a tensor i at sorted position p, the tensors j after it with
// alloc_j < free_i are exactly its overlapping partners that start no earlier
// (alloc_i <= alloc_j < free_i implies overlap), so each overlapping pair is
// visited once, from its earlier-starting member.  The work is
// O(N + T + overlapping pairs) per trace instead of N^2 / 2, while the
// verdict still certifies all N (N - 1) / 2 pairs.  The reported conflict is
// the minimum of the packed (min id, max id) over all violating pairs, i.e.
// the lexicographically smallest, independent of visiting order.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

struct ValidateLayout {
    size_t off, end, f, bya, bend, total;
    __host__ __device__ ValidateLayout(int64_t n, int64_t T) {
        off = 0;
        end = off + align_up((size_t)n * 8);
        f = end + align_up((size_t)n * 8);
        bya = f + align_up((size_t)n * 4);
        bend = bya + align_up((size_t)n * 4);
        total = bend + align_up((size_t)T * 4);
    }
};

template <bool kSmem>
__global__ void __launch_bounds__(kValidateThreads)
k_validate(mp_batch bt, const int64_t* __restrict__ offsets, int32_t* __restrict__ verdict,
           int32_t* __restrict__ conflict, int32_t* __restrict__ status, unsigned char* __restrict__ ws,
           size_t ws_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[64];
    __shared__ unsigned long long s_key;
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const ValidateLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * ws_stride;
    int64_t* OFF = reinterpret_cast<int64_t*>(base + L.off);
    int64_t* END = reinterpret_cast<int64_t*>(base + L.end);
    int32_t* F = reinterpret_cast<int32_t*>(base + L.f);
    int32_t* BYA = reinterpret_cast<int32_t*>(base + L.bya);
    int32_t* BEND = reinterpret_cast<int32_t*>(base + L.bend);

    for (int t = threadIdx.x; t < T; t += blockDim.x) BEND[t] = 0;
    if (threadIdx.x == 0) s_key = ~0ull;
    __syncthreads();

    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    const int64_t* __restrict__ Og = offsets + tv.lo;
    bool bad = false, ovf = false;
    uint64_t sum = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t s = __ldg(Sg + k), o = __ldg(Og + k);
        if (!tensor_ok(a, f, s, T) || o < 0) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        if (o > INT64_MAX - s) {
            ovf = true;
            continue;
        }
        OFF[k] = o;
        END[k] = o + s;
        F[k] = f;
        atomicAdd(BEND + a, 1);
    }
    bad = __syncthreads_or(bad);
    ovf = __syncthreads_or(ovf);
    sum = block_sat_sum(sum, reinterpret_cast<uint64_t*>(red));
    if (bad || ovf || sum > (uint64_t)INT64_MAX) {
        if (threadIdx.x == 0) {
            status[b] = bad ? MP_EINVAL : MP_EOVERFLOW;
            verdict[b] = 0;
            if (conflict) conflict[2 * b] = conflict[2 * b + 1] = -1;
        }
        return;
    }
    // Counting sort by alloc step: bucket starts, then scatter; afterwards
    // BEND[t] is the end of bucket t (tensors with alloc <= t).
    block_excl_scan_array<int32_t, 4>(BEND, T, reinterpret_cast<int32_t*>(red));
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k);
        BYA[atomicAdd(BEND + a, 1)] = k;
    }
    __syncthreads();

    for (int p = threadIdx.x; p < n; p += blockDim.x) {
        const int32_t i = BYA[p];
        const int32_t stop = BEND[F[i] - 1];
        const int64_t oi = OFF[i], ei = END[i];
        for (int q = p + 1; q < stop; ++q) {
            const int32_t j = BYA[q];
            if (oi < END[j] && OFF[j] < ei) {
                const uint32_t lo = (uint32_t)(i < j ? i : j), hi = (uint32_t)(i < j ? j : i);
                atomicMin(&s_key, ((unsigned long long)lo << 32) | hi);
            }
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned long long key = s_key;
        const bool ok = key == ~0ull;
        verdict[b] = ok ? 1 : 0;
        if (conflict) {
            conflict[2 * b] = ok ? -1 : (int32_t)(key >> 32);
            conflict[2 * b + 1] = ok ? -1 : (int32_t)(key & 0xffffffffu);
        }
        status[b] = MP_OK;
    }
}

__global__ void __launch_bounds__(kPeakThreads)
k_peak(mp_batch bt, const int64_t* __restrict__ offsets, int64_t* __restrict__ plan_peak,
       int32_t* __restrict__ status) {
    __shared__ int64_t red[64];
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    bool bad = false, ovf = false;
    uint64_t sum = 0;
    int64_t mx = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(bt.alloc_step + tv.lo + k), f = __ldg(bt.free_step + tv.lo + k);
        const int64_t s = __ldg(bt.size_bytes + tv.lo + k), o = __ldg(offsets + tv.lo + k);
        if (!tensor_ok(a, f, s, T) || o < 0) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        if (o > INT64_MAX - s) {
            ovf = true;
            continue;
        }
        mx = o + s > mx ? o + s : mx;
    }
    bad = __syncthreads_or(bad);
    ovf = __syncthreads_or(ovf);
    sum = block_sat_sum(sum, reinterpret_cast<uint64_t*>(red));
    mx = block_max_i64(mx, red);
    if (threadIdx.x == 0) {
        const int32_t st = bad ? MP_EINVAL : (ovf || sum > (uint64_t)INT64_MAX) ? MP_EOVERFLOW : MP_OK;
        status[b] = st;
        plan_peak[b] = st == MP_OK ? mx : 0;
    }
}

}  // namespace

static bool validate_fits_smem(const mp_batch& bt) {
    return ValidateLayout(bt.max_tensors, bt.max_steps).total <= kValidateSmemLimit;
}

size_t validate_workspace_bytes(const mp_batch& bt) {
    if (bt.n_traces == 0 || validate_fits_smem(bt)) return 0;
    return (size_t)bt.n_traces * ValidateLayout(bt.max_tensors, bt.max_steps).total;
}

cudaError_t launch_validate(const mp_batch& bt, const int64_t* offsets, int32_t* verdict, int32_t* conflict,
                            int32_t* status, void* workspace, cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    dim3 grid((unsigned)bt.n_traces), block(kValidateThreads);
    if (validate_fits_smem(bt)) {
        const size_t smem = ValidateLayout(bt.max_tensors, bt.max_steps).total;
        cudaError_t e = set_smem_limit((const void*)k_validate<true>, smem);
        if (e != cudaSuccess) return e;
        k_validate<true><<<grid, block, smem, stream>>>(bt, offsets, verdict, conflict, status, nullptr, 0);
    } else {
        const size_t stride = ValidateLayout(bt.max_tensors, bt.max_steps).total;
        k_validate<false><<<grid, block, 0, stream>>>(bt, offsets, verdict, conflict, status,
                                                       static_cast<unsigned char*>(workspace), stride);
    }
    return cudaGetLastError();
}

cudaError_t launch_peak(const mp_batch& bt, const int64_t* offsets, int64_t* plan_peak, int32_t* status,
                        cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    k_peak<<<(unsigned)bt.n_traces, kPeakThreads, 0, stream>>>(bt, offsets, plan_peak, status);
    return cudaGetLastError();
}

}  // namespace mp
