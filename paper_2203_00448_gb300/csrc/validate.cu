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

// Per-trace working set: tensors scattered into alloc-step order as packed
// (offset, end) records with their id and free step, plus the bucket ends.
struct ValidateLayout {
    size_t rec, id, fp, bend, total;
    __host__ __device__ ValidateLayout(int64_t n, int64_t T) {
        rec = 0;
        id = rec + align_up((size_t)n * 16);
        fp = id + align_up((size_t)n * 4);
        bend = fp + align_up((size_t)n * 4);
        total = bend + align_up((size_t)T * 4);
    }
};

struct ValidateShared {
    unsigned long long key, sum_hi, sum_lo;
    int bad, ovf;
};

template <bool kSmem>
__global__ void __launch_bounds__(kValidateThreads, kSmem ? 12 : 1)
k_validate(mp_batch bt, const int64_t* __restrict__ offsets, int32_t* __restrict__ verdict,
           int32_t* __restrict__ conflict, int32_t* __restrict__ status, unsigned char* __restrict__ ws,
           size_t ws_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int32_t red[40];
    __shared__ ValidateShared sh;
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) status[b] = tv.st;
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const ValidateLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * ws_stride;
    longlong2* REC = reinterpret_cast<longlong2*>(base + L.rec);
    int32_t* ID = reinterpret_cast<int32_t*>(base + L.id);
    int32_t* FP = reinterpret_cast<int32_t*>(base + L.fp);
    int32_t* BEND = reinterpret_cast<int32_t*>(base + L.bend);

    for (int t = threadIdx.x; t < T; t += blockDim.x) BEND[t] = 0;
    if (threadIdx.x == 0) {
        sh.key = ~0ull;
        sh.sum_hi = sh.sum_lo = 0;
        sh.bad = sh.ovf = 0;
    }
    __syncthreads();

    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    const int64_t* __restrict__ Og = offsets + tv.lo;
    bool bad = false, ovf = false;
    uint64_t sum = 0;
    auto check = [&](int32_t a, int32_t f, int64_t sz, int64_t o) {
        if (!tensor_ok(a, f, sz, T) || o < 0) {
            bad = true;
            return;
        }
        sum = sat_add(sum, (uint64_t)sz);
        if (o > INT64_MAX - sz) ovf = true;
        atomicAdd(BEND + a, 1);
    };
    const bool vec_in = ((reinterpret_cast<uintptr_t>(Ag) | reinterpret_cast<uintptr_t>(Fg) |
                          reinterpret_cast<uintptr_t>(Sg) | reinterpret_cast<uintptr_t>(Og)) & 15) == 0;
    int k0 = 0;
    if (vec_in) {
        const int n4 = n >> 2;
        for (int q = threadIdx.x; q < n4; q += blockDim.x) {
            const int4 a = __ldg(reinterpret_cast<const int4*>(Ag) + q);
            const int4 f = __ldg(reinterpret_cast<const int4*>(Fg) + q);
            const longlong2 s01 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * q);
            const longlong2 s23 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * q + 1);
            const longlong2 o01 = __ldg(reinterpret_cast<const longlong2*>(Og) + 2 * q);
            const longlong2 o23 = __ldg(reinterpret_cast<const longlong2*>(Og) + 2 * q + 1);
            check(a.x, f.x, s01.x, o01.x);
            check(a.y, f.y, s01.y, o01.y);
            check(a.z, f.z, s23.x, o23.x);
            check(a.w, f.w, s23.y, o23.y);
        }
        k0 = n4 << 2;
    }
    for (int k = k0 + threadIdx.x; k < n; k += blockDim.x)
        check(__ldg(Ag + k), __ldg(Fg + k), __ldg(Sg + k), __ldg(Og + k));
    block_add_size_sum(sum, &sh.sum_hi, &sh.sum_lo);
    if (bad) sh.bad = 1;
    if (ovf) sh.ovf = 1;
    __syncthreads();
    if (sh.bad || sh.ovf || size_sum_overflows(sh.sum_hi, sh.sum_lo)) {
        if (threadIdx.x == 0) {
            status[b] = sh.bad ? MP_EINVAL : MP_EOVERFLOW;
            verdict[b] = 0;
            if (conflict) conflict[2 * b] = conflict[2 * b + 1] = -1;
        }
        return;
    }
    // Counting sort by alloc step: bucket starts, then scatter; afterwards
    // BEND[t] is the end of bucket t (tensors with alloc <= t).
    block_excl_scan_array<int32_t, 8>(BEND, T, red);
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k);
        const int64_t o = __ldg(Og + k);
        const int32_t pos = atomicAdd(BEND + a, 1);
        REC[pos] = make_longlong2(o, o + __ldg(Sg + k));
        ID[pos] = k;
        FP[pos] = __ldg(Fg + k);
    }
    __syncthreads();

    // Each overlapping pair once, from its earlier member in alloc order.
    for (int p = threadIdx.x; p < n; p += blockDim.x) {
        const int32_t stop = BEND[FP[p] - 1];
        if (stop <= p + 1) continue;
        const longlong2 ri = REC[p];
        for (int q = p + 1; q < stop; ++q) {
            const longlong2 rj = REC[q];
            if (ri.x < rj.y && rj.x < ri.y) {
                const uint32_t i = (uint32_t)ID[p], j = (uint32_t)ID[q];
                const uint32_t lo = i < j ? i : j, hi = i < j ? j : i;
                atomicMin(&sh.key, ((unsigned long long)lo << 32) | hi);
            }
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned long long key = sh.key;
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
