// bump.cu -- bump_allocation, the baseline strategy of Sec. 2.3: in allocation
// order (alloc step ascending, then id ascending) every tensor gets the
// running offset, the sum of the sizes allocated before it, and the plan's
// peak is the sum of all sizes (no address range is ever reused).
//
// GPU form: one CTA per trace.  offset_i = SX[a_i] + (sizes of the tensors
// allocated at step a_i with a smaller id), SX being the exclusive scan over
// steps of the per-step size sums.  The same-step part comes from a counting
// sort of the tensors into per-step buckets and, per tensor, a pass over its
// own bucket (a few tensors on the traces this library is built for).
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

// Per-trace working set: per-step size sums (then their exclusive scan) and
// bucket ends; per bucket position the tensor's id, size and alloc step.
struct BumpLayout {
    size_t sx, bend, id, sz, al, total;
    __host__ __device__ BumpLayout(int64_t n, int64_t T) {
        sx = 0;
        bend = sx + align_up((size_t)T * 8);
        sz = bend + align_up((size_t)T * 4);
        id = sz + align_up((size_t)n * 8);
        al = id + align_up((size_t)n * 4);
        total = al + align_up((size_t)n * 4);
    }
};

struct BumpShared {
    unsigned long long sum_hi, sum_lo;
    int bad;
};

template <bool kSmem>
__global__ void __launch_bounds__(kBumpThreads, kSmem ? 8 : 1)
k_bump(mp_batch bt, int64_t* __restrict__ offsets, int64_t* __restrict__ plan_peak, int32_t* __restrict__ status,
       unsigned char* __restrict__ ws, size_t ws_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int64_t red[72];
    __shared__ BumpShared sh;
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) {
            status[b] = tv.st;
            plan_peak[b] = 0;
        }
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const BumpLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * ws_stride;
    int64_t* SX = reinterpret_cast<int64_t*>(base + L.sx);
    int32_t* BEND = reinterpret_cast<int32_t*>(base + L.bend);
    int64_t* SZ = reinterpret_cast<int64_t*>(base + L.sz);
    int32_t* ID = reinterpret_cast<int32_t*>(base + L.id);
    int32_t* AL = reinterpret_cast<int32_t*>(base + L.al);

    for (int t = threadIdx.x; t < T; t += blockDim.x) {
        SX[t] = 0;
        BEND[t] = 0;
    }
    if (threadIdx.x == 0) {
        sh.sum_hi = sh.sum_lo = 0;
        sh.bad = 0;
    }
    __syncthreads();

    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    bool bad = false;
    uint64_t sum = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t s = __ldg(Sg + k);
        if (!tensor_ok(a, f, s, T)) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        atomicAdd(BEND + a, 1);
        atomic_add_u64_split(SX + a, (uint64_t)s);
    }
    block_add_size_sum(sum, &sh.sum_hi, &sh.sum_lo);
    if (bad) sh.bad = 1;
    __syncthreads();
    if (sh.bad || size_sum_overflows(sh.sum_hi, sh.sum_lo)) {
        if (threadIdx.x == 0) {
            status[b] = sh.bad ? MP_EINVAL : MP_EOVERFLOW;
            plan_peak[b] = 0;
        }
        return;
    }

    // Bucket starts and bytes allocated before each step; then the scatter
    // leaves BEND[t] as the end of bucket t.
    block_excl_scan_array<int32_t, 8>(BEND, T, reinterpret_cast<int32_t*>(red));
    const int64_t total = block_excl_scan_array<int64_t, 8>(SX, T, red);
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k);
        const int32_t pos = atomicAdd(BEND + a, 1);
        ID[pos] = k;
        SZ[pos] = __ldg(Sg + k);
        AL[pos] = a;
    }
    __syncthreads();

    int64_t* __restrict__ out = offsets + tv.lo;
    for (int p = threadIdx.x; p < n; p += blockDim.x) {
        const int32_t a = AL[p], id = ID[p];
        const int32_t lo = a == 0 ? 0 : BEND[a - 1], hi = BEND[a];
        int64_t off = SX[a];
        for (int q = lo; q < hi; ++q)
            if (ID[q] < id) off += SZ[q];
        out[id] = off;
    }
    if (threadIdx.x == 0) {
        plan_peak[b] = total;
        status[b] = MP_OK;
    }
}

bool bump_fits_smem(const mp_batch& bt) { return BumpLayout(bt.max_tensors, bt.max_steps).total <= kSmemCeiling; }

}  // namespace

size_t bump_workspace_bytes(const mp_batch& bt) {
    if (bt.n_traces == 0 || bump_fits_smem(bt)) return 0;
    return mul_sat((size_t)bt.n_traces, BumpLayout(bt.max_tensors, bt.max_steps).total);
}

cudaError_t launch_bump(const mp_batch& bt, int64_t* offsets, int64_t* plan_peak, int32_t* status, void* workspace,
                        cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    dim3 grid((unsigned)bt.n_traces), block(kBumpThreads);
    const size_t bytes = BumpLayout(bt.max_tensors, bt.max_steps).total;
    if (bump_fits_smem(bt)) {
        cudaError_t e = set_smem_limit((const void*)k_bump<true>, bytes);
        if (e != cudaSuccess) return e;
        k_bump<true><<<grid, block, bytes, stream>>>(bt, offsets, plan_peak, status, nullptr, 0);
    } else {
        k_bump<false><<<grid, block, 0, stream>>>(bt, offsets, plan_peak, status,
                                                   static_cast<unsigned char*>(workspace), bytes);
    }
    return cudaGetLastError();
}

}  // namespace mp
