// replay.cu -- a plan materialised on device memory and replayed, the check
// on real memory of what Eq. 2.1 states on paper.  Sec. 3.3 materialises a
// plan as one slab per graph (prim::AllocateSlab[total_size]) with every
// tensor a view at its offset (prim::AllocateTensor); here every trace gets a
// slab in one device buffer (mp_slab_layout), and mp_replay_plan walks the
// trace's steps in order: at step t every tensor allocated at t fills its
// byte range with a pattern of its own (a mix of its id and the byte
// address), then every tensor whose last live step is t checks its range.
// If two tensors overlap in lifetime and in address, one of them is written
// while the other is live and fails its check; tensors that only touch in
// time (free_i = alloc_j) never meet, because i is checked before j writes.
// So a plan replays cleanly iff it is valid.
#include "common.cuh"
#include "launch.h"

namespace mp {

namespace {

// Per-trace working set: bucket ends by alloc step and by last live step,
// then the tensor ids in each order.
struct ReplayLayout {
    size_t ba, bf, la, lf, total;
    __host__ __device__ ReplayLayout(int64_t n, int64_t T) {
        ba = 0;
        bf = ba + align_up((size_t)T * 4);
        la = bf + align_up((size_t)T * 4);
        lf = la + align_up((size_t)n * 4);
        total = lf + align_up((size_t)n * 4);
    }
};

// Pattern word of tensor `id` at slab word `w` (never zero).
__device__ __forceinline__ uint32_t pattern(uint32_t id, uint64_t w) {
    uint32_t x = id * 0x9E3779B1u ^ (uint32_t)w * 0x85EBCA77u ^ (uint32_t)(w >> 32) * 0xC2B2AE3Du;
    x ^= x >> 15;
    x *= 0x2C1B3C6Du;
    x ^= x >> 12;
    return x | 1u;
}

// Writes (check = false) or compares (check = true) tensor id's pattern over
// slab bytes [lo, hi), the whole block cooperating; returns false if a
// compared byte differs (block-wide result).
__device__ bool fill_or_check(unsigned char* __restrict__ slab, int64_t lo, int64_t hi, uint32_t id, bool check,
                              int* s_flag) {
    const int64_t wlo = (lo + 3) >> 2, whi = hi >> 2;  // whole words inside [lo, hi)
    bool good = true;
    auto byte_of = [&](int64_t x) { return (unsigned char)(pattern(id, (uint64_t)x >> 2) >> (8 * (x & 3))); };
    if (wlo <= whi) {
        for (int64_t x = lo + threadIdx.x; x < (wlo << 2); x += blockDim.x) {  // head bytes
            if (check) good &= slab[x] == byte_of(x);
            else slab[x] = byte_of(x);
        }
        uint32_t* words = reinterpret_cast<uint32_t*>(slab);
        for (int64_t w = wlo + threadIdx.x; w < whi; w += blockDim.x) {
            if (check) good &= words[w] == pattern(id, (uint64_t)w);
            else words[w] = pattern(id, (uint64_t)w);
        }
        for (int64_t x = (whi << 2) + threadIdx.x; x < hi; x += blockDim.x) {  // tail bytes
            if (check) good &= slab[x] == byte_of(x);
            else slab[x] = byte_of(x);
        }
    } else {  // inside one word
        for (int64_t x = lo + threadIdx.x; x < hi; x += blockDim.x) {
            if (check) good &= slab[x] == byte_of(x);
            else slab[x] = byte_of(x);
        }
    }
    if (!check) return true;
    if (!good) atomicExch(s_flag, 0);
    return true;
}

template <bool kSmem>
__global__ void __launch_bounds__(kReplayThreads)
k_replay(mp_batch bt, const int64_t* __restrict__ offsets, const int64_t* __restrict__ slab_base,
         unsigned char* __restrict__ slab, int64_t slab_bytes, int32_t* __restrict__ ok,
         int32_t* __restrict__ first_bad, int32_t* __restrict__ status, unsigned char* __restrict__ ws,
         size_t ws_stride) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ int32_t red[40];
    __shared__ int s_bad, s_good, s_first;
    __shared__ unsigned long long s_hi, s_lo;
    const int b = blockIdx.x;
    const TraceView tv = load_trace(bt, b, false);
    if (tv.st != MP_OK) {
        if (threadIdx.x == 0) {
            status[b] = tv.st;
            ok[b] = 0;
            first_bad[b] = -1;
        }
        return;
    }
    const int32_t n = tv.n, T = tv.T;
    const ReplayLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * ws_stride;
    int32_t* BA = reinterpret_cast<int32_t*>(base + L.ba);
    int32_t* BF = reinterpret_cast<int32_t*>(base + L.bf);
    int32_t* LA = reinterpret_cast<int32_t*>(base + L.la);
    int32_t* LF = reinterpret_cast<int32_t*>(base + L.lf);
    const int64_t sb0 = __ldg(slab_base + b), sb1 = __ldg(slab_base + b + 1);
    for (int t = threadIdx.x; t < T; t += blockDim.x) BA[t] = BF[t] = 0;
    if (threadIdx.x == 0) {
        s_bad = 0;
        s_good = 1;
        s_first = INT32_MAX;
        s_hi = s_lo = 0;
    }
    __syncthreads();

    // Checks: valid tensors, the trace's slab inside the buffer, every tensor
    // inside the trace's slab -- before any byte is written.
    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    const int64_t* __restrict__ Og = offsets + tv.lo;
    bool bad = !(0 <= sb0 && sb0 <= sb1 && sb1 <= slab_bytes);
    uint64_t sum = 0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        const int32_t a = __ldg(Ag + k), f = __ldg(Fg + k);
        const int64_t s = __ldg(Sg + k), o = __ldg(Og + k);
        if (!tensor_ok(a, f, s, T) || o < 0 || o > (sb1 - sb0) - s) {
            bad = true;
            continue;
        }
        sum = sat_add(sum, (uint64_t)s);
        atomicAdd(BA + a, 1);
        atomicAdd(BF + (f - 1), 1);
    }
    block_add_size_sum(sum, &s_hi, &s_lo);
    if (bad) s_bad = 1;
    __syncthreads();
    if (s_bad || size_sum_overflows(s_hi, s_lo)) {
        if (threadIdx.x == 0) {
            status[b] = s_bad ? MP_EINVAL : MP_EOVERFLOW;
            ok[b] = 0;
            first_bad[b] = -1;
        }
        return;
    }
    block_excl_scan_array<int32_t, 8>(BA, T, red);
    block_excl_scan_array<int32_t, 8>(BF, T, red);
    for (int k = threadIdx.x; k < n; k += blockDim.x) {
        LA[atomicAdd(BA + __ldg(Ag + k), 1)] = k;
        LF[atomicAdd(BF + (__ldg(Fg + k) - 1), 1)] = k;
    }
    __syncthreads();

    // Replay: after the scatter, BA[t] / BF[t] are the bucket ends.
    for (int t = 0; t < T; ++t) {
        const int a0 = t == 0 ? 0 : BA[t - 1], a1 = BA[t];
        for (int q = a0; q < a1; ++q) {
            const int k = LA[q];
            const int64_t lo = sb0 + __ldg(Og + k);
            fill_or_check(slab, lo, lo + __ldg(Sg + k), (uint32_t)k, false, &s_good);
        }
        __syncthreads();  // this step's tensors are written
        const int f0 = t == 0 ? 0 : BF[t - 1], f1 = BF[t];
        for (int q = f0; q < f1; ++q) {
            const int k = LF[q];
            const int64_t lo = sb0 + __ldg(Og + k);
            if (threadIdx.x == 0) s_good = 1;
            __syncthreads();
            fill_or_check(slab, lo, lo + __ldg(Sg + k), (uint32_t)k, true, &s_good);
            __syncthreads();
            if (threadIdx.x == 0 && !s_good) s_first = min(s_first, k);
        }
        __syncthreads();  // checks done before the next step writes
    }
    if (threadIdx.x == 0) {
        ok[b] = s_first == INT32_MAX ? 1 : 0;
        first_bad[b] = s_first == INT32_MAX ? -1 : s_first;
        status[b] = MP_OK;
    }
}

// Slab of every trace: plan_peak rounded up to kAlign, 0 for a failed trace
// (trace_status non-zero) or a negative peak; slab_base is their exclusive
// scan, with the total after the last trace.
__global__ void __launch_bounds__(1024) k_slab_layout(int32_t n_traces, const int64_t* __restrict__ plan_peak,
                                                     const int32_t* __restrict__ trace_status,
                                                     int64_t* __restrict__ slab_base) {
    __shared__ int64_t red[40];
    int64_t carry = 0;
    for (int64_t base = 0; base < n_traces; base += blockDim.x) {
        const int64_t b = base + threadIdx.x;
        int64_t v = 0;
        if (b < n_traces && (trace_status == nullptr || trace_status[b] == MP_OK))
            v = (int64_t)align_up((size_t)max(plan_peak[b], (int64_t)0));
        int64_t tot;
        const int64_t pre = block_excl_scan<int64_t>(v, red, &tot) + carry;
        if (b < n_traces) slab_base[b] = pre;
        carry += tot;
    }
    if (threadIdx.x == 0) slab_base[n_traces] = carry;
}

// Byte address of every tensor in the slab buffer (Sec. 3.3's
// prim::AllocateTensor[size, offset] view of prim::AllocateSlab): one CTA per
// trace; slab_base[b] + offset for a trace with status 0 whose CSR range is
// sound, -1 for the tensors of a failed trace.
__global__ void __launch_bounds__(256) k_slab_addresses(mp_batch bt, const int64_t* __restrict__ offsets,
                                                       const int32_t* __restrict__ trace_status,
                                                       const int64_t* __restrict__ slab_base,
                                                       int64_t* __restrict__ tensor_addr) {
    const int b = blockIdx.x;
    const int64_t lo = bt.trace_ptr[b], hi = bt.trace_ptr[b + 1];
    if (lo < 0 || hi < lo || hi > bt.n_tensors) return;  // no sound range to write
    const bool ok = trace_status == nullptr || trace_status[b] == MP_OK;
    const int64_t sb = slab_base[b];
    for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) tensor_addr[i] = ok ? sb + offsets[i] : -1;
}

bool replay_fits_smem(const mp_batch& bt) {
    return ReplayLayout(bt.max_tensors, bt.max_steps).total <= kSmemCeiling;
}

}  // namespace

size_t replay_workspace_bytes(const mp_batch& bt) {
    if (bt.n_traces == 0 || replay_fits_smem(bt)) return 0;
    return mul_sat((size_t)bt.n_traces, ReplayLayout(bt.max_tensors, bt.max_steps).total);
}

cudaError_t launch_slab_layout(const mp_batch& bt, const int64_t* plan_peak, const int32_t* trace_status,
                               const int64_t* offsets, int64_t* slab_base, int64_t* tensor_addr, cudaStream_t stream) {
    k_slab_layout<<<1, 1024, 0, stream>>>(bt.n_traces, plan_peak, trace_status, slab_base);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || tensor_addr == nullptr || bt.n_traces == 0) return e;
    k_slab_addresses<<<(unsigned)bt.n_traces, 256, 0, stream>>>(bt, offsets, trace_status, slab_base, tensor_addr);
    return cudaGetLastError();
}

cudaError_t launch_replay(const mp_batch& bt, const int64_t* offsets, const int64_t* slab_base, unsigned char* slab,
                          int64_t slab_bytes, int32_t* ok, int32_t* first_bad, int32_t* status, void* workspace,
                          cudaStream_t stream) {
    if (bt.n_traces == 0) return cudaSuccess;
    const size_t bytes = ReplayLayout(bt.max_tensors, bt.max_steps).total;
    if (replay_fits_smem(bt)) {
        cudaError_t e = set_smem_limit((const void*)k_replay<true>, bytes);
        if (e != cudaSuccess) return e;
        k_replay<true><<<(unsigned)bt.n_traces, kReplayThreads, bytes, stream>>>(
            bt, offsets, slab_base, slab, slab_bytes, ok, first_bad, status, nullptr, 0);
    } else {
        k_replay<false><<<(unsigned)bt.n_traces, kReplayThreads, 0, stream>>>(
            bt, offsets, slab_base, slab, slab_bytes, ok, first_bad, status, static_cast<unsigned char*>(workspace),
            bytes);
    }
    return cudaGetLastError();
}

}  // namespace mp
