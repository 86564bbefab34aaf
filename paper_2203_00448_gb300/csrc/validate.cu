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

// Per-trace working set: tensors scattered into alloc-step order as 16-byte
// records -- (offset, end, free step, id) as 32-bit words when every end of
// the trace is below 2^32, else (offset, end) as 64-bit words with the (free
// step, id) pairs beside them -- plus the bucket ends.
struct ValidateLayout {
    size_t rec, fi, bend, total;
    __host__ __device__ ValidateLayout(int64_t n, int64_t T) {
        rec = 0;
        fi = rec + align_up((size_t)n * 16);
        bend = fi + align_up((size_t)n * 8);
        total = bend + align_up((size_t)T * 4);
    }
};

// Per-trace flags, or-ed over the block.
constexpr int kFlagInvalid = 1;  // a tensor breaks 0 <= a < f <= T, s >= 1, or has offset < 0
constexpr int kFlagEndOvf = 2;   // offset + size past INT64_MAX
constexpr int kFlagWide = 4;     // an end at or above 2^32
constexpr int kFlagBigSize = 8;  // a size at or above 2^32: the size sum needs the exact check

struct ValidateShared {
    unsigned long long key;
    unsigned int sum[3];  // the sizes' sum in three 21-bit limbs (carries kept)
    int flags;
};

constexpr int kValCached = 4;  // tensors per thread held in registers between the two passes
constexpr int kValItems = 8;   // bucket counts scanned per thread per tile

// Adds a warp's per-lane saturated size sums into the three 21-bit limbs of
// sum: every lane's limb is below 2^22, so a 32-bit warp reduction of each
// cannot wrap, nor can the block's 32-bit shared sums (at most 32 warps).
__device__ __forceinline__ void block_add_size_limbs(uint64_t v, unsigned int* sum) {
    const unsigned full = 0xffffffffu;
    const unsigned l0 = __reduce_add_sync(full, (unsigned)(v & 0x1fffffu));
    const unsigned l1 = __reduce_add_sync(full, (unsigned)((v >> 21) & 0x1fffffu));
    const unsigned l2 = __reduce_add_sync(full, (unsigned)(v >> 42));
    if ((threadIdx.x & 31) == 0 && (l0 | l1 | l2)) {
        atomicAdd(sum, l0);
        atomicAdd(sum + 1, l1);
        atomicAdd(sum + 2, l2);
    }
}

// True if the limbs add up to more than INT64_MAX.
__device__ __forceinline__ bool size_limbs_overflow(const unsigned int* sum) {
    const uint64_t l0 = sum[0], l1 = sum[1] + (l0 >> 21), l2 = sum[2] + (l1 >> 21);
    return l2 >= (1ull << 21);  // bits 42 and up reach 2^63
}

// In-place exclusive scan of the shared, 16-byte aligned x[0, len) by the
// whole block, kValItems consecutive entries per thread per tile; ends with a
// barrier.
__device__ void block_excl_scan_i32(int32_t* x, int32_t len, int32_t* red) {
    int32_t carry = 0;
    const int32_t tile = (int32_t)blockDim.x * kValItems;
    for (int32_t base = 0; base < len; base += tile) {
        const int32_t my = base + (int32_t)threadIdx.x * kValItems;
        const bool full = my + kValItems <= len;
        int32_t v[kValItems];
        if (full) {
            const int4 u = *reinterpret_cast<const int4*>(x + my), w = *reinterpret_cast<const int4*>(x + my + 4);
            v[0] = u.x, v[1] = u.y, v[2] = u.z, v[3] = u.w, v[4] = w.x, v[5] = w.y, v[6] = w.z, v[7] = w.w;
        } else {
#pragma unroll
            for (int k = 0; k < kValItems; ++k) v[k] = my + k < len ? x[my + k] : 0;
        }
        int32_t sum = 0;
#pragma unroll
        for (int k = 0; k < kValItems; ++k) sum += v[k];
        int32_t tot;
        int32_t pre = block_excl_scan<int32_t>(sum, red, &tot) + carry;
#pragma unroll
        for (int k = 0; k < kValItems; ++k) {
            const int32_t t = v[k];
            v[k] = pre;
            pre += t;
        }
        if (full) {
            *reinterpret_cast<int4*>(x + my) = make_int4(v[0], v[1], v[2], v[3]);
            *reinterpret_cast<int4*>(x + my + 4) = make_int4(v[4], v[5], v[6], v[7]);
        } else {
#pragma unroll
            for (int k = 0; k < kValItems; ++k)
                if (my + k < len) x[my + k] = v[k];
        }
        carry += tot;
    }
    __syncthreads();
}

__device__ __forceinline__ unsigned long long pair_key(uint32_t i, uint32_t j) {
    const uint32_t lo = i < j ? i : j, hi = i < j ? j : i;
    return ((unsigned long long)lo << 32) | hi;
}

// Every lifetime-overlapping pair once, from its earlier member in alloc
// order (positions p < q < BEND[f_p - 1]), over narrow records.
__device__ __forceinline__ void check_pairs_narrow(const uint4* __restrict__ rec, const int32_t* __restrict__ bend,
                                                   int32_t n, unsigned long long* key) {
    for (int32_t p = threadIdx.x; p < n; p += blockDim.x) {
        const uint4 ri = rec[p];
        const int32_t stop = bend[(int32_t)ri.z - 1];
        for (int32_t q = p + 1; q < stop; ++q) {
            const uint4 rj = rec[q];
            if (ri.x < rj.y && rj.x < ri.y) atomicMin(key, pair_key(ri.w, rj.w));
        }
    }
}

// The same over 64-bit (offset, end) records with the (free step, id) pairs beside them.
__device__ __forceinline__ void check_pairs_wide(const longlong2* __restrict__ rec, const int2* __restrict__ fi_arr,
                                                 const int32_t* __restrict__ bend, int32_t n,
                                                 unsigned long long* key) {
    for (int32_t p = threadIdx.x; p < n; p += blockDim.x) {
        const int2 fi = fi_arr[p];
        const int32_t stop = bend[fi.x - 1];
        if (stop <= p + 1) continue;
        const longlong2 ri = rec[p];
        for (int32_t q = p + 1; q < stop; ++q) {
            const longlong2 rj = rec[q];
            if (ri.x < rj.y && rj.x < ri.y) atomicMin(key, pair_key((uint32_t)fi.y, (uint32_t)fi_arr[q].y));
        }
    }
}

// One CTA per trace.  A trace of at most kValCached * blockDim tensors is
// loaded into registers before anything else (16-byte loads when its slices
// are aligned) and kept there for the scatter, so its inputs are read from
// memory once; a larger trace is read twice, by plain loops.  The two cases
// are separate code paths (kCached), so that no cached value is live across
// a loop that reads memory: inlined together, those loops made the kernel
// spill registers even for traces that never ran them.  Traces whose ends all lie
// below 2^32 (the flag reduction tells) take 8-byte records and 32-bit
// compares; the exact size sum is only formed when some size reaches 2^32
// (below that, n < 2^31 sizes cannot sum past INT64_MAX).
template <bool kSmem, bool kCached>
__device__ __forceinline__ void validate_trace(const mp_batch& bt, const TraceView& tv, int b,
                                               const int64_t* __restrict__ offsets, int32_t* __restrict__ verdict,
                                               int32_t* __restrict__ conflict, int32_t* __restrict__ status,
                                               unsigned char* __restrict__ ws, size_t ws_stride,
                                               unsigned char* smem_raw, int32_t* red, ValidateShared& sh) {
    const int32_t n = tv.n, T = tv.T;
    const int32_t tid = (int32_t)threadIdx.x, nthr = (int32_t)blockDim.x;
    const int32_t* __restrict__ Ag = bt.alloc_step + tv.lo;
    const int32_t* __restrict__ Fg = bt.free_step + tv.lo;
    const int64_t* __restrict__ Sg = bt.size_bytes + tv.lo;
    const int64_t* __restrict__ Og = offsets + tv.lo;
    const bool vec = ((reinterpret_cast<uintptr_t>(Ag) | reinterpret_cast<uintptr_t>(Fg) |
                       reinterpret_cast<uintptr_t>(Sg) | reinterpret_cast<uintptr_t>(Og)) & 15) == 0;
    auto cidx = [&](int j) -> int32_t { return vec ? 4 * tid + j : tid + j * nthr; };
    int32_t ca[kValCached] = {}, cf[kValCached] = {};
    int64_t cs[kValCached] = {}, co[kValCached] = {};
    if (!kCached) {
        // nothing held: every tensor is read by the loops below
    } else if (vec && 4 * tid + 3 < n) {
        const int4 a = __ldg(reinterpret_cast<const int4*>(Ag) + tid);
        const int4 f = __ldg(reinterpret_cast<const int4*>(Fg) + tid);
        const longlong2 s01 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * tid);
        const longlong2 s23 = __ldg(reinterpret_cast<const longlong2*>(Sg) + 2 * tid + 1);
        const longlong2 o01 = __ldg(reinterpret_cast<const longlong2*>(Og) + 2 * tid);
        const longlong2 o23 = __ldg(reinterpret_cast<const longlong2*>(Og) + 2 * tid + 1);
        ca[0] = a.x, ca[1] = a.y, ca[2] = a.z, ca[3] = a.w;
        cf[0] = f.x, cf[1] = f.y, cf[2] = f.z, cf[3] = f.w;
        cs[0] = s01.x, cs[1] = s01.y, cs[2] = s23.x, cs[3] = s23.y;
        co[0] = o01.x, co[1] = o01.y, co[2] = o23.x, co[3] = o23.y;
    } else {
#pragma unroll
        for (int j = 0; j < kValCached; ++j) {
            const int32_t k = cidx(j);
            ca[j] = cf[j] = 0;
            cs[j] = co[j] = 0;
            if (k < n) {
                ca[j] = __ldg(Ag + k);
                cf[j] = __ldg(Fg + k);
                cs[j] = __ldg(Sg + k);
                co[j] = __ldg(Og + k);
            }
        }
    }

    const ValidateLayout L(kSmem ? n : bt.max_tensors, kSmem ? T : bt.max_steps);
    unsigned char* base = kSmem ? smem_raw : ws + (size_t)b * ws_stride;
    int2* FI = reinterpret_cast<int2*>(base + L.fi);
    int32_t* BEND = reinterpret_cast<int32_t*>(base + L.bend);
    if ((T & 3) == 0) {
        for (int32_t t = tid; t < (T >> 2); t += nthr) reinterpret_cast<int4*>(BEND)[t] = make_int4(0, 0, 0, 0);
    } else {
        for (int32_t t = tid; t < T; t += nthr) BEND[t] = 0;
    }
    if (tid == 0) {
        sh.key = ~0ull;
        sh.sum[0] = sh.sum[1] = sh.sum[2] = 0;
        sh.flags = 0;
    }
    __syncthreads();

    // Checks, flags and the alloc-step histogram.  The cached tensors keep
    // their offset and end as 32-bit words from here on (all the narrow path
    // needs); the wide path and the exact size sum read memory again.
    uint32_t bad = 0;
    uint64_t or_e = 0, or_s = 0;
    // (0 <= a < f <= T as two unsigned compares, T being >= 0; the flags are
    // or-ed over the thread's tensors and read once.  An invalid tensor's
    // bits are garbage there, but its trace fails with MP_EINVAL anyway.)
    auto take = [&](int32_t a, int32_t f, int64_t sz, int64_t o) -> uint64_t {
        const bool ok = (uint32_t)a < (uint32_t)f && (uint32_t)f <= (uint32_t)T && sz > 0 && o >= 0;
        const uint64_t e = (uint64_t)o + (uint64_t)sz;  // both below 2^63 when ok: no wrap
        bad |= ok ? 0u : 1u;
        or_e |= e;
        or_s |= (uint64_t)sz;
        if (ok) atomicAdd(BEND + a, 1);
        return e;
    };
    uint32_t co32[kValCached] = {}, ce32[kValCached] = {};
    if constexpr (kCached) {
#pragma unroll
        for (int j = 0; j < kValCached; ++j) {
            co32[j] = (uint32_t)co[j];
            ce32[j] = cidx(j) < n ? (uint32_t)take(ca[j], cf[j], cs[j], co[j]) : 0u;
        }
    } else {
        for (int32_t k = tid; k < n; k += nthr) take(__ldg(Ag + k), __ldg(Fg + k), __ldg(Sg + k), __ldg(Og + k));
    }
    int flags = (bad ? kFlagInvalid : 0) | ((or_e >> 63) ? kFlagEndOvf : 0) | ((or_e >> 32) ? kFlagWide : 0) |
                ((or_s >> 32) ? kFlagBigSize : 0);
    flags = (int)__reduce_or_sync(0xffffffffu, (unsigned)flags);
    if ((tid & 31) == 0 && flags) atomicOr(&sh.flags, flags);
    __syncthreads();
    const int F = sh.flags;
    bool sum_ovf = false;
    if ((F & (kFlagInvalid | kFlagBigSize)) == kFlagBigSize) {  // the exact size sum (rare)
        uint64_t sum = 0;
        for (int32_t k = tid; k < n; k += nthr) sum = sat_add(sum, (uint64_t)__ldg(Sg + k));
        block_add_size_limbs(sum, sh.sum);
        __syncthreads();
        sum_ovf = size_limbs_overflow(sh.sum);
    }
    if ((F & (kFlagInvalid | kFlagEndOvf)) || sum_ovf) {
        if (tid == 0) {
            status[b] = (F & kFlagInvalid) ? MP_EINVAL : MP_EOVERFLOW;
            verdict[b] = 0;
            if (conflict) conflict[2 * b] = conflict[2 * b + 1] = -1;
        }
        return;
    }
    // Counting sort by alloc step: bucket starts, then scatter; afterwards
    // BEND[t] is the end of bucket t (tensors with alloc <= t).
    block_excl_scan_i32(BEND, T, red);
    const bool wide = (F & kFlagWide) != 0;
    uint4* REC32 = reinterpret_cast<uint4*>(base + L.rec);
    longlong2* REC64 = reinterpret_cast<longlong2*>(base + L.rec);
    auto scatter = [&](int32_t k, int32_t a, int32_t f, uint32_t o32, uint32_t e32) {
        const int32_t pos = atomicAdd(BEND + a, 1);
        if (wide) {
            const int64_t o = __ldg(Og + k);
            REC64[pos] = make_longlong2(o, o + __ldg(Sg + k));
            FI[pos] = make_int2(f, k);
        } else {
            REC32[pos] = make_uint4(o32, e32, (uint32_t)f, (uint32_t)k);
        }
    };
    if constexpr (kCached) {
#pragma unroll
        for (int j = 0; j < kValCached; ++j) {
            const int32_t k = cidx(j);
            if (k < n) scatter(k, ca[j], cf[j], co32[j], ce32[j]);
        }
    } else {
        for (int32_t k = tid; k < n; k += nthr) {
            const uint32_t o32 = wide ? 0u : (uint32_t)__ldg(Og + k);
            scatter(k, __ldg(Ag + k), __ldg(Fg + k), o32, wide ? 0u : o32 + (uint32_t)__ldg(Sg + k));
        }
    }
    __syncthreads();

    if (wide)
        check_pairs_wide(REC64, FI, BEND, n, &sh.key);
    else
        check_pairs_narrow(REC32, BEND, n, &sh.key);
    __syncthreads();
    if (tid == 0) {
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

template <bool kSmem>
__global__ void __launch_bounds__(kValidateThreads, kSmem ? 9 : 1)
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
    if (tv.n <= kValCached * (int32_t)blockDim.x)
        validate_trace<kSmem, true>(bt, tv, b, offsets, verdict, conflict, status, ws, ws_stride, smem_raw, red, sh);
    else
        validate_trace<kSmem, false>(bt, tv, b, offsets, verdict, conflict, status, ws, ws_stride, smem_raw, red,
                                     sh);
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
    return mul_sat((size_t)bt.n_traces, ValidateLayout(bt.max_tensors, bt.max_steps).total);
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
