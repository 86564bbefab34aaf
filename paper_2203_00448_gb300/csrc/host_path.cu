// host_path.cu -- the whole path from host memory: mp_plan_and_validate_host.
//
// The batch is cut into chunks of consecutive traces with about equal tensor
// counts.  Three streams overlap the work: chunk k's inputs are copied to the
// device on the copy-in stream, planned (mp_plan_and_validate's fused
// launches) on the compute stream once they have landed, and its profile and
// offsets copied back on the copy-out stream once planned.  The copy engines
// of the two directions and the SMs then work on different chunks at once.
// Cross-stream order uses events from a pool the library creates once per
// device; a per-device mutex serialises the enqueueing of concurrent callers,
// so each call's waits always refer to its own records.
#include <algorithm>
#include <cstdint>
#include <map>
#include <mutex>
#include <vector>

#include "launch.h"
#include "memplan.h"

namespace {

// Device buffer layout: inputs, outputs, then the planner's workspace for
// the largest chunk; every region starts on a kAlign boundary.  The per-trace
// inputs sit in one region (pertrace, room for trace_ptr, profile_ptr and
// steps with up to 15 bytes between them) and the per-trace results in
// another, adjacent in the order peak_lb, plan_peak, verdict, conflict,
// status, so that each can move in one copy when the host arrays are laid
// out the same way.
struct HostPathLayout {
    size_t pertrace, alloc, free_, size, profile, offsets, results, peak_lb, plan_peak, verdict, conflict, status,
        workspace, total;
};

HostPathLayout host_path_layout(const mp_batch& hb, size_t ws_bytes) {
    using mp::align_up;
    const size_t B = (size_t)hb.n_traces, N = (size_t)hb.n_tensors, S = (size_t)hb.n_steps;
    HostPathLayout L;
    size_t at = 0;
    auto take = [&](size_t bytes) {  // saturates at SIZE_MAX: such a layout never fits a buffer
        const size_t here = at;
        at = bytes > SIZE_MAX - mp::kAlign ? SIZE_MAX : mp::add_sat(at, align_up(bytes));
        return here;
    };
    using mp::mul_sat;
    L.pertrace = take(mp::add_sat(mul_sat(mul_sat(B + 1, 8), 2), mp::add_sat(mul_sat(B, 4), 32)));
    L.alloc = take(mul_sat(N, 4));
    L.free_ = take(mul_sat(N, 4));
    L.size = take(mul_sat(N, 8));
    L.profile = take(mul_sat(S, 8));
    L.offsets = take(mul_sat(N, 8));
    L.results = take(mp::add_sat(mul_sat(B, 16), mul_sat(B, 16)));
    L.peak_lb = L.results;
    L.plan_peak = L.peak_lb + (size_t)B * 8;
    L.verdict = L.plan_peak + (size_t)B * 8;
    L.conflict = L.verdict + (size_t)B * 4;
    L.status = L.conflict + (size_t)B * 8;
    L.workspace = take(ws_bytes);
    L.total = at;
    return L;
}

// Trace boundaries of the chunks: chunk k is [bounds[k], bounds[k + 1]).
std::vector<int32_t> chunk_bounds(const mp_batch& hb, int32_t chunks) {
    std::vector<int32_t> b{0};
    const int64_t N = hb.n_tensors;
    for (int32_t k = 1; k < chunks; ++k) {
        const int64_t target = N * k / chunks;
        const int64_t* it = std::lower_bound(hb.trace_ptr, hb.trace_ptr + hb.n_traces + 1, target);
        const int32_t bk = (int32_t)std::min<int64_t>(it - hb.trace_ptr, hb.n_traces);
        if (bk > b.back()) b.push_back(bk);
    }
    if (hb.n_traces > b.back()) b.push_back(hb.n_traces);
    return b;
}

// The planner workspace of the largest chunk.
size_t chunk_workspace_bytes(const mp_batch& hb, const std::vector<int32_t>& bounds) {
    size_t ws = 0;
    for (size_t k = 0; k + 1 < bounds.size(); ++k) {
        mp_batch c = hb;
        c.n_traces = bounds[k + 1] - bounds[k];
        ws = std::max(ws, mp::plan_workspace_bytes(c));
    }
    return ws;
}

// Host-side checks of the host batch: pointers, scalars, and CSR arrays that
// start at 0, never decrease and end at n_tensors / n_steps (the chunk
// copies are cut along them).
mp_status check_host_batch(const mp_batch* hb) {
    if (hb == nullptr) return MP_EINVAL;
    if (hb->n_traces < 0 || hb->max_tensors < 0 || hb->max_steps < 0 || hb->reserved0 != 0 || hb->n_tensors < 0 ||
        hb->n_steps < 0 || hb->max_tensors > mp::kPlanMaxTensors)
        return MP_EINVAL;
    const int64_t B = hb->n_traces, N = hb->n_tensors;
    auto ok = [](const void* p, int64_t len, size_t align) {
        return len <= 0 || (p != nullptr && reinterpret_cast<uintptr_t>(p) % align == 0);
    };
    if (hb->trace_ptr == nullptr || hb->profile_ptr == nullptr || !ok(hb->trace_ptr, B + 1, 8) ||
        !ok(hb->profile_ptr, B + 1, 8) || !ok(hb->steps, B, 4) || !ok(hb->alloc_step, N, 4) ||
        !ok(hb->free_step, N, 4) || !ok(hb->size_bytes, N, 8))
        return MP_EINVAL;
    if (hb->trace_ptr[0] != 0 || hb->profile_ptr[0] != 0 || hb->trace_ptr[B] != N || hb->profile_ptr[B] != hb->n_steps)
        return MP_EINVAL;
    for (int64_t b = 0; b < B; ++b)
        if (hb->trace_ptr[b + 1] < hb->trace_ptr[b] || hb->profile_ptr[b + 1] < hb->profile_ptr[b]) return MP_EINVAL;
    return MP_OK;
}

struct EventPool {
    std::mutex mu;
    std::vector<cudaEvent_t> ev;  // 2 per chunk: inputs landed, chunk planned
};

// The event pool of the current device, created on first use.
cudaError_t device_pool(EventPool** out) {
    static std::mutex mu;
    static std::map<int, EventPool*> pools;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    auto it = pools.find(dev);
    if (it == pools.end()) {
        EventPool* p = new EventPool;  // lives until exit, like the device context
        for (int i = 0; i < 2 * MP_HOST_PATH_MAX_CHUNKS; ++i) {
            cudaEvent_t x;
            e = cudaEventCreateWithFlags(&x, cudaEventDisableTiming);
            if (e != cudaSuccess) {
                for (cudaEvent_t y : p->ev) cudaEventDestroy(y);
                delete p;
                return e;
            }
            p->ev.push_back(x);
        }
        it = pools.emplace(dev, p).first;
    }
    *out = it->second;
    return cudaSuccess;
}

// The device address of a host array the GPU can reach directly (page-locked
// memory registered with CUDA, mapped into the device's address space);
// nullptr if it cannot.
template <typename T>
T* device_view(const T* host, int64_t len) {
    if (len <= 0) return nullptr;
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, host) != cudaSuccess) {
        cudaGetLastError();  // an unregistered pointer: not an error of the context
        return nullptr;
    }
    if (attr.type != cudaMemoryTypeHost || attr.devicePointer == nullptr) return nullptr;
    return static_cast<T*>(attr.devicePointer);
}

// chunks == 0: the fused kernels read the inputs from, and write the results
// to, the host buffers themselves over the CPU-GPU link; the device buffer
// only holds the planner's workspace.
mp_status direct_path(const mp_batch& hb, mp_fit_policy policy, const mp_host_results& out, void* device_buffer,
                      size_t device_bytes, void* compute_stream, void* copy_out_stream) {
    const int64_t B = hb.n_traces, N = hb.n_tensors, S = hb.n_steps;
    const size_t ws = mp::plan_workspace_bytes(hb);
    if (device_buffer == nullptr || reinterpret_cast<uintptr_t>(device_buffer) % mp::kAlign != 0) return MP_EINVAL;
    if (device_bytes < std::max<size_t>(ws, mp::kAlign)) return MP_ENOMEM;
    if (B == 0) return MP_OK;
    bool reachable = true;
    auto view = [&](auto* host, int64_t len) {
        auto* d = device_view(host, len);
        if (len > 0 && d == nullptr) reachable = false;
        return d;
    };
    mp_batch dev = hb;
    dev.trace_ptr = view(hb.trace_ptr, B + 1);
    dev.steps = view(hb.steps, B);
    dev.profile_ptr = view(hb.profile_ptr, B + 1);
    dev.alloc_step = view(hb.alloc_step, N);
    dev.free_step = view(hb.free_step, N);
    dev.size_bytes = view(hb.size_bytes, N);
    int64_t* profile = view(out.profile, S);
    int64_t* peak_lb = view(out.peak_lb, B);
    int64_t* offsets = view(out.offsets, N);
    int64_t* plan_peak = view(out.plan_peak, B);
    int32_t* verdict = view(out.verdict, B);
    int32_t* conflict = out.conflict != nullptr ? view(out.conflict, 2 * B) : nullptr;
    int32_t* status = view(out.trace_status, B);
    if (!reachable) return MP_EINVAL;  // some host array is not mapped into the device's address space
    cudaStream_t s_run = static_cast<cudaStream_t>(compute_stream);
    cudaStream_t s_out = static_cast<cudaStream_t>(copy_out_stream);
    cudaError_t e = mp::launch_plan_fused(dev, (int32_t)policy, profile, peak_lb, offsets, plan_peak, verdict,
                                          conflict, status, device_buffer, s_run);
    if (e == cudaSuccess && s_out != s_run) {
        EventPool* pool = nullptr;
        e = device_pool(&pool);
        if (e == cudaSuccess) {
            std::lock_guard<std::mutex> lock(pool->mu);
            e = cudaEventRecord(pool->ev[0], s_run);
            if (e == cudaSuccess) e = cudaStreamWaitEvent(s_out, pool->ev[0], 0);
        }
    }
    return e == cudaSuccess ? MP_OK : MP_ECUDA;
}

template <typename T>
T* at(void* base, size_t off) {
    return reinterpret_cast<T*>(static_cast<unsigned char*>(base) + off);
}

}  // namespace

extern "C" {

__attribute__((visibility("default"))) size_t mp_host_path_bytes(const mp_batch* host_batch, int32_t chunks) {
    if (check_host_batch(host_batch) != MP_OK || chunks < 0 || chunks > MP_HOST_PATH_MAX_CHUNKS) return 0;
    if (chunks == 0) return std::max<size_t>(mp::plan_workspace_bytes(*host_batch), mp::kAlign);
    const std::vector<int32_t> bounds = chunk_bounds(*host_batch, chunks);
    return host_path_layout(*host_batch, chunk_workspace_bytes(*host_batch, bounds)).total;
}

__attribute__((visibility("default"))) mp_status mp_plan_and_validate_host(
    const mp_batch* host_batch, mp_fit_policy policy, const mp_host_results* out, int32_t chunks,
    void* device_buffer, size_t device_bytes, void* copy_in_stream, void* compute_stream, void* copy_out_stream) {
    mp_status st = check_host_batch(host_batch);
    if (st != MP_OK) return st;
    if (policy != MP_FIT_FIRST && policy != MP_FIT_BEST) return MP_EINVAL;
    if (chunks < 0 || chunks > MP_HOST_PATH_MAX_CHUNKS || out == nullptr) return MP_EINVAL;
    const mp_batch& hb = *host_batch;
    const int64_t B = hb.n_traces, N = hb.n_tensors, S = hb.n_steps;
    auto ok = [](const void* p, int64_t len, size_t align) {
        return len <= 0 || (p != nullptr && reinterpret_cast<uintptr_t>(p) % align == 0);
    };
    if (!ok(out->profile, S, 8) || !ok(out->peak_lb, B, 8) || !ok(out->offsets, N, 8) || !ok(out->plan_peak, B, 8) ||
        !ok(out->verdict, B, 4) || !ok(out->trace_status, B, 4) ||
        (out->conflict != nullptr && reinterpret_cast<uintptr_t>(out->conflict) % 4 != 0))
        return MP_EINVAL;
    if (chunks == 0) return direct_path(hb, policy, *out, device_buffer, device_bytes, compute_stream, copy_out_stream);
    const std::vector<int32_t> bounds = chunk_bounds(hb, chunks);
    const HostPathLayout L = host_path_layout(hb, chunk_workspace_bytes(hb, bounds));
    if (device_buffer == nullptr || reinterpret_cast<uintptr_t>(device_buffer) % mp::kAlign != 0) return MP_EINVAL;
    if (device_bytes < L.total) return MP_ENOMEM;
    if (B == 0) return MP_OK;

    EventPool* pool = nullptr;
    if (device_pool(&pool) != cudaSuccess) return MP_ECUDA;
    std::lock_guard<std::mutex> lock(pool->mu);
    cudaStream_t s_in = static_cast<cudaStream_t>(copy_in_stream);
    cudaStream_t s_run = static_cast<cudaStream_t>(compute_stream);
    cudaStream_t s_out = static_cast<cudaStream_t>(copy_out_stream);
    void* d = device_buffer;
    const cudaMemcpyKind h2d = cudaMemcpyHostToDevice, d2h = cudaMemcpyDeviceToHost;
    cudaError_t e = cudaSuccess;
    auto copy = [&](void* dst, const void* src, size_t bytes, cudaMemcpyKind kind, cudaStream_t s) {
        if (e == cudaSuccess && bytes > 0) e = cudaMemcpyAsync(dst, src, bytes, kind, s);
    };
    // the per-trace arrays, whole, ahead of the first chunk: one copy when the
    // host keeps trace_ptr, profile_ptr and steps in this order with fewer
    // than 16 bytes between them (those bytes are read, never written)
    mp_batch dev = hb;
    {
        const size_t tp = (size_t)(B + 1) * 8, st = (size_t)B * 4;
        const char* htp = reinterpret_cast<const char*>(hb.trace_ptr);
        const char* hpp = reinterpret_cast<const char*>(hb.profile_ptr);
        const char* hst = reinterpret_cast<const char*>(hb.steps);
        char* dpt = at<char>(d, L.pertrace);
        if (hpp >= htp + tp && hpp < htp + tp + 16 && hst >= hpp + tp && hst < hpp + tp + 16) {
            dev.trace_ptr = reinterpret_cast<int64_t*>(dpt);
            dev.profile_ptr = reinterpret_cast<int64_t*>(dpt + (hpp - htp));
            dev.steps = reinterpret_cast<int32_t*>(dpt + (hst - htp));
            copy(dpt, htp, (size_t)(hst - htp) + st, h2d, s_in);
        } else {
            dev.trace_ptr = reinterpret_cast<int64_t*>(dpt);
            dev.profile_ptr = reinterpret_cast<int64_t*>(dpt + tp);
            dev.steps = reinterpret_cast<int32_t*>(dpt + 2 * tp);
            copy(dpt, hb.trace_ptr, tp, h2d, s_in);
            copy(dpt + tp, hb.profile_ptr, tp, h2d, s_in);
            copy(dpt + 2 * tp, hb.steps, st, h2d, s_in);
        }
    }
    dev.alloc_step = at<int32_t>(d, L.alloc);
    dev.free_step = at<int32_t>(d, L.free_);
    dev.size_bytes = at<int64_t>(d, L.size);
    const size_t nchunks = bounds.size() - 1;
    for (size_t k = 0; k < nchunks && e == cudaSuccess; ++k) {
        const int32_t b0 = bounds[k], b1 = bounds[k + 1];
        const int64_t lo = hb.trace_ptr[b0], hi = hb.trace_ptr[b1];
        const int64_t plo = hb.profile_ptr[b0], phi = hb.profile_ptr[b1];
        cudaEvent_t landed = pool->ev[2 * k], planned = pool->ev[2 * k + 1];
        copy(at<int32_t>(d, L.alloc) + lo, hb.alloc_step + lo, (size_t)(hi - lo) * 4, h2d, s_in);
        copy(at<int32_t>(d, L.free_) + lo, hb.free_step + lo, (size_t)(hi - lo) * 4, h2d, s_in);
        copy(at<int64_t>(d, L.size) + lo, hb.size_bytes + lo, (size_t)(hi - lo) * 8, h2d, s_in);
        if (e == cudaSuccess) e = cudaEventRecord(landed, s_in);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s_run, landed, 0);
        mp_batch c = dev;
        c.n_traces = b1 - b0;
        c.trace_ptr += b0;
        c.steps += b0;
        c.profile_ptr += b0;
        if (e == cudaSuccess)
            e = mp::launch_plan_fused(c, (int32_t)policy, at<int64_t>(d, L.profile), at<int64_t>(d, L.peak_lb) + b0,
                                      at<int64_t>(d, L.offsets), at<int64_t>(d, L.plan_peak) + b0,
                                      at<int32_t>(d, L.verdict) + b0, at<int32_t>(d, L.conflict) + 2 * b0,
                                      at<int32_t>(d, L.status) + b0, at<void>(d, L.workspace), s_run);
        if (e == cudaSuccess) e = cudaEventRecord(planned, s_run);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s_out, planned, 0);
        copy(out->profile + plo, at<int64_t>(d, L.profile) + plo, (size_t)(phi - plo) * 8, d2h, s_out);
        copy(out->offsets + lo, at<int64_t>(d, L.offsets) + lo, (size_t)(hi - lo) * 8, d2h, s_out);
    }
    // the per-trace results, after the last chunk (the copy-out stream has
    // waited for every chunk's planning by now): one copy when the host
    // arrays are adjacent in the device block's order, with nothing between
    // them (a copy back writes every byte it spans)
    auto bytes_at = [](const void* p) { return reinterpret_cast<const char*>(p); };
    const bool packed_out = out->conflict != nullptr && bytes_at(out->plan_peak) == bytes_at(out->peak_lb) + B * 8 &&
                            bytes_at(out->verdict) == bytes_at(out->plan_peak) + B * 8 &&
                            bytes_at(out->conflict) == bytes_at(out->verdict) + B * 4 &&
                            bytes_at(out->trace_status) == bytes_at(out->conflict) + B * 8;
    if (packed_out) {
        copy(out->peak_lb, at<int64_t>(d, L.results), (size_t)B * 32, d2h, s_out);
    } else {
        copy(out->peak_lb, at<int64_t>(d, L.peak_lb), (size_t)B * 8, d2h, s_out);
        copy(out->plan_peak, at<int64_t>(d, L.plan_peak), (size_t)B * 8, d2h, s_out);
        copy(out->verdict, at<int32_t>(d, L.verdict), (size_t)B * 4, d2h, s_out);
        if (out->conflict != nullptr) copy(out->conflict, at<int32_t>(d, L.conflict), (size_t)B * 8, d2h, s_out);
        copy(out->trace_status, at<int32_t>(d, L.status), (size_t)B * 4, d2h, s_out);
    }
    return e == cudaSuccess ? MP_OK : MP_ECUDA;
}

}  // extern "C"
