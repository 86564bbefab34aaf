// abi.cu -- extern "C" entry points of libmemplan.so (declared in memplan.h).
//
// Host-side argument checks, then one kernel launch per call on the caller's
// stream.  No entry point allocates device memory or synchronises.
#include <algorithm>
#include <cstdint>
#include <map>
#include <mutex>
#include <set>
#include <tuple>
#include <utility>

#include "launch.h"
#include "memplan.h"

namespace mp {

cudaError_t set_smem_limit(const void* func, size_t bytes) {
    if (bytes <= 48 * 1024) return cudaSuccess;
    static std::mutex mu;
    static std::set<std::pair<int, const void*>> done;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    if (done.count({dev, func})) return cudaSuccess;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)std::max(bytes, kSmemCeiling));
    if (e == cudaSuccess) done.insert({dev, func});
    return e;
}

cudaError_t max_resident_ctas(const void* func, int threads, size_t smem, int* ctas) {
    static std::mutex mu;
    static std::map<std::tuple<int, const void*, int, size_t>, int> cache;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const auto key = std::make_tuple(dev, func, threads, smem);
    std::lock_guard<std::mutex> lock(mu);
    auto it = cache.find(key);
    if (it == cache.end()) {
        int sms = 0, per_sm = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, func, threads, smem);
        if (e != cudaSuccess) return e;
        it = cache.emplace(key, std::max(1, sms * per_sm)).first;
    }
    *ctas = it->second;
    return cudaSuccess;
}

}  // namespace mp

namespace {

template <typename T>
bool aligned(const T* p) {
    return (reinterpret_cast<uintptr_t>(p) % alignof(T)) == 0;
}

// Non-null (when the array is non-empty) and naturally aligned.
template <typename T>
bool array_ok(const T* p, int64_t len) {
    if (len <= 0) return p == nullptr || aligned(p);
    return p != nullptr && aligned(p);
}

mp_status check_batch(const mp_batch* bt, bool need_profile) {
    if (bt == nullptr) return MP_EINVAL;
    if (bt->n_traces < 0 || bt->max_tensors < 0 || bt->max_steps < 0 || bt->reserved0 != 0 ||
        bt->n_tensors < 0 || bt->n_steps < 0)
        return MP_EINVAL;
    const int64_t B = bt->n_traces;
    if (!array_ok(bt->trace_ptr, B ? B + 1 : 0) || !array_ok(bt->steps, B)) return MP_EINVAL;
    if (need_profile && !array_ok(bt->profile_ptr, B ? B + 1 : 0)) return MP_EINVAL;
    if (!array_ok(bt->alloc_step, bt->n_tensors) || !array_ok(bt->free_step, bt->n_tensors) ||
        !array_ok(bt->size_bytes, bt->n_tensors))
        return MP_EINVAL;
    return MP_OK;
}

mp_status check_workspace(size_t need, const void* ws, size_t ws_bytes) {
    if (need == 0) return MP_OK;
    if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) % mp::kAlign) != 0) return MP_EINVAL;
    if (ws_bytes < need) return MP_ENOMEM;
    return MP_OK;
}

mp_status from_cuda(cudaError_t e) { return e == cudaSuccess ? MP_OK : MP_ECUDA; }

}  // namespace

extern "C" {

__attribute__((visibility("default"))) int32_t mp_abi_version(void) { return 2; }

__attribute__((visibility("default"))) const char* mp_status_string(mp_status status) {
    switch (status) {
        case MP_OK: return "MP_OK";
        case MP_EINVAL: return "MP_EINVAL";
        case MP_EOVERFLOW: return "MP_EOVERFLOW";
        case MP_ECUDA: return "MP_ECUDA";
        case MP_ETIMEOUT: return "MP_ETIMEOUT";
        case MP_ENOMEM: return "MP_ENOMEM";
        case MP_EINTERNAL: return "MP_EINTERNAL";
    }
    return "MP_UNKNOWN";
}

__attribute__((visibility("default"))) mp_status mp_live_profile(const mp_batch* batch, int64_t* profile,
                                                                 int64_t* peak_lb, int32_t* trace_status,
                                                                 void* stream) {
    mp_status st = check_batch(batch, true);
    if (st != MP_OK) return st;
    if (!array_ok(profile, batch->n_steps) || !array_ok(peak_lb, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    return from_cuda(mp::launch_live_profile(*batch, profile, peak_lb, trace_status,
                                             static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) size_t mp_plan_workspace_bytes(const mp_batch* batch) {
    if (check_batch(batch, false) != MP_OK) return 0;
    return mp::plan_workspace_bytes(*batch);
}

__attribute__((visibility("default"))) mp_status mp_plan_greedy_by_size(
    const mp_batch* batch, mp_fit_policy policy, int64_t* offsets, int64_t* plan_peak, int32_t* trace_status,
    void* workspace, size_t workspace_bytes, void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (policy != MP_FIT_FIRST && policy != MP_FIT_BEST) return MP_EINVAL;
    if (batch->max_tensors > mp::kPlanMaxTensors) return MP_EINVAL;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(plan_peak, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    st = check_workspace(mp::plan_workspace_bytes(*batch), workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_plan(*batch, (int32_t)policy, offsets, plan_peak, trace_status, workspace,
                                     static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) mp_status mp_plan_and_validate(
    const mp_batch* batch, mp_fit_policy policy, int64_t* profile, int64_t* peak_lb, int64_t* offsets,
    int64_t* plan_peak, int32_t* verdict, int32_t* conflict, int32_t* trace_status, void* workspace,
    size_t workspace_bytes, void* stream) {
    const bool want_profile = profile != nullptr || peak_lb != nullptr;
    mp_status st = check_batch(batch, want_profile);
    if (st != MP_OK) return st;
    if (policy != MP_FIT_FIRST && policy != MP_FIT_BEST) return MP_EINVAL;
    if (batch->max_tensors > mp::kPlanMaxTensors) return MP_EINVAL;
    if (want_profile && (!array_ok(profile, batch->n_steps) || !array_ok(peak_lb, batch->n_traces)))
        return MP_EINVAL;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(plan_peak, batch->n_traces) ||
        !array_ok(verdict, batch->n_traces) || !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    if (conflict != nullptr && !aligned(conflict)) return MP_EINVAL;
    st = check_workspace(mp::plan_workspace_bytes(*batch), workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_plan_fused(*batch, (int32_t)policy, want_profile ? profile : nullptr,
                                           want_profile ? peak_lb : nullptr, offsets, plan_peak, verdict, conflict,
                                           trace_status, workspace, static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) size_t mp_validate_workspace_bytes(const mp_batch* batch) {
    if (check_batch(batch, false) != MP_OK) return 0;
    return mp::validate_workspace_bytes(*batch);
}

__attribute__((visibility("default"))) mp_status mp_validate_plan(const mp_batch* batch, const int64_t* offsets,
                                                                  int32_t* verdict, int32_t* conflict,
                                                                  int32_t* trace_status, void* workspace,
                                                                  size_t workspace_bytes, void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(verdict, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    if (conflict != nullptr && !aligned(conflict)) return MP_EINVAL;
    st = check_workspace(mp::validate_workspace_bytes(*batch), workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_validate(*batch, offsets, verdict, conflict, trace_status, workspace,
                                         static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) size_t mp_bump_workspace_bytes(const mp_batch* batch) {
    if (check_batch(batch, false) != MP_OK) return 0;
    return mp::bump_workspace_bytes(*batch);
}

__attribute__((visibility("default"))) mp_status mp_plan_bump(const mp_batch* batch, int64_t* offsets,
                                                              int64_t* plan_peak, int32_t* trace_status,
                                                              void* workspace, size_t workspace_bytes, void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(plan_peak, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    st = check_workspace(mp::bump_workspace_bytes(*batch), workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_bump(*batch, offsets, plan_peak, trace_status, workspace,
                                     static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) size_t mp_optimal_workspace_bytes(const mp_batch* batch) {
    if (check_batch(batch, false) != MP_OK) return 0;
    return mp::optimal_workspace_bytes(*batch);
}

__attribute__((visibility("default"))) mp_status mp_plan_optimal(const mp_batch* batch, int64_t* offsets,
                                                                 int64_t* opt_peak, int32_t* trace_status,
                                                                 void* workspace, size_t workspace_bytes,
                                                                 void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(opt_peak, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    const size_t need = mp::optimal_workspace_bytes(*batch);
    if (need > 0 && (int64_t)need / (int64_t)sizeof(longlong2) > INT32_MAX) return MP_EINVAL;  // grid too large
    st = check_workspace(need, workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_optimal(*batch, offsets, opt_peak, trace_status, workspace,
                                        static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) mp_status mp_slab_layout(const mp_batch* batch, const int64_t* plan_peak,
                                                                const int32_t* trace_status, const int64_t* offsets,
                                                                int64_t* slab_base, int64_t* tensor_addr,
                                                                void* stream) {
    if (batch == nullptr || batch->n_traces < 0 || batch->n_tensors < 0) return MP_EINVAL;
    const int64_t B = batch->n_traces;
    if (!array_ok(plan_peak, B) || !array_ok(slab_base, B + 1)) return MP_EINVAL;
    if (trace_status != nullptr && !aligned(trace_status)) return MP_EINVAL;
    if (tensor_addr != nullptr) {  // the per-tensor views need the CSR and the offsets
        if (!array_ok(batch->trace_ptr, B ? B + 1 : 0) || !array_ok(offsets, batch->n_tensors) ||
            !array_ok(tensor_addr, batch->n_tensors))
            return MP_EINVAL;
    }
    return from_cuda(mp::launch_slab_layout(*batch, plan_peak, trace_status, offsets, slab_base, tensor_addr,
                                            static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) size_t mp_replay_workspace_bytes(const mp_batch* batch) {
    if (check_batch(batch, false) != MP_OK) return 0;
    return mp::replay_workspace_bytes(*batch);
}

__attribute__((visibility("default"))) mp_status mp_replay_plan(const mp_batch* batch, const int64_t* offsets,
                                                                const int64_t* slab_base, void* slab,
                                                                int64_t slab_bytes, int32_t* ok, int32_t* first_bad,
                                                                int32_t* trace_status, void* workspace,
                                                                size_t workspace_bytes, void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(slab_base, batch->n_traces ? batch->n_traces + 1 : 0) ||
        !array_ok(ok, batch->n_traces) || !array_ok(first_bad, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces) || slab_bytes < 0 ||
        !array_ok(static_cast<const int32_t*>(slab), slab_bytes > 0 ? 1 : 0))
        return MP_EINVAL;
    st = check_workspace(mp::replay_workspace_bytes(*batch), workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_replay(*batch, offsets, slab_base, static_cast<unsigned char*>(slab), slab_bytes, ok,
                                       first_bad, trace_status, workspace, static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) size_t mp_breadth_workspace_bytes(const mp_batch* batch) {
    if (check_batch(batch, false) != MP_OK) return 0;
    return mp::breadth_workspace_bytes(*batch);
}

__attribute__((visibility("default"))) mp_status mp_plan_greedy_by_breadth(
    const mp_batch* batch, mp_fit_policy policy, int64_t* offsets, int64_t* plan_peak, int32_t* trace_status,
    void* workspace, size_t workspace_bytes, void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (policy != MP_FIT_FIRST && policy != MP_FIT_BEST) return MP_EINVAL;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(plan_peak, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    st = check_workspace(mp::breadth_workspace_bytes(*batch), workspace, workspace_bytes);
    if (st != MP_OK) return st;
    return from_cuda(mp::launch_breadth(*batch, policy, offsets, plan_peak, trace_status, workspace,
                                        static_cast<cudaStream_t>(stream)));
}

__attribute__((visibility("default"))) mp_status mp_peak(const mp_batch* batch, const int64_t* offsets,
                                                         int64_t* plan_peak, int32_t* trace_status,
                                                         void* stream) {
    mp_status st = check_batch(batch, false);
    if (st != MP_OK) return st;
    if (!array_ok(offsets, batch->n_tensors) || !array_ok(plan_peak, batch->n_traces) ||
        !array_ok(trace_status, batch->n_traces))
        return MP_EINVAL;
    return from_cuda(mp::launch_peak(*batch, offsets, plan_peak, trace_status, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
