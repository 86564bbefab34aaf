// plan_static.cu -- mp_plan_greedy_by_size_static: greedy_by_size with its
// scratch in a fixed device array owned by this library, for callers that
// cannot allocate device memory.
//
// Who needs it: a caller on a latency-critical serving path that must not
// call cudaMalloc (which can block on the driver's allocator lock and
// synchronise the device -- the very contention this planner exists to take
// out of inference), or code running inside a framework that owns the
// device allocator and gives its plug-ins no way to request scratch.  Such a
// caller still owns and passes every input and output buffer; only the
// planner's scratch moves into the library.
//
// The scratch is one file-scope __device__ array of kPlanStaticScratchBytes
// (MP_PLAN_STATIC_SCRATCH_BYTES), created when a device loads this library and
// held by every such device until the process exits.  Host code cannot use
// the array's name as a device address, so the first call on each device
// (made with that device current) looks the address up once with
// cudaGetSymbolAddress and caches it; make that first call before any stream
// capture.  The cached address outlives a cudaDeviceReset, after which the
// module may be loaded again elsewhere, so the entry point must not be used on
// a device after it has been reset.  Every call shares the one array: two calls whose kernels overlap
// on a GPU (different streams, or different host threads) race on it and
// must be serialised by the caller.  The planner writes every scratch byte it
// later reads, so nothing has to be cleared between calls.
#include <mutex>

#include "launch.h"
#include "memplan.h"

namespace {

constexpr size_t kPlanStaticScratchBytes = MP_PLAN_STATIC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_plan_scratch[kPlanStaticScratchBytes];

std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_plan_scratch on the current device, looked up once.
cudaError_t scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_scratch_ptr[dev] == nullptr) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_plan_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

template <typename T>
bool aligned(const T* p) {
    return (reinterpret_cast<uintptr_t>(p) % alignof(T)) == 0;
}

template <typename T>
bool array_ok(const T* p, int64_t len) {
    if (len <= 0) return p == nullptr || aligned(p);
    return p != nullptr && aligned(p);
}

}  // namespace

extern "C" {

__attribute__((visibility("default"))) mp_status mp_plan_greedy_by_size_static(
    const mp_batch* batch, mp_fit_policy policy, int64_t* offsets, int64_t* plan_peak, int32_t* trace_status,
    void* stream) {
    if (batch == nullptr) return MP_EINVAL;
    const mp_batch& b = *batch;
    if (b.n_traces < 0 || b.max_tensors < 0 || b.max_steps < 0 || b.reserved0 != 0 || b.n_tensors < 0 ||
        b.n_steps < 0 || b.max_tensors > mp::kPlanMaxTensors)
        return MP_EINVAL;
    const int64_t B = b.n_traces;
    if (!array_ok(b.trace_ptr, B ? B + 1 : 0) || !array_ok(b.steps, B) || !array_ok(b.alloc_step, b.n_tensors) ||
        !array_ok(b.free_step, b.n_tensors) || !array_ok(b.size_bytes, b.n_tensors))
        return MP_EINVAL;
    if (policy != MP_FIT_FIRST && policy != MP_FIT_BEST) return MP_EINVAL;
    if (!array_ok(offsets, b.n_tensors) || !array_ok(plan_peak, B) || !array_ok(trace_status, B))
        return MP_EINVAL;
    const size_t need = mp::plan_workspace_bytes(b);
    if (need > kPlanStaticScratchBytes) return MP_ENOMEM;  // batch too large for the fixed scratch
    void* scratch = nullptr;
    if (scratch_address(&scratch) != cudaSuccess) return MP_ECUDA;
    const cudaError_t e = mp::launch_plan(b, (int32_t)policy, offsets, plan_peak, trace_status, scratch,
                                          static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? MP_OK : MP_ECUDA;
}

}  // extern "C"
