// launch.h -- internal launch interface between the C ABI (abi.cu) and the
// kernel translation units.  Not part of the public header.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "memplan.h"

namespace mp {

constexpr int kProfileThreads = 128;  // one CTA per trace
constexpr int kValidateThreads = 128;
constexpr int kPeakThreads = 256;
constexpr int kBumpThreads = 128;
constexpr int kOptThreads = 128;
constexpr int kReplayThreads = 256;
constexpr int kBreadthThreads = 128;
constexpr int kPlanThreadsSmem = 128;    // one CTA per trace, data in shared memory
constexpr int kPlanThreadsGlobal = 1024; // one CTA per trace, data in the workspace
constexpr int kPlanThreadsWide = 512;    // the 64-bit launch: deferred traces, CTA tier included

// Largest dynamic shared memory a kernel of this library requests per CTA
// (sm_103a allows 227 KB); above it a kernel keeps its data in the workspace.
constexpr size_t kSmemCeiling = 200 * 1024;
constexpr size_t kProfileSmemLimit = kSmemCeiling;
constexpr size_t kValidateSmemLimit = kSmemCeiling;
constexpr size_t kPlanSmemLimit = kSmemCeiling;

// Raises the kernel's dynamic shared memory ceiling once per device (to
// kSmemCeiling, or to `bytes` for a kernel that asks for more).
cudaError_t set_smem_limit(const void* func, size_t bytes);

// CTAs of `func` (threads, dynamic shared memory smem) the current device holds
// at once: SM count x resident CTAs per SM (at least 1); cached per device.
cudaError_t max_resident_ctas(const void* func, int threads, size_t smem, int* ctas);

// Alignment of every workspace slice.
constexpr size_t kAlign = 256;
__host__ __device__ constexpr size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Workspace sizes saturate at SIZE_MAX instead of wrapping: a batch whose
// need does not fit in size_t can then never pass a workspace-size check.
inline size_t mul_sat(size_t a, size_t b) {
    size_t r;
    return __builtin_mul_overflow(a, b, &r) ? SIZE_MAX : r;
}
inline size_t add_sat(size_t a, size_t b) {
    size_t r;
    return __builtin_add_overflow(a, b, &r) ? SIZE_MAX : r;
}

cudaError_t launch_live_profile(const mp_batch& bt, int64_t* profile, int64_t* peak_lb, int32_t* status,
                                cudaStream_t stream);

size_t validate_workspace_bytes(const mp_batch& bt);
cudaError_t launch_validate(const mp_batch& bt, const int64_t* offsets, int32_t* verdict, int32_t* conflict,
                            int32_t* status, void* workspace, cudaStream_t stream);

size_t bump_workspace_bytes(const mp_batch& bt);
cudaError_t launch_bump(const mp_batch& bt, int64_t* offsets, int64_t* plan_peak, int32_t* status, void* workspace,
                        cudaStream_t stream);

size_t optimal_workspace_bytes(const mp_batch& bt);
cudaError_t launch_optimal(const mp_batch& bt, int64_t* offsets, int64_t* opt_peak, int32_t* status, void* workspace,
                           cudaStream_t stream);

size_t replay_workspace_bytes(const mp_batch& bt);
cudaError_t launch_slab_layout(const mp_batch& bt, const int64_t* plan_peak, const int32_t* trace_status,
                               const int64_t* offsets, int64_t* slab_base, int64_t* tensor_addr, cudaStream_t stream);
cudaError_t launch_replay(const mp_batch& bt, const int64_t* offsets, const int64_t* slab_base, unsigned char* slab,
                          int64_t slab_bytes, int32_t* ok, int32_t* first_bad, int32_t* status, void* workspace,
                          cudaStream_t stream);

size_t breadth_workspace_bytes(const mp_batch& bt);
cudaError_t launch_breadth(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak, int32_t* status,
                           void* workspace, cudaStream_t stream);

cudaError_t launch_peak(const mp_batch& bt, const int64_t* offsets, int64_t* plan_peak, int32_t* status,
                        cudaStream_t stream);

// Batches of at most kGridMaxTraces traces whose max_tensors exceeds
// kGridMinTensors -- a few large traces -- are planned by the grid-wide
// dataflow (grid.cu); every other batch by one CTA per trace (plan.cu).
constexpr int32_t kGridMinTensors = 1024;
constexpr int32_t kGridMaxTraces = 32;
bool grid_path(const mp_batch& bt);
size_t grid_workspace_bytes(const mp_batch& bt);
// hold >= 0 is a test hook: the tensor with that slot id (trace * max_tensors
// + alloc-order position) is never queued, so the bounded wait runs out.
cudaError_t launch_grid_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                             int32_t* status, void* workspace, int32_t hold, cudaStream_t stream);
cudaError_t launch_grid_fused(const mp_batch& bt, int32_t policy, int64_t* profile, int64_t* peak_lb,
                              int64_t* offsets, int64_t* plan_peak, int32_t* verdict, int32_t* conflict,
                              int32_t* status, void* workspace, cudaStream_t stream);

// Largest max_tensors mp_plan_greedy_by_size accepts (per-trace counts are
// packed with a 2-bit tier tag into one int32).
constexpr int32_t kPlanMaxTensors = (1 << 28) - 1;
size_t plan_workspace_bytes(const mp_batch& bt);
cudaError_t launch_plan(const mp_batch& bt, int32_t policy, int64_t* offsets, int64_t* plan_peak,
                        int32_t* status, void* workspace, cudaStream_t stream);
cudaError_t launch_plan_fused(const mp_batch& bt, int32_t policy, int64_t* profile, int64_t* peak_lb,
                              int64_t* offsets, int64_t* plan_peak, int32_t* verdict, int32_t* conflict,
                              int32_t* status, void* workspace, cudaStream_t stream);

}  // namespace mp
