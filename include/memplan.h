/*
 * memplan.h -- C ABI of the GB300 memory-planning library (libmemplan.so).
 *
 * The library builds and checks static memory plans for batches of
 * allocation traces, the static-analysis half of MemoMalloc ("Memory Planning
 * for Deep Neural Networks", arXiv 2203.00448).  A trace lists the
 * intermediate tensors of one forward pass; tensor i has a lifetime
 * [alloc_step_i, free_step_i) over op steps (half-open) and a size in bytes.
 * A plan gives every tensor an offset into one slab (Sec. 3.3,
 * prim::AllocateSlab[total_size] / prim::AllocateTensor[size, offset]).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All array pointers inside mp_batch and all output pointers are DEVICE
 *   pointers (cudaMalloc'd or managed), owned by the caller; the library never
 *   frees or retains them.  The mp_batch struct itself is read on the host
 *   during the call and may be discarded afterwards.
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   Every call only enqueues work on that stream and returns without
 *   synchronising; outputs are valid once the stream reaches that point.
 * - The return value reports host-side problems only: MP_EINVAL for a NULL
 *   or misaligned pointer, a negative count or a too-small workspace;
 *   MP_ECUDA when a launch fails.  After MP_EINVAL or MP_ENOMEM nothing was
 *   enqueued; after MP_ECUDA (a failed launch, copy or event call) part of a
 *   call's work may already be on its streams.
 * - Per-trace data errors are written to trace_status[b] on the device:
 *     MP_EINVAL    bad CSR range (trace_ptr not non-decreasing, beyond
 *                  n_tensors, or more than max_tensors tensors), T_b < 0 or
 *                  T_b > max_steps, a tensor with alloc < 0, free <= alloc,
 *                  free > T_b or size <= 0, or (where offsets are inputs)
 *                  offset < 0;
 *     MP_EOVERFLOW the sizes of the trace sum past INT64_MAX, or (where
 *                  offsets are inputs) some offset + size does;
 *   EINVAL takes precedence.  Outputs of a failed trace are unspecified but
 *   nothing outside that trace's own output range is written.
 * - Tensor ids are local indices within their trace.  A trace with no
 *   tensors is valid; its profile is all zero and both peaks are 0.
 * - All arithmetic is integer (int64 bytes/offsets, int32 steps/ids), so
 *   results are bit-identical to the plain definitions, whatever the launch
 *   configuration.
 */
#ifndef MEMPLAN_H
#define MEMPLAN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum mp_status {
    MP_OK = 0,
    MP_EINVAL = 1,
    MP_EOVERFLOW = 2,
    MP_ECUDA = 3,
    MP_ETIMEOUT = 4, /* per-trace only: a wait of the planner on another warp or
                        CTA gave up after its bound (see mp_plan_greedy_by_size);
                        that trace's outputs are unspecified */
    MP_ENOMEM = 5,   /* workspace smaller than the matching *_workspace_bytes */
    MP_EINTERNAL = 6 /* per-trace only: a kernel found an inconsistency in its own
                        state (a library defect); that trace's outputs are unspecified */
} mp_status;

/* Fit criterion of greedy_by_size.  Sec. 2.3 describes a best-fit criterion;
 * first fit is the lowest feasible offset.  Both are exact. */
typedef enum mp_fit_policy { MP_FIT_FIRST = 0, MP_FIT_BEST = 1 } mp_fit_policy;

/* A batch of B traces as a structure of arrays with CSR offsets.
 * Host scalars (read on the host, used to size launches and workspace):
 *   n_traces     B >= 0
 *   max_tensors  upper bound on N_b = trace_ptr[b+1] - trace_ptr[b]
 *   max_steps    upper bound on T_b
 *   n_tensors    length of alloc_step / free_step / size_bytes (= trace_ptr[B])
 *   n_steps      length of the profile output (= profile_ptr[B])
 * A trace breaking a declared bound is rejected with MP_EINVAL in
 * trace_status; it never causes an access outside the arrays.
 * Device arrays:
 *   trace_ptr    int64[B+1]  tensors of trace b: [trace_ptr[b], trace_ptr[b+1])
 *   steps        int32[B]    T_b, number of op steps of trace b
 *   profile_ptr  int64[B+1]  profile of trace b: [profile_ptr[b], +T_b);
 *                            only mp_live_profile reads it (may be NULL elsewhere)
 *   alloc_step   int32[n_tensors]  first live step
 *   free_step    int32[n_tensors]  first step no longer live (exclusive)
 *   size_bytes   int64[n_tensors]  size, >= 1
 * int64 arrays must be 8-byte aligned, int32 arrays 4-byte aligned. */
typedef struct mp_batch {
    int32_t n_traces;
    int32_t max_tensors;
    int32_t max_steps;
    int32_t reserved0; /* must be 0 */
    int64_t n_tensors;
    int64_t n_steps;
    const int64_t *trace_ptr;
    const int32_t *steps;
    const int64_t *profile_ptr;
    const int32_t *alloc_step;
    const int32_t *free_step;
    const int64_t *size_bytes;
} mp_batch;

/* Live-bytes profile and its peak (stage 1).
 * profile[profile_ptr[b] + t] = sum of size_i over tensors with
 *   alloc_i <= t < free_i, for 0 <= t < T_b                      int64[n_steps]
 * peak_lb[b] = max_t profile (0 when T_b = 0): every feasible total_mem of
 *   Eq. 2.1 is at least this, because the tensors live at one step must all
 *   fit side by side (Sec. 1 and Sec. 2.3).                        int64[B]
 * trace_status[b]                                                   int32[B]
 * Needs no workspace (the profile output doubles as the difference array). */
mp_status mp_live_profile(const mp_batch *batch, int64_t *profile, int64_t *peak_lb,
                          int32_t *trace_status, void *stream);

/* Bytes of device workspace mp_plan_greedy_by_size needs for this batch
 * (depends on the host scalars only).  0 means none; SIZE_MAX means the need
 * does not fit in size_t (every call on such a batch returns MP_ENOMEM).
 * Every *_workspace_bytes function below follows the same rule. */
size_t mp_plan_workspace_bytes(const mp_batch *batch);

/* greedy_by_size offset assignment (stage 2; Sec. 2.3, default strategy of
 * Sec. 3.2).  Tensors are taken in priority order -- size descending, then
 * alloc_step ascending, then id ascending -- and each is given, among the
 * already placed tensors whose lifetimes overlap its own, the first gap
 * (MP_FIT_FIRST: the lowest offset where it fits) or the smallest gap that
 * fits, lowest on ties (MP_FIT_BEST), gaps being measured against the running
 * maximum end in address order; if no gap fits it goes above them all.
 * offsets[trace_ptr[b] + i]   int64[n_tensors]
 * plan_peak[b] = max_i offset_i + size_i, the plan's total_mem   int64[B]
 * trace_status[b]                                               int32[B]
 * max_tensors must be below 2^28 (MP_EINVAL otherwise).
 * workspace: device memory of at least mp_plan_workspace_bytes(batch) bytes,
 * 256-byte aligned, owned by the caller, not used concurrently by another
 * call.  Its contents need not be initialised. */
mp_status mp_plan_greedy_by_size(const mp_batch *batch, mp_fit_policy policy, int64_t *offsets,
                                 int64_t *plan_peak, int32_t *trace_status, void *workspace,
                                 size_t workspace_bytes, void *stream);

/* Size of the fixed device scratch array behind mp_plan_greedy_by_size_static. */
#define MP_PLAN_STATIC_SCRATCH_BYTES ((size_t)16 << 20)

/* greedy_by_size without any device allocation by anyone: the same planner
 * and results as mp_plan_greedy_by_size, but its scratch is a 16 MiB array
 * that lives inside this library (a file-scope __device__ array), so the
 * caller passes no workspace.  The paper has no counterpart; this exists for
 * callers that may not allocate device memory -- a latency-critical serving
 * path that must not take the allocator's lock, or a plug-in whose host
 * framework owns the device allocator.  The caller still owns every input
 * and output buffer.
 * Limits and rules:
 * - a batch whose mp_plan_workspace_bytes exceeds MP_PLAN_STATIC_SCRATCH_BYTES
 *   is rejected with MP_ENOMEM before anything is enqueued;
 * - the first call on each device (with that device current) looks up the
 *   array's device address once; make that first call before any stream
 *   capture;
 * - all calls share the one array: calls whose kernels overlap on a GPU race
 *   and must be serialised by the caller; the planner writes every scratch
 *   byte before reading it, so nothing needs clearing between calls;
 * - the array occupies device memory on every device that loads this library
 *   until the process exits;
 * - the looked-up address is kept for the life of the process: after
 *   cudaDeviceReset on a device this entry point must not be called on that
 *   device again (the array may then live at another address).
 * Other arguments and return codes as for mp_plan_greedy_by_size. */
mp_status mp_plan_greedy_by_size_static(const mp_batch *batch, mp_fit_policy policy, int64_t *offsets,
                                        int64_t *plan_peak, int32_t *trace_status, void *stream);

/* The whole path in one pass: each trace is read once and the live profile
 * (stage 1), the greedy_by_size plan (stage 2) and the validation of that
 * plan (stage 3) are all computed from it, for batches planned and validated
 * in one call.  Results are identical to mp_live_profile, then
 * mp_plan_greedy_by_size, then mp_validate_plan on its offsets; the
 * validation is a separate pass over the trace in alloc-step order that
 * checks every lifetime-overlapping pair of the plan just made.
 * profile / peak_lb: as for mp_live_profile; pass both NULL to skip the
 * profile (profile_ptr is then not read).  offsets, plan_peak: as for
 * mp_plan_greedy_by_size.  verdict, conflict (nullable): as for
 * mp_validate_plan.  One trace_status per trace covers all outputs.
 * workspace: at least mp_plan_workspace_bytes(batch) bytes. */
mp_status mp_plan_and_validate(const mp_batch *batch, mp_fit_policy policy, int64_t *profile, int64_t *peak_lb,
                               int64_t *offsets, int64_t *plan_peak, int32_t *verdict, int32_t *conflict,
                               int32_t *trace_status, void *workspace, size_t workspace_bytes, void *stream);

/* Host buffers receiving the results of mp_plan_and_validate_host; the same
 * arrays, sizes and meaning as the device outputs of mp_plan_and_validate.
 * conflict may be NULL. */
typedef struct mp_host_results {
    int64_t *profile;      /* int64[n_steps] */
    int64_t *peak_lb;      /* int64[B] */
    int64_t *offsets;      /* int64[n_tensors] */
    int64_t *plan_peak;    /* int64[B] */
    int32_t *verdict;      /* int32[B] */
    int32_t *conflict;     /* int32[2B], nullable */
    int32_t *trace_status; /* int32[B] */
} mp_host_results;

/* Most chunks mp_plan_and_validate_host cuts a batch into. */
#define MP_HOST_PATH_MAX_CHUNKS 64

/* Bytes of device memory mp_plan_and_validate_host needs for this host batch
 * cut into `chunks` pieces (inputs, outputs and planner workspace); 0 if the
 * batch or chunk count is rejected, SIZE_MAX if the need does not fit in
 * size_t. */
size_t mp_host_path_bytes(const mp_batch *host_batch, int32_t chunks);

/* The whole path (as mp_plan_and_validate: profile, greedy_by_size plan,
 * validation) from HOST memory to HOST memory.  host_batch has the layout of
 * mp_batch but every array pointer is a host pointer; its CSR arrays must
 * start at 0, never decrease and end at n_tensors / n_steps (MP_EINVAL
 * otherwise), and profile_ptr is required.  The batch is cut into at most
 * `chunks` (0..MP_HOST_PATH_MAX_CHUNKS) runs of consecutive traces with about
 * equal tensor counts; each run's inputs are copied to the device on
 * copy_in_stream, planned on compute_stream once they have landed, and its
 * profile and offsets copied back on copy_out_stream once planned, so the
 * copies of both directions overlap the planning of other runs; the
 * per-trace results follow the last run.  The per-trace arrays move in one
 * copy each way when the host keeps trace_ptr, profile_ptr and steps in this
 * order with fewer than 16 bytes between them (read, never written), and
 * peak_lb, plan_peak, verdict, conflict, trace_status adjacent in this order
 * with no byte between them; otherwise one copy per array.  Page-locked (pinned) host memory
 * is needed for the copies to overlap; pageable memory is correct but
 * serialises them.  chunks = 0 stages nothing: the kernels read the inputs
 * from, and write the results to, the host arrays themselves over the
 * CPU-GPU link; every host array must then be page-locked memory mapped into
 * the device's address space (cudaHostAlloc / cudaMallocHost, or
 * cudaHostRegister with cudaHostRegisterMapped), else MP_EINVAL, and the
 * device buffer holds only the planner's workspace.  device_buffer:
 * caller-owned device memory of at least
 * mp_host_path_bytes(host_batch, chunks) bytes, 256-byte aligned, holding the
 * device copies and the workspace; not used concurrently by another call.
 * The call only enqueues work: the host outputs are complete once
 * copy_out_stream has reached its end (e.g. cudaStreamSynchronize), and the
 * host inputs must stay unchanged until copy_in_stream has.  The three
 * streams may be the same stream (no overlap).  Cross-stream order uses
 * events the library creates once per device; concurrent callers on one
 * device are serialised while they enqueue.  Return codes as for
 * mp_plan_and_validate; per-trace errors in out->trace_status. */
mp_status mp_plan_and_validate_host(const mp_batch *host_batch, mp_fit_policy policy, const mp_host_results *out,
                                    int32_t chunks, void *device_buffer, size_t device_bytes, void *copy_in_stream,
                                    void *compute_stream, void *copy_out_stream);

/* Bytes of device workspace mp_validate_plan needs for this batch. */
size_t mp_validate_workspace_bytes(const mp_batch *batch);

/* Plan validation (stage 3; pairwise constraints of Eq. 2.1).
 * verdict[b] = 1 iff for all i < j with overlapping lifetimes the address
 *   ranges [offset, offset + size) are disjoint (touching is allowed), else 0.
 * conflict[2b], conflict[2b+1] = the violating pair (i, j), i < j, with the
 *   smallest i and then the smallest j, or (-1, -1); may be NULL.
 * offsets: int64[n_tensors] device array, one per tensor.
 * workspace as for mp_plan_greedy_by_size, sized by
 * mp_validate_workspace_bytes. */
mp_status mp_validate_plan(const mp_batch *batch, const int64_t *offsets, int32_t *verdict,
                           int32_t *conflict, int32_t *trace_status, void *workspace,
                           size_t workspace_bytes, void *stream);

/* Peak of a given plan: plan_peak[b] = max_i offset_i + size_i (0 for an
 * empty trace), Eq. 2.1's total_mem.  Needs no workspace. */
mp_status mp_peak(const mp_batch *batch, const int64_t *offsets, int64_t *plan_peak,
                  int32_t *trace_status, void *stream);

/* Bytes of device workspace mp_plan_bump needs for this batch (depends on the
 * host scalars only).  0 means none. */
size_t mp_bump_workspace_bytes(const mp_batch *batch);

/* bump_allocation, the baseline strategy of Sec. 2.3: in allocation order
 * (alloc_step ascending, then id ascending) every tensor is given the running
 * offset, the sum of the sizes of the tensors allocated before it, so no
 * address range is reused whatever the lifetimes.
 * offsets[trace_ptr[b] + i]                                   int64[n_tensors]
 * plan_peak[b] = the sum of the trace's sizes (its total_mem)   int64[B]
 * trace_status[b]: MP_EINVAL / MP_EOVERFLOW as for mp_plan_greedy_by_size;
 *   a failed trace gets plan_peak 0 and unspecified offsets.     int32[B]
 * workspace: at least mp_bump_workspace_bytes(batch) bytes, rules as for
 * mp_plan_greedy_by_size. */
mp_status mp_plan_bump(const mp_batch *batch, int64_t *offsets, int64_t *plan_peak, int32_t *trace_status,
                       void *workspace, size_t workspace_bytes, void *stream);

/* Bytes of device workspace mp_plan_greedy_by_breadth needs for this batch. */
size_t mp_breadth_workspace_bytes(const mp_batch *batch);

/* Greedy by breadth, the strategy of Pisarchyk et al. discussed in Sec. 6:
 * operators in order of breadth (the sizes of their input and output
 * tensors) descending, each assigning offsets to its tensors not yet placed,
 * largest first, with greedy_by_size's gap search (policy as for
 * mp_plan_greedy_by_size).  A trace has one operator per step and no consumer
 * lists, so the operator at step t is read as producing the tensors allocated
 * at t and using for the last time the tensors freed at t + 1: its breadth is
 * the bytes of both, a tensor of one step counting once (ties: the earlier
 * step first), and a tensor is placed with the wider of its producer and its
 * last user.
 * offsets, plan_peak, trace_status as for mp_plan_greedy_by_size (a failed
 * trace gets plan_peak 0).  workspace: at least
 * mp_breadth_workspace_bytes(batch) bytes, rules as for
 * mp_plan_greedy_by_size. */
mp_status mp_plan_greedy_by_breadth(const mp_batch *batch, mp_fit_policy policy, int64_t *offsets,
                                    int64_t *plan_peak, int32_t *trace_status, void *workspace,
                                    size_t workspace_bytes, void *stream);

/* Traces of at most this many tensors are searched exhaustively by
 * mp_plan_optimal. */
#define MP_OPTIMAL_MAX_TENSORS 10

/* Bytes of device workspace mp_plan_optimal needs for this batch (depends on
 * the host scalars only). */
size_t mp_optimal_workspace_bytes(const mp_batch *batch);

/* The exact optimum of Eq. 2.1 (the smallest total_mem of any valid plan) for
 * traces of at most MP_OPTIMAL_MAX_TENSORS tensors, by exhaustive search over
 * every order of the tensors, each placed at its lowest feasible offset among
 * the lifetime-overlapping tensors placed before it (some order reproduces any
 * optimal packing).  It measures how far greedy_by_size is from optimal.
 * offsets[trace_ptr[b] + i]: the plan of the first optimal order in
 *   lexicographic order of tensor ids                        int64[n_tensors]
 * opt_peak[b] = the optimum (0 for an empty trace)                int64[B]
 * trace_status[b]: as for mp_plan_greedy_by_size; a trace of more than
 *   MP_OPTIMAL_MAX_TENSORS tensors gets MP_EINVAL.                 int32[B]
 * The search costs n! placements per trace of n tensors.
 * workspace: at least mp_optimal_workspace_bytes(batch) bytes, rules as for
 * mp_plan_greedy_by_size.  Two kernels are enqueued. */
mp_status mp_plan_optimal(const mp_batch *batch, int64_t *offsets, int64_t *opt_peak, int32_t *trace_status,
                          void *workspace, size_t workspace_bytes, void *stream);

/* Alignment of every trace's slab placed by mp_slab_layout. */
#define MP_SLAB_ALIGN 256

/* Places one slab per trace in a single device buffer and every tensor in it
 * (Sec. 3.3: prim::AllocateSlab[total_size] per graph, every tensor a view
 * prim::AllocateTensor[size, offset] into it).
 * batch: n_traces is required; trace_ptr and n_tensors are read only when
 *   tensor_addr is given (the other fields are not used).
 * plan_peak: int64[n_traces] device, each trace's total_mem.
 * trace_status: int32[n_traces] device or NULL; a trace whose status is not
 *   MP_OK (a failed plan) gets an empty slab.  Negative peaks count as 0.
 * slab_base: int64[n_traces + 1] device out: slab_base[b] = sum over earlier
 *   traces of their slab rounded up to MP_SLAB_ALIGN; slab_base[n_traces] =
 *   the buffer's size in bytes.
 * offsets: int64[n_tensors] device, the plan (required with tensor_addr).
 * tensor_addr: int64[n_tensors] device out or NULL: tensor_addr[i] =
 *   slab_base[b] + offsets[i], the byte address of tensor i of trace b in the
 *   buffer, or -1 for every tensor of a trace whose status is not MP_OK;
 *   entries of a trace whose CSR range is unsound (as for trace_status
 *   MP_EINVAL) and entries outside every trace are not written.
 * Returns MP_EINVAL for a NULL or misaligned required array.  One kernel, two
 * with tensor_addr. */
mp_status mp_slab_layout(const mp_batch *batch, const int64_t *plan_peak, const int32_t *trace_status,
                         const int64_t *offsets, int64_t *slab_base, int64_t *tensor_addr, void *stream);

/* Bytes of device workspace mp_replay_plan needs for this batch. */
size_t mp_replay_workspace_bytes(const mp_batch *batch);

/* Replays each trace's plan on its slab, the check on real memory of Eq. 2.1:
 * steps in order, at step t every tensor allocated at t fills its byte range
 * [slab_base[b] + offset, + size) with a pattern of its own, then every tensor
 * whose last live step is t (free = t + 1) compares its range with its
 * pattern.  Two tensors that overlap in lifetime and in address make one of
 * them fail, so ok[b] = 1 iff the plan is valid; first_bad[b] = the smallest id
 * whose range was overwritten while it was live, or -1.
 * slab: device buffer of slab_bytes bytes (4-byte aligned), for example sized
 * by mp_slab_layout; its contents are overwritten.  Every tensor must lie in
 * its trace's slab [0, slab_base[b+1] - slab_base[b]) and every slab in the
 * buffer, else the trace gets MP_EINVAL and nothing of it is written.
 * trace_status: as for mp_validate_plan.  workspace: at least
 * mp_replay_workspace_bytes(batch) bytes. */
mp_status mp_replay_plan(const mp_batch *batch, const int64_t *offsets, const int64_t *slab_base, void *slab,
                         int64_t slab_bytes, int32_t *ok, int32_t *first_bad, int32_t *trace_status,
                         void *workspace, size_t workspace_bytes, void *stream);

/* Static, NUL-terminated name of a status code. */
const char *mp_status_string(mp_status status);

/* ABI version of this header (incremented on incompatible changes). */
int32_t mp_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* MEMPLAN_H */
