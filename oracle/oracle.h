/*
 * oracle.h -- plain single-threaded CPU reference of the memory-planning path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may include, link or
 * call this code; the parity tests, the package's smoke check and the bench's
 * CPU-baseline leg are its only users.  It shares no code, header or constant
 * with the CUDA library: the status values below restate the public error
 * contract on purpose so that error codes can be compared.
 *
 * A batch is a structure of arrays with CSR offsets (all host pointers):
 *   trace_ptr[B+1]   tensors of trace b are [trace_ptr[b], trace_ptr[b+1])
 *   steps[B]         T_b, op steps of trace b
 *   profile_ptr[B+1] profile entries of trace b are [profile_ptr[b], +T_b)
 *   alloc_step, free_step (int32), size_bytes (int64), one per tensor;
 *   the lifetime of tensor i is the half-open step range [a_i, f_i).
 */
#ifndef MEMPLAN_ORACLE_H
#define MEMPLAN_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { OR_OK = 0, OR_EINVAL = 1, OR_EOVERFLOW = 2 };
enum { OR_FIT_FIRST = 0, OR_FIT_BEST = 1 };

typedef struct {
    int32_t n_traces;
    const int64_t *trace_ptr;
    const int32_t *steps;
    const int64_t *profile_ptr; /* may be NULL except for or_live_profile */
    const int32_t *alloc_step;
    const int32_t *free_step;
    const int64_t *size_bytes;
} or_batch;

/* Live bytes at every step (sum of sizes of tensors with a <= t < f) and its
 * maximum, the lower bound on any feasible total_mem of Eq. 2.1. */
int or_live_profile(const or_batch *b, int64_t *profile, int64_t *peak_lb, int32_t *trace_status);

/* greedy_by_size (Sec. 2.3): priority order size desc, alloc asc, id asc;
 * each tensor goes to the first (policy 0) or the smallest (policy 1) gap
 * among the already placed tensors that overlap it in lifetime. */
int or_plan_greedy_by_size(const or_batch *b, int32_t policy, int64_t *offsets, int64_t *plan_peak,
                           int32_t *trace_status);

/* Greedy by breadth (the strategy of Pisarchyk et al. discussed in Sec. 6):
 * operators by breadth -- the sizes of their input and output tensors --
 * descending.  A trace has one operator per step and no consumer lists, so
 * the operator at step t is read as producing the tensors allocated at t
 * (outputs) and using for the last time the tensors freed at t + 1 (inputs);
 * its breadth is the bytes of both, a tensor of one step counting once.
 * Operators are taken by breadth descending (earlier step on ties), each
 * taking its not yet placed tensors by the greedy_by_size priority; so a
 * tensor's place in the order is the wider of its producer and its last user,
 * then size desc, alloc asc, id asc.  Placement as greedy_by_size with the
 * given policy. */
int or_plan_greedy_by_breadth(const or_batch *b, int32_t policy, int64_t *offsets, int64_t *plan_peak,
                              int32_t *trace_status);

/* Pairwise constraints of Eq. 2.1: verdict 1 iff no two lifetime-overlapping
 * tensors have intersecting [offset, offset + size); conflict[2b], [2b+1] is
 * the lexicographically smallest violating (i, j), i < j, local ids, or -1. */
int or_validate_plan(const or_batch *b, const int64_t *offsets, int32_t *verdict, int32_t *conflict,
                     int32_t *trace_status);

/* total_mem of a plan: max over tensors of offset + size (0 for no tensors). */
int or_peak(const or_batch *b, const int64_t *offsets, int64_t *plan_peak, int32_t *trace_status);

/* bump_allocation (Sec. 2.3): in allocation order (alloc asc, id asc) every
 * tensor takes the running offset, which then grows by its size. */
int or_plan_bump(const or_batch *b, int64_t *offsets, int64_t *plan_peak, int32_t *trace_status);

/* Exact optimum of the offline DSA problem (Eq. 2.1) for one tiny trace
 * (n <= 10): the minimum over all n! placement orders of the plan that puts
 * each tensor at its lowest non-conflicting offset.  Returns -1 if n > 10. */
int64_t or_bruteforce_opt(int32_t n, const int32_t *alloc_step, const int32_t *free_step,
                          const int64_t *size_bytes, int64_t *best_offsets);

#ifdef __cplusplus
}
#endif
#endif
