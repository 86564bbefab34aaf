"""GB300-native memory planning for DNN allocation traces (MemoMalloc's static-analysis path).

Stages (all in libmemplan.so's CUDA kernels, reached through the C ABI in
include/memplan.h):

1. live-bytes profile per op step and its peak lower bound;
2. greedy_by_size offset assignment (first- or best-fit gaps) and the plan peak;
3. pairwise validation of a plan against Eq. 2.1's ordering constraints;

and bump_allocation (the baseline strategy of Sec. 2.3), greedy by breadth
(Sec. 6), the exact optimum of
Eq. 2.1 for traces of at most 10 tensors, and plans materialised on device
slabs and replayed on real memory (Sec. 3.3).
"""
from ._lib import (EINTERNAL, EINVAL, ENOMEM, EOVERFLOW, ETIMEOUT, FIT_BEST, FIT_FIRST, OK, SLAB_ALIGN,
                   MemplanError, status_string)
from .api import (DeviceBatch, HostPath, PathBuffers, PathResult, Workspace, bump_workspace_bytes, live_profile,
                  materialize, peak, plan_and_validate, plan_bump, plan_greedy_by_breadth, plan_greedy_by_size,
                  plan_optimal,
                  plan_workspace_bytes, replay_plan, run_path, slab_layout, validate_plan,
                  validate_workspace_bytes)

__all__ = [
    "DeviceBatch", "HostPath", "PathBuffers", "PathResult", "Workspace", "bump_workspace_bytes", "live_profile", "peak",
    "plan_and_validate", "plan_bump", "plan_greedy_by_breadth", "plan_greedy_by_size", "plan_optimal",
    "plan_workspace_bytes", "run_path",
    "materialize", "replay_plan", "slab_layout", "validate_plan", "validate_workspace_bytes", "MemplanError",
    "status_string", "OK", "EINVAL", "EOVERFLOW", "ENOMEM", "EINTERNAL", "ETIMEOUT", "FIT_FIRST", "FIT_BEST",
    "SLAB_ALIGN",
]
