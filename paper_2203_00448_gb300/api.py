"""Python binding of the memory-planning C ABI (argument marshalling only).

Device memory and streams come from PyTorch; every step of the path runs in
libmemplan.so's CUDA kernels.  Function names follow the C ABI:

    live_profile(batch)                  -> profile, peak_lb, status     (stage 1)
    plan_greedy_by_size(batch, policy)   -> offsets, plan_peak, status   (stage 2)
    validate_plan(batch, offsets)        -> verdict, conflict, status    (stage 3)
    peak(batch, offsets)                 -> plan_peak, status

All calls are asynchronous on the current (or given) CUDA stream.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass

import torch

from . import _lib
from ._lib import FIT_BEST, FIT_FIRST, MemplanError, MpBatch

_POLICIES = {"first": FIT_FIRST, "best": FIT_BEST, FIT_FIRST: FIT_FIRST, FIT_BEST: FIT_BEST}


def _policy(p) -> int:
    try:
        return _POLICIES[p]
    except KeyError:
        raise ValueError(f"unknown fit policy {p!r}; use 'first' or 'best'") from None


def _stream_ptr(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


def _ptr(t):
    return None if t is None or t.numel() == 0 else t.data_ptr()


@dataclass
class DeviceBatch:
    """A batch of traces resident on one CUDA device (structure of arrays + CSR).

    The host scalars (n_traces, max_tensors, max_steps, n_tensors, n_steps)
    size launches and workspace; the kernels re-check every trace against
    them.
    """

    trace_ptr: torch.Tensor
    steps: torch.Tensor
    profile_ptr: torch.Tensor
    alloc_step: torch.Tensor
    free_step: torch.Tensor
    size_bytes: torch.Tensor
    n_traces: int
    max_tensors: int
    max_steps: int
    n_tensors: int
    n_steps: int

    @classmethod
    def from_host(cls, ts, device="cuda", non_blocking: bool = False) -> "DeviceBatch":
        """Copies a host batch (numpy arrays, e.g. tracegen.TraceSet) to `device`."""
        def dev(a, dt):
            t = torch.as_tensor(a).to(dt)
            return t.to(device, non_blocking=non_blocking)

        return cls(
            trace_ptr=dev(ts.trace_ptr, torch.int64),
            steps=dev(ts.steps, torch.int32),
            profile_ptr=dev(ts.profile_ptr, torch.int64),
            alloc_step=dev(ts.alloc_step, torch.int32),
            free_step=dev(ts.free_step, torch.int32),
            size_bytes=dev(ts.size_bytes, torch.int64),
            n_traces=int(ts.n_traces),
            max_tensors=int(ts.max_tensors),
            max_steps=int(ts.max_steps),
            n_tensors=int(ts.n_tensors),
            n_steps=int(ts.n_steps),
        )

    @property
    def device(self) -> torch.device:
        return self.alloc_step.device

    def slice_traces(self, t0: int, t1: int) -> "DeviceBatch":
        """The traces [t0, t1) as a batch of their own, sharing this batch's
        device arrays (the CSR offsets stay global, so per-tensor and per-step
        outputs keep their positions)."""
        return DeviceBatch(self.trace_ptr[t0:t1 + 1], self.steps[t0:t1], self.profile_ptr[t0:t1 + 1],
                           self.alloc_step, self.free_step, self.size_bytes, t1 - t0, self.max_tensors,
                           self.max_steps, self.n_tensors, self.n_steps)

    def struct(self) -> MpBatch:
        return MpBatch(self.n_traces, self.max_tensors, self.max_steps, 0, self.n_tensors, self.n_steps,
                       _ptr(self.trace_ptr), _ptr(self.steps), _ptr(self.profile_ptr), _ptr(self.alloc_step),
                       _ptr(self.free_step), _ptr(self.size_bytes))


class Workspace:
    """Caller-owned scratch for the calls that need it; grows on demand, never shrinks."""

    def __init__(self, device="cuda"):
        self.device = torch.device(device)
        self.buf = None

    def get(self, nbytes: int):
        if nbytes == 0:
            return None, 0
        if self.buf is None or self.buf.numel() < nbytes:
            # 256-byte alignment: the caching allocator returns 512-byte aligned blocks
            self.buf = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        return self.buf.data_ptr(), self.buf.numel()


_default_ws = {}


def _workspace(ws, device):
    if ws is not None:
        return ws
    key = torch.device(device)
    if key not in _default_ws:
        _default_ws[key] = Workspace(key)
    return _default_ws[key]


def _check(fn, st):
    if st != _lib.OK:
        raise MemplanError(fn, st)


def _empty(n, dtype, device):
    return torch.empty(max(int(n), 0), dtype=dtype, device=device)


def plan_workspace_bytes(batch: DeviceBatch) -> int:
    s = batch.struct()
    return int(_lib.load().mp_plan_workspace_bytes(ctypes.byref(s)))


def validate_workspace_bytes(batch: DeviceBatch) -> int:
    s = batch.struct()
    return int(_lib.load().mp_validate_workspace_bytes(ctypes.byref(s)))


def live_profile(batch: DeviceBatch, profile=None, peak_lb=None, status=None, stream=None):
    """Stage 1: live bytes per step (int64[n_steps]) and its max per trace."""
    lib, dev = _lib.load(), batch.device
    profile = _empty(batch.n_steps, torch.int64, dev) if profile is None else profile
    peak_lb = _empty(batch.n_traces, torch.int64, dev) if peak_lb is None else peak_lb
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    _check("mp_live_profile", lib.mp_live_profile(ctypes.byref(s), _ptr(profile), _ptr(peak_lb), _ptr(status),
                                                  _stream_ptr(stream)))
    return profile, peak_lb, status


def plan_greedy_by_size(batch: DeviceBatch, policy="first", offsets=None, plan_peak=None, status=None,
                        workspace: Workspace | None = None, stream=None):
    """Stage 2: greedy_by_size offsets (int64[n_tensors]) and the plan peak per trace."""
    lib, dev = _lib.load(), batch.device
    offsets = _empty(batch.n_tensors, torch.int64, dev) if offsets is None else offsets
    plan_peak = _empty(batch.n_traces, torch.int64, dev) if plan_peak is None else plan_peak
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    need = int(lib.mp_plan_workspace_bytes(ctypes.byref(s)))
    wptr, wbytes = _workspace(workspace, dev).get(need)
    _check("mp_plan_greedy_by_size",
           lib.mp_plan_greedy_by_size(ctypes.byref(s), _policy(policy), _ptr(offsets), _ptr(plan_peak),
                                      _ptr(status), wptr, wbytes, _stream_ptr(stream)))
    return offsets, plan_peak, status


def validate_plan(batch: DeviceBatch, offsets: torch.Tensor, verdict=None, conflict=None, status=None,
                  workspace: Workspace | None = None, stream=None, want_conflict: bool = True):
    """Stage 3: per-trace verdict (1 valid) and first conflicting pair (int32[B, 2])."""
    lib, dev = _lib.load(), batch.device
    verdict = _empty(batch.n_traces, torch.int32, dev) if verdict is None else verdict
    if conflict is None and want_conflict:
        conflict = _empty(2 * batch.n_traces, torch.int32, dev)
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    need = int(lib.mp_validate_workspace_bytes(ctypes.byref(s)))
    wptr, wbytes = _workspace(workspace, dev).get(need)
    _check("mp_validate_plan",
           lib.mp_validate_plan(ctypes.byref(s), _ptr(offsets), _ptr(verdict), _ptr(conflict), _ptr(status),
                                wptr, wbytes, _stream_ptr(stream)))
    return verdict, (conflict.view(-1, 2) if conflict is not None else None), status


def plan_and_validate(batch: DeviceBatch, policy="first", buffers: "PathBuffers | None" = None, profile: bool = True,
                      stream=None) -> "PathResult":
    """The whole path in one kernel pass: profile (optional), greedy_by_size plan and its validation.

    Same results as live_profile + plan_greedy_by_size + validate_plan; the
    single status row applies to every output of a trace.
    """
    lib = _lib.load()
    buf = buffers or PathBuffers(batch)
    s = batch.struct()
    need = int(lib.mp_plan_workspace_bytes(ctypes.byref(s)))
    wptr, wbytes = buf.plan_ws.get(need)
    _check("mp_plan_and_validate",
           lib.mp_plan_and_validate(ctypes.byref(s), _policy(policy), _ptr(buf.profile) if profile else None,
                                    _ptr(buf.peak_lb) if profile else None, _ptr(buf.offsets), _ptr(buf.plan_peak),
                                    _ptr(buf.verdict), _ptr(buf.conflict), _ptr(buf.status[0]), wptr, wbytes,
                                    _stream_ptr(stream)))
    return PathResult(buf.profile, buf.peak_lb, buf.offsets, buf.plan_peak, buf.verdict,
                      buf.conflict.view(-1, 2), buf.status[0])


def bump_workspace_bytes(batch: DeviceBatch) -> int:
    s = batch.struct()
    return int(_lib.load().mp_bump_workspace_bytes(ctypes.byref(s)))


def plan_bump(batch: DeviceBatch, offsets=None, plan_peak=None, status=None, workspace: "Workspace | None" = None,
              stream=None):
    """bump_allocation (the baseline strategy of Sec. 2.3): each tensor at the
    running offset in allocation order.  Returns (offsets, plan_peak, status)."""
    lib, dev = _lib.load(), batch.device
    offsets = _empty(batch.n_tensors, torch.int64, dev) if offsets is None else offsets
    plan_peak = _empty(batch.n_traces, torch.int64, dev) if plan_peak is None else plan_peak
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    wptr, wbytes = _workspace(workspace, dev).get(int(lib.mp_bump_workspace_bytes(ctypes.byref(s))))
    _check("mp_plan_bump", lib.mp_plan_bump(ctypes.byref(s), _ptr(offsets), _ptr(plan_peak), _ptr(status), wptr,
                                            wbytes, _stream_ptr(stream)))
    return offsets, plan_peak, status


def plan_greedy_by_breadth(batch: DeviceBatch, policy="first", offsets=None, plan_peak=None, status=None,
                           workspace: "Workspace | None" = None, stream=None):
    """Greedy by breadth (Sec. 6; the operator at step t produces the tensors
    allocated at t and uses last the tensors freed at t + 1).  Returns
    (offsets, plan_peak, status)."""
    lib, dev = _lib.load(), batch.device
    offsets = _empty(batch.n_tensors, torch.int64, dev) if offsets is None else offsets
    plan_peak = _empty(batch.n_traces, torch.int64, dev) if plan_peak is None else plan_peak
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    wptr, wbytes = _workspace(workspace, dev).get(int(lib.mp_breadth_workspace_bytes(ctypes.byref(s))))
    _check("mp_plan_greedy_by_breadth",
           lib.mp_plan_greedy_by_breadth(ctypes.byref(s), _policy(policy), _ptr(offsets), _ptr(plan_peak),
                                         _ptr(status), wptr, wbytes, _stream_ptr(stream)))
    return offsets, plan_peak, status


def plan_optimal(batch: DeviceBatch, offsets=None, opt_peak=None, status=None, workspace: "Workspace | None" = None,
                 stream=None):
    """The exact optimum of Eq. 2.1 for traces of at most 10 tensors (exhaustive
    search over tensor orders).  Returns (offsets, opt_peak, status)."""
    lib, dev = _lib.load(), batch.device
    offsets = _empty(batch.n_tensors, torch.int64, dev) if offsets is None else offsets
    opt_peak = _empty(batch.n_traces, torch.int64, dev) if opt_peak is None else opt_peak
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    wptr, wbytes = _workspace(workspace, dev).get(int(lib.mp_optimal_workspace_bytes(ctypes.byref(s))))
    _check("mp_plan_optimal", lib.mp_plan_optimal(ctypes.byref(s), _ptr(offsets), _ptr(opt_peak), _ptr(status),
                                                  wptr, wbytes, _stream_ptr(stream)))
    return offsets, opt_peak, status


def slab_layout(plan_peak: torch.Tensor, plan_status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Byte offset of every trace's slab in one buffer (Sec. 3.3's
    prim::AllocateSlab per trace): int64[B + 1], the last entry the total.
    Traces whose plan_status is non-zero get an empty slab."""
    lib = _lib.load()
    n = plan_peak.numel()
    base = torch.empty(n + 1, dtype=torch.int64, device=plan_peak.device)
    s = _lib.MpBatch(n, 0, 0, 0, 0, 0, None, None, None, None, None, None)
    _check("mp_slab_layout", lib.mp_slab_layout(ctypes.byref(s), _ptr(plan_peak), _ptr(plan_status), None,
                                                base.data_ptr(), None, _stream_ptr(stream)))
    return base


def materialize(batch: DeviceBatch, offsets: torch.Tensor, plan_peak: torch.Tensor,
                plan_status: torch.Tensor | None = None, stream=None):
    """One device buffer holding every trace's slab, and every tensor's byte
    address in it (Sec. 3.3's prim::AllocateTensor views; -1 for the tensors
    of a failed trace): returns (slab uint8 tensor, slab_base int64[B + 1],
    address of each tensor int64[n_tensors])."""
    lib = _lib.load()
    base = torch.empty(batch.n_traces + 1, dtype=torch.int64, device=batch.device)
    where = _empty(batch.n_tensors, torch.int64, batch.device)
    s = batch.struct()
    _check("mp_slab_layout", lib.mp_slab_layout(ctypes.byref(s), _ptr(plan_peak), _ptr(plan_status), _ptr(offsets),
                                                base.data_ptr(), _ptr(where), _stream_ptr(stream)))
    total = int(base[-1].item())
    slab = torch.empty(max(total, 1), dtype=torch.uint8, device=batch.device)
    return slab, base, where


def replay_plan(batch: DeviceBatch, offsets: torch.Tensor, slab_base: torch.Tensor, slab: torch.Tensor,
                workspace: "Workspace | None" = None, stream=None):
    """Replays the plan on the slab (every tensor writes its pattern at its
    alloc step and checks it at its last live step).  Returns (ok, first_bad,
    status): ok[b] = 1 iff nothing was overwritten while live."""
    lib, dev = _lib.load(), batch.device
    ok = _empty(batch.n_traces, torch.int32, dev)
    first_bad = _empty(batch.n_traces, torch.int32, dev)
    status = _empty(batch.n_traces, torch.int32, dev)
    s = batch.struct()
    wptr, wbytes = _workspace(workspace, dev).get(int(lib.mp_replay_workspace_bytes(ctypes.byref(s))))
    _check("mp_replay_plan", lib.mp_replay_plan(ctypes.byref(s), _ptr(offsets), _ptr(slab_base), slab.data_ptr(),
                                                slab.numel(), _ptr(ok), _ptr(first_bad), _ptr(status), wptr, wbytes,
                                                _stream_ptr(stream)))
    return ok, first_bad, status


def peak(batch: DeviceBatch, offsets: torch.Tensor, plan_peak=None, status=None, stream=None):
    """total_mem of a given plan per trace: max(offset + size)."""
    lib, dev = _lib.load(), batch.device
    plan_peak = _empty(batch.n_traces, torch.int64, dev) if plan_peak is None else plan_peak
    status = _empty(batch.n_traces, torch.int32, dev) if status is None else status
    s = batch.struct()
    _check("mp_peak", lib.mp_peak(ctypes.byref(s), _ptr(offsets), _ptr(plan_peak), _ptr(status),
                                  _stream_ptr(stream)))
    return plan_peak, status


@dataclass
class PathResult:
    profile: torch.Tensor
    peak_lb: torch.Tensor
    offsets: torch.Tensor
    plan_peak: torch.Tensor
    verdict: torch.Tensor
    conflict: torch.Tensor
    status: torch.Tensor  # int32[3, B]: profile, plan, validate


class PathBuffers:
    """Preallocated outputs for repeated runs of the whole path on one batch."""

    def __init__(self, batch: DeviceBatch):
        dev = batch.device
        B = batch.n_traces
        self.profile = _empty(batch.n_steps, torch.int64, dev)
        self.peak_lb = _empty(B, torch.int64, dev)
        self.offsets = _empty(batch.n_tensors, torch.int64, dev)
        self.plan_peak = _empty(B, torch.int64, dev)
        self.verdict = _empty(B, torch.int32, dev)
        self.conflict = _empty(2 * B, torch.int32, dev)
        self.status = torch.empty((3, B), dtype=torch.int32, device=dev)
        self.plan_ws = Workspace(dev)
        self.validate_ws = Workspace(dev)
        self.plan_ws.get(plan_workspace_bytes(batch))
        self.validate_ws.get(validate_workspace_bytes(batch))

    def slice_traces(self, t0: int, t1: int) -> "PathBuffers":
        """Views of the outputs for traces [t0, t1) (profile and offsets whole,
        as their positions are global), sharing the workspaces."""
        v = object.__new__(PathBuffers)
        v.profile, v.offsets = self.profile, self.offsets
        v.peak_lb, v.plan_peak, v.verdict = self.peak_lb[t0:t1], self.plan_peak[t0:t1], self.verdict[t0:t1]
        v.conflict, v.status = self.conflict[2 * t0:2 * t1], self.status[:, t0:t1]
        v.plan_ws, v.validate_ws = self.plan_ws, self.validate_ws
        return v


def run_path(batch: DeviceBatch, policy="first", buffers: PathBuffers | None = None, stream=None) -> PathResult:
    """One pass of the whole path: profile, greedy_by_size plan (with its peak), validation."""
    buf = buffers or PathBuffers(batch)
    live_profile(batch, buf.profile, buf.peak_lb, buf.status[0], stream=stream)
    plan_greedy_by_size(batch, policy, buf.offsets, buf.plan_peak, buf.status[1], workspace=buf.plan_ws,
                        stream=stream)
    validate_plan(batch, buf.offsets, buf.verdict, buf.conflict, buf.status[2], workspace=buf.validate_ws,
                  stream=stream)
    return PathResult(buf.profile, buf.peak_lb, buf.offsets, buf.plan_peak, buf.verdict,
                      buf.conflict.view(-1, 2), buf.status)


def _packed(specs, device=None, pin_memory=False):
    """One byte buffer holding the named arrays (each start 16-byte aligned),
    and a typed view of each: returns (buffer, {name: view})."""
    starts, pos = [], 0
    for _, shape, dt in specs:
        pos = (pos + 15) & ~15
        starts.append(pos)
        pos += int(torch.Size(shape).numel()) * torch.empty((), dtype=dt).element_size()
    buf = torch.empty(max(pos, 16), dtype=torch.uint8, device=device, pin_memory=pin_memory)
    views = {}
    for (name, shape, dt), o in zip(specs, starts):
        nbytes = int(torch.Size(shape).numel()) * torch.empty((), dtype=dt).element_size()
        views[name] = buf[o:o + nbytes].view(dt).view(shape)
    return buf, views


class HostPath:
    """End-to-end use from host memory through mp_plan_and_validate_host: the
    batch sits in pinned host buffers, and one call copies it to the device,
    runs the whole path (profile, plan, validation) and copies every result
    back, cut into `chunks` runs of traces so that the copies of both
    directions overlap the planning of other runs (three streams).  With
    ``chunks=0`` nothing is staged: the kernels read the pinned inputs and
    write the pinned results directly over the CPU-GPU link.

    ``run(ts)`` takes a host batch (numpy arrays, e.g. tracegen.TraceSet) with
    the same shape as the one the object was built for and returns host
    numpy views of profile, peak_lb, offsets, plan_peak, verdict, conflict,
    status; it returns once the results are on the host.
    """

    _IN = ("trace_ptr", "steps", "profile_ptr", "alloc_step", "free_step", "size_bytes")
    _OUT = ("profile", "peak_lb", "offsets", "plan_peak", "verdict", "conflict", "status")

    def __init__(self, ts, device="cuda", policy="first", stream=None, chunks: int = 4):
        self.policy = policy
        dev = torch.device(device)
        B, N, S = int(ts.n_traces), int(ts.n_tensors), int(ts.n_steps)
        # the per-trace arrays in the orders mp_plan_and_validate_host moves in
        # one copy each way: trace_ptr, profile_ptr, steps (at most 15 bytes
        # apart); peak_lb, plan_peak, verdict, conflict, status (adjacent, which
        # the 16-byte alignment of the packing keeps when B is a multiple of 4)
        in_specs = [("trace_ptr", (B + 1,), torch.int64), ("profile_ptr", (B + 1,), torch.int64),
                    ("steps", (B,), torch.int32), ("alloc_step", (N,), torch.int32),
                    ("free_step", (N,), torch.int32), ("size_bytes", (N,), torch.int64)]
        out_specs = [("profile", (S,), torch.int64), ("offsets", (N,), torch.int64), ("peak_lb", (B,), torch.int64),
                     ("plan_peak", (B,), torch.int64), ("verdict", (B,), torch.int32),
                     ("conflict", (2 * B,), torch.int32), ("status", (B,), torch.int32)]
        self.host_in_buf, self.host_in = _packed(in_specs, pin_memory=True)
        self.host_out_buf, self.host_out = _packed(out_specs, pin_memory=True)
        self._h2d = sum(int(self.host_in[k].numel()) * self.host_in[k].element_size() for k in self._IN)
        self._d2h = sum(int(self.host_out[k].numel()) * self.host_out[k].element_size() for k in self._OUT)
        self.stage(ts)
        self.hb = _lib.MpBatch(B, int(ts.max_tensors), int(ts.max_steps), 0, N, S,
                               *(self.host_in[k].data_ptr() for k in self._IN))
        self.res = _lib.MpHostResults(*(self.host_out[k].data_ptr() for k in self._OUT))
        self.chunks = max(0, min(int(chunks), _lib.HOST_PATH_MAX_CHUNKS))
        need = int(_lib.load().mp_host_path_bytes(ctypes.byref(self.hb), self.chunks))
        if need == 0 and B > 0:
            raise MemplanError("mp_host_path_bytes", _lib.EINVAL)
        self.dev_buf = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
        with torch.cuda.device(dev):
            self.compute_stream = stream or torch.cuda.current_stream(dev)
            self.copy_in_stream = torch.cuda.Stream(dev)
            self.copy_out_stream = torch.cuda.Stream(dev)

    @property
    def h2d_bytes(self) -> int:
        return self._h2d

    @property
    def d2h_bytes(self) -> int:
        return self._d2h

    def stage(self, ts):
        """Places a host batch into the pinned input buffer (host-side memcpy)."""
        for k in self._IN:
            self.host_in[k].numpy()[...] = getattr(ts, k)

    def run(self, ts=None):
        if ts is not None:
            self.stage(ts)
        # the device buffer is reused: the previous call's compute must not
        # overlap this call's copies (stream order covers the rest)
        self.copy_in_stream.wait_stream(self.compute_stream)
        _check("mp_plan_and_validate_host",
               _lib.load().mp_plan_and_validate_host(
                   ctypes.byref(self.hb), _policy(self.policy), ctypes.byref(self.res), self.chunks,
                   self.dev_buf.data_ptr(), self.dev_buf.numel(), self.copy_in_stream.cuda_stream,
                   self.compute_stream.cuda_stream, self.copy_out_stream.cuda_stream))
        self.copy_out_stream.synchronize()
        return {k: v.numpy() for k, v in self.host_out.items()}
