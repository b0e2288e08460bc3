"""ctypes binding of libdynacomm.so (the C ABI in include/dynacomm.h).

The ``dc_*`` functions keep the C names and argument order and only marshal
arguments: torch tensors (or raw integer addresses) become device pointers and
the stream defaults to torch's current CUDA stream. Every step of the
scheduling path runs in the library's kernels; there is no CPU fallback, and
loading fails loudly when the library has not been built.

The convenience wrappers at the bottom (``profile_gen``, ``schedule``,
``eval_timeline``) allocate output tensors with torch and call the ``dc_*``
functions.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

_PKG = os.path.dirname(os.path.abspath(__file__))
# DC_CHECKED=1 loads the checked build (index checks that count failures
# instead of trapping; build it with `python -m paper_2101_07968_gb300.build --checked`)
LIB_PATH = os.path.join(_PKG, "libdynacomm_checked.so" if os.environ.get("DC_CHECKED") == "1"
                        else "libdynacomm.so")
CHECKED_UNITS = ("dp_deep", "dp_mid", "dp_small", "dp_group", "dp_fused")

DC_OK, DC_ERR_NULL, DC_ERR_BAD_SHAPE, DC_ERR_NEGATIVE, DC_ERR_RANGE = 0, 1, 2, 3, 4
DC_ERR_WORKSPACE, DC_ERR_CUDA, DC_ERR_BAD_CONFIG, DC_ERR_INTERNAL = 5, 6, 7, 8
DC_L_MAX = 4096
DC_STATIC_MAX_BATCH = 1048576
FWD, BWD = 0, 1


class DynaCommError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {dc_status_string(status)} (status {status})")
        self.status = status


class dc_profile_cfg(ctypes.Structure):
    _fields_ = [
        ("L", ctypes.c_int32), ("layer_mode", ctypes.c_int32),
        ("batch", ctypes.c_int64), ("inst0", ctypes.c_int64), ("seed", ctypes.c_uint64),
        ("fixed_params", ctypes.POINTER(ctypes.c_int64)),
        ("fixed_flops", ctypes.POINTER(ctypes.c_int64)),
        ("params_lo", ctypes.c_int64), ("params_hi", ctypes.c_int64),
        ("flops_lo", ctypes.c_int64), ("flops_hi", ctypes.c_int64),
        ("rate_dist", ctypes.c_int32), ("bw_dist", ctypes.c_int32),
        ("rate_lo", ctypes.c_int64), ("rate_hi", ctypes.c_int64),
        ("bw_lo", ctypes.c_int64), ("bw_hi", ctypes.c_int64),
        ("dt_lo", ctypes.c_int64), ("dt_hi", ctypes.c_int64),
        ("bwd_flops_mult", ctypes.c_int32), ("bits_per_param", ctypes.c_int32),
    ]


_lib = None

# name -> (restype, argtypes); the exported C ABI
_VP, _I32, _I64, _SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
_SIGNATURES = {
    "dc_profile_gen": (_I32, [ctypes.POINTER(dc_profile_cfg), _VP, _VP, _VP, _VP, _VP, _VP]),
    "dc_schedule_workspace_bytes": (_SZ, [_I64, _I32]),
    "dc_schedule_kernel_launches": (_I32, [_I64, _I32]),
    "dc_schedule_forward_batch": (_I32, [_I64, _I32, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                         _SZ, _VP]),
    "dc_schedule_backward_batch": (_I32, [_I64, _I32, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                          _SZ, _VP]),
    "dc_eval_timeline_batch": (_I32, [_I64, _I32, _I32, _VP, _VP, _VP, _VP, _VP, _VP]),
    "dc_schedule_batch_static": (_I32, [_I32, _I64, _I32, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                        _VP]),
    "dc_schedule_generated_workspace_bytes": (_SZ, [_I64, _I32]),
    "dc_schedule_generated_batch": (_I32, [ctypes.POINTER(dc_profile_cfg), _VP, _VP, _VP, _VP,
                                           _VP, _SZ, _VP]),
    "dc_greedy_forward_batch": (_I32, [_I64, _I32, _VP, _VP, _VP, _VP, _VP, _VP]),
    "dc_greedy_backward_batch": (_I32, [_I64, _I32, _VP, _VP, _VP, _VP, _VP, _VP]),
    "dc_status_string": (ctypes.c_char_p, [_I32]),
    "dc_roof_int_probe": (_I32, [_I32, _I32, _I32, _I64, _VP, _VP]),
    "dc_time_next_pass": (_I32, [_VP, _VP]),
}


def lib():
    """Load libdynacomm.so (raises if it is missing: build it first)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(
                f"{LIB_PATH} is missing: build it with `python -m paper_2101_07968_gb300.build`")
        l = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(l, name)
            fn.restype = res
            fn.argtypes = args
        _lib = l
    return _lib


def exported_names():
    return list(_SIGNATURES)


def checked_failures(reset: bool = False) -> dict:
    """Index-check counters of the checked build, per translation unit:
    {unit: (failed checks, source line of the first)}. reset=True clears them.
    Raises if the loaded library is not the checked build."""
    l = lib()
    out = {}
    for unit in CHECKED_UNITS:
        fn = getattr(l, "dc_checked_" + unit, None)
        if fn is None:
            raise RuntimeError(f"{LIB_PATH} is not the checked build")
        fn.restype = ctypes.c_int
        fn.argtypes = [ctypes.POINTER(ctypes.c_uint), ctypes.POINTER(ctypes.c_uint), ctypes.c_int]
        count, line = ctypes.c_uint(0), ctypes.c_uint(0)
        if fn(ctypes.byref(count), ctypes.byref(line), int(reset)) != 0:
            raise RuntimeError(f"reading the check counters of {unit} failed")
        out[unit] = (int(count.value), int(line.value))
    return out


# ------------------------------------------------------------- marshalling
def _ptr(x) -> Optional[int]:
    """torch tensor -> device address (must be CUDA); int -> itself; None -> NULL."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_cuda:
        raise ValueError("device tensor expected (the library takes device pointers)")
    if not x.is_contiguous():
        raise ValueError("contiguous tensor expected")
    return x.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        if not torch.cuda.is_available():
            return None
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(st: int, what: str):
    if st != DC_OK:
        raise DynaCommError(st, what)
    return st


# -------------------------------------------------------------- C ABI names
def dc_status_string(status: int) -> str:
    return lib().dc_status_string(int(status)).decode()


def dc_schedule_kernel_launches(batch: int, L: int) -> int:
    return int(lib().dc_schedule_kernel_launches(int(batch), int(L)))


def dc_schedule_workspace_bytes(batch: int, L: int) -> int:
    return int(lib().dc_schedule_workspace_bytes(int(batch), int(L)))


def make_cfg(cfg: dict, keep: list) -> dc_profile_cfg:
    """dict (see workloads.config) -> dc_profile_cfg; `keep` holds host arrays alive."""
    c = dc_profile_cfg()
    c.L = int(cfg["L"])
    c.layer_mode = int(cfg["layer_mode"])
    c.batch = int(cfg["batch"])
    c.inst0 = int(cfg.get("inst0", 0))
    c.seed = int(cfg["seed"])
    if int(cfg["layer_mode"]) == 0:
        import numpy as np
        fp = np.ascontiguousarray(cfg["fixed_params"], dtype=np.int64)
        ff = np.ascontiguousarray(cfg["fixed_flops"], dtype=np.int64)
        keep += [fp, ff]
        c.fixed_params = fp.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))
        c.fixed_flops = ff.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))
    for k in ("params_lo", "params_hi", "flops_lo", "flops_hi", "rate_lo", "rate_hi",
              "bw_lo", "bw_hi", "dt_lo", "dt_hi"):
        setattr(c, k, int(cfg.get(k, 0)))
    c.rate_dist = int(cfg["rate_dist"])
    c.bw_dist = int(cfg["bw_dist"])
    c.bwd_flops_mult = int(cfg.get("bwd_flops_mult", 2))
    c.bits_per_param = int(cfg.get("bits_per_param", 32))
    return c


def dc_profile_gen(cfg, fc, pt, bc, gt, dt, stream=None) -> int:
    keep: list = []
    c = cfg if isinstance(cfg, dc_profile_cfg) else make_cfg(cfg, keep)
    return int(lib().dc_profile_gen(ctypes.byref(c), _ptr(fc), _ptr(pt), _ptr(bc), _ptr(gt),
                                    _ptr(dt), _stream(stream)))


def dc_schedule_forward_batch(batch, L, fc, pt, dt, makespan, bits, nseg, status, workspace,
                              workspace_bytes, stream=None) -> int:
    return int(lib().dc_schedule_forward_batch(
        int(batch), int(L), _ptr(fc), _ptr(pt), _ptr(dt), _ptr(makespan), _ptr(bits),
        _ptr(nseg), _ptr(status), _ptr(workspace), int(workspace_bytes), _stream(stream)))


def dc_schedule_backward_batch(batch, L, bc, gt, dt, makespan, bits, nseg, status, workspace,
                               workspace_bytes, stream=None) -> int:
    return int(lib().dc_schedule_backward_batch(
        int(batch), int(L), _ptr(bc), _ptr(gt), _ptr(dt), _ptr(makespan), _ptr(bits),
        _ptr(nseg), _ptr(status), _ptr(workspace), int(workspace_bytes), _stream(stream)))


def dc_schedule_batch_static(direction, batch, L, comp, xfer, dt, makespan, bits, nseg, status,
                             stream=None) -> int:
    """Workspace-free solve for 1 <= L <= 16 and batch <= DC_STATIC_MAX_BATCH, for
    callers that cannot allocate device memory; its scratch is a fixed array in the
    library shared by every call on a device (overlapping calls race)."""
    return int(lib().dc_schedule_batch_static(
        int(direction), int(batch), int(L), _ptr(comp), _ptr(xfer), _ptr(dt), _ptr(makespan),
        _ptr(bits), _ptr(nseg), _ptr(status), _stream(stream)))


def dc_eval_timeline_batch(batch, L, direction, comp, xfer, dt, bits, makespan,
                           stream=None) -> int:
    return int(lib().dc_eval_timeline_batch(
        int(batch), int(L), int(direction), _ptr(comp), _ptr(xfer), _ptr(dt), _ptr(bits),
        _ptr(makespan), _stream(stream)))


def dc_schedule_generated_workspace_bytes(batch: int, L: int) -> int:
    return int(lib().dc_schedule_generated_workspace_bytes(int(batch), int(L)))


def dc_schedule_generated_batch(cfg, makespan, bits, nseg, status, workspace, workspace_bytes,
                                stream=None) -> int:
    keep: list = []
    c = cfg if isinstance(cfg, dc_profile_cfg) else make_cfg(cfg, keep)
    return int(lib().dc_schedule_generated_batch(
        ctypes.byref(c), _ptr(makespan), _ptr(bits), _ptr(nseg), _ptr(status), _ptr(workspace),
        int(workspace_bytes), _stream(stream)))


def dc_greedy_forward_batch(batch, L, fc, pt, dt, makespan, bits, stream=None) -> int:
    return int(lib().dc_greedy_forward_batch(int(batch), int(L), _ptr(fc), _ptr(pt), _ptr(dt),
                                             _ptr(makespan), _ptr(bits), _stream(stream)))


def dc_greedy_backward_batch(batch, L, bc, gt, dt, makespan, bits, stream=None) -> int:
    return int(lib().dc_greedy_backward_batch(int(batch), int(L), _ptr(bc), _ptr(gt), _ptr(dt),
                                              _ptr(makespan), _ptr(bits), _stream(stream)))


def dc_roof_int_probe(variant, blocks, threads, iters, sink, stream=None) -> int:
    return int(lib().dc_roof_int_probe(int(variant), int(blocks), int(threads), int(iters),
                                       _ptr(sink), _stream(stream)))


def dc_time_next_pass(start, stop) -> int:
    """start, stop: torch.cuda.Event (recorded at least once, so that their CUDA
    events exist), raw cudaEvent_t addresses, or None for both."""
    def ev(e):
        if e is None:
            return None
        return e if isinstance(e, int) else int(e.cuda_event)
    return int(lib().dc_time_next_pass(ev(start), ev(stop)))


# ------------------------------------------------------------ conveniences
def words(L: int) -> int:
    return (L - 1 + 31) // 32


def profile_gen(cfg: dict, device="cuda", stream=None) -> dict:
    """Allocate and fill fc, pt, bc, gt [batch, L] and dt [batch] (int64, device)."""
    import torch
    B, L = int(cfg["batch"]), int(cfg["L"])
    out = {k: torch.empty((B, L), dtype=torch.int64, device=device)
           for k in ("fc", "pt", "bc", "gt")}
    out["dt"] = torch.empty(B, dtype=torch.int64, device=device)
    _check(dc_profile_gen(cfg, out["fc"], out["pt"], out["bc"], out["gt"], out["dt"], stream),
           "dc_profile_gen")
    return out


class Scheduler:
    """Owns a reusable workspace and output buffers for one (batch, L)."""

    def __init__(self, batch: int, L: int, device="cuda"):
        import torch
        self.batch, self.L, self.W = int(batch), int(L), words(L)
        self.ws_bytes = dc_schedule_workspace_bytes(batch, L)
        self.workspace = torch.empty(max(self.ws_bytes, 1), dtype=torch.uint8, device=device)
        self.out = {}
        for d in (FWD, BWD):
            self.out[d] = dict(
                makespan=torch.empty(self.batch, dtype=torch.int64, device=device),
                bits=torch.empty((self.batch, max(self.W, 1)), dtype=torch.int32,
                                 device=device),
                nseg=torch.empty(self.batch, dtype=torch.int32, device=device),
                status=torch.empty(self.batch, dtype=torch.int32, device=device))

    def run(self, direction: int, comp, xfer, dt, stream=None) -> dict:
        o = self.out[direction]
        fn = dc_schedule_forward_batch if direction == FWD else dc_schedule_backward_batch
        _check(fn(self.batch, self.L, comp, xfer, dt, o["makespan"], o["bits"], o["nseg"],
                  o["status"], self.workspace, self.ws_bytes, stream),
               "dc_schedule_forward_batch" if direction == FWD else "dc_schedule_backward_batch")
        return o


def schedule(direction: int, comp, xfer, dt, stream=None) -> dict:
    """One direction for a batch: makespan, bits (int32 view of uint32 words), nseg, status."""
    B, L = comp.shape
    s = Scheduler(B, L, device=comp.device)
    return s.run(direction, comp, xfer, dt, stream)


def eval_timeline(direction: int, comp, xfer, dt, bits, stream=None):
    import torch
    B, L = comp.shape
    out = torch.empty(B, dtype=torch.int64, device=comp.device)
    _check(dc_eval_timeline_batch(B, L, direction, comp, xfer, dt, bits, out, stream),
           "dc_eval_timeline_batch")
    return out


class GeneratedScheduler:
    """Generate-and-solve (L <= 16) for a config dict with fixed batch and L:
    both directions without materialising the profiles. run() returns dict of
    makespan [2, B] int64, bits [2, B, max(W,1)] int32 view, nseg and status
    [2, B] int32 (index 0 forward, 1 backward)."""

    def __init__(self, cfg: dict, device="cuda"):
        import torch
        self.cfg, self.keep = cfg, []
        self.c = make_cfg(cfg, self.keep)
        B, L = int(cfg["batch"]), int(cfg["L"])
        self.W = words(L)
        self.ws_bytes = dc_schedule_generated_workspace_bytes(B, L)
        if self.ws_bytes == 0:
            raise DynaCommError(DC_ERR_BAD_SHAPE, "dc_schedule_generated_workspace_bytes")
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        self.out = {"makespan": torch.empty((2, B), dtype=torch.int64, device=device),
                    "bits": torch.empty((2, B, max(self.W, 1)), dtype=torch.int32, device=device),
                    "nseg": torch.empty((2, B), dtype=torch.int32, device=device),
                    "status": torch.empty((2, B), dtype=torch.int32, device=device)}

    def run(self, stream=None) -> dict:
        o = self.out
        _check(dc_schedule_generated_batch(self.c, o["makespan"], o["bits"], o["nseg"],
                                           o["status"], self.ws, self.ws_bytes, stream),
               "dc_schedule_generated_batch")
        return o


def greedy(direction: int, comp, xfer, dt, stream=None) -> dict:
    """The paper's competing greedy scheduler for one direction (Algorithm 1
    forward, Algorithm 2 backward): dict(makespan [B] int64, bits [B, max(W,1)]
    int32 view of the uint32 decision words)."""
    import torch
    B, L = comp.shape
    W = words(L)
    out = {"makespan": torch.empty(B, dtype=torch.int64, device=comp.device),
           "bits": torch.empty((B, max(W, 1)), dtype=torch.int32, device=comp.device)}
    fn = dc_greedy_forward_batch if direction == 0 else dc_greedy_backward_batch
    _check(fn(B, L, comp, xfer, dt, out["makespan"], out["bits"], stream),
           "dc_greedy_forward_batch" if direction == 0 else "dc_greedy_backward_batch")
    return out


class StepGraph:
    """One whole step for a fixed config -- dc_profile_gen, the forward and backward
    DPs and the f_m replay of both decisions -- captured once as a CUDA graph and
    replayed. For small batches the host cost of the step's launches exceeds the
    kernels' own time; replay() issues them as one graph launch. The two
    directions are independent, so after the generator they run on two branches
    of the graph (each with its own workspace): one direction's kernels start on
    the SMs the other's tail leaves free, and a replay kernel (memory-bound) can
    run beside the other direction's DP (integer-ALU-bound). After each replay():
    prof (fc, pt, bc, gt, dt), sched.out[d] and replay_out[d] for d in (FWD, BWD)
    hold that step's results."""

    def __init__(self, cfg: dict, device="cuda"):
        import torch
        self.B, self.L = int(cfg["batch"]), int(cfg["L"])
        self.keep: list = []
        self.c = make_cfg(cfg, self.keep)
        B, L = self.B, self.L
        self.prof = {k: torch.empty((B, L), dtype=torch.int64, device=device)
                     for k in ("fc", "pt", "bc", "gt")}
        self.prof["dt"] = torch.empty(B, dtype=torch.int64, device=device)
        self.sched = Scheduler(B, L, device=device)
        self.sched_b = Scheduler(B, L, device=device)  # the backward branch's workspace
        self.sched.out[BWD] = self.sched_b.out[BWD]
        self.replay_out = {d: torch.empty(B, dtype=torch.int64, device=device)
                           for d in (FWD, BWD)}
        self._branch = torch.cuda.Stream(device=device)
        # one eager step first: one-time setup (function attributes, occupancy
        # queries) happens outside the capture
        side = torch.cuda.Stream(device=device)
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            self._step()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self._step()

    def _direction(self, d, sched):
        p = self.prof
        c, x = ("fc", "pt") if d == FWD else ("bc", "gt")
        o = sched.run(d, p[c], p[x], p["dt"])
        _check(dc_eval_timeline_batch(self.B, self.L, d, p[c], p[x], p["dt"], o["bits"],
                                      self.replay_out[d]), "dc_eval_timeline_batch")

    def _step(self):
        import torch
        p = self.prof
        _check(dc_profile_gen(self.c, p["fc"], p["pt"], p["bc"], p["gt"], p["dt"]),
               "dc_profile_gen")
        main = torch.cuda.current_stream()
        self._branch.wait_stream(main)  # the backward branch starts after the generator
        self._direction(FWD, self.sched)
        with torch.cuda.stream(self._branch):
            self._direction(BWD, self.sched_b)
        main.wait_stream(self._branch)

    def replay(self):
        self.graph.replay()


def shared_inputs(host_in, keys):
    """Key -> the first key whose tensor is the same buffer (same address, size and
    dtype); every key maps to itself when host_in is None."""
    if host_in is None:
        return {k: k for k in keys}
    seen, canon = {}, {}
    for k in keys:
        x = host_in[k]
        canon[k] = seen.setdefault((x.data_ptr(), x.numel(), x.dtype), k)
    return canon


class HostPipeline:
    """End-to-end scheduling of profiles that live in pinned host memory.

    The batch is cut into `chunks` contiguous pieces. Three CUDA streams overlap
    the host->device copy of piece c+1 with the forward DP, backward DP and
    timeline replay of piece c (all through the C ABI on slices of the device
    buffers), and with the device->host copy of piece c-1's results. Inputs and
    outputs are dicts of pinned CPU tensors: inputs fc, pt, bc, gt [batch, L] and
    dt [batch]; outputs, per direction d in (FWD, BWD), (d, "makespan"),
    (d, "bits"), (d, "nseg"), (d, "replay"). Inputs that are the same host
    buffer (same address and size, e.g. gt passed as pt when the two transfers
    cost the same) are copied once and read by both solves.
    """

    IN_KEYS = ("fc", "pt", "bc", "gt", "dt")

    def __init__(self, batch: int, L: int, chunks: Optional[int] = None, device="cuda"):
        import torch
        self.batch, self.L, self.W = int(batch), int(L), words(L)
        if not chunks:  # one piece per 65,536 instances, 1 to 8: a piece costs a few
            # host-side calls, and its DP launches should still fill the GPU
            chunks = max(1, min(8, self.batch // 65536))
        self.chunks = max(1, min(int(chunks), self.batch))
        self.bounds = [self.batch * c // self.chunks for c in range(self.chunks + 1)]
        step = max(b - a for a, b in zip(self.bounds, self.bounds[1:]))
        self.ws_bytes = dc_schedule_workspace_bytes(step, L)
        self.workspace = torch.empty(max(self.ws_bytes, 1), dtype=torch.uint8, device=device)
        B = self.batch
        self.dev = {k: torch.empty((B, L), dtype=torch.int64, device=device)
                    for k in ("fc", "pt", "bc", "gt")}
        self.dev["dt"] = torch.empty(B, dtype=torch.int64, device=device)
        self.out = {}
        for d in (FWD, BWD):
            self.out[(d, "makespan")] = torch.empty(B, dtype=torch.int64, device=device)
            self.out[(d, "bits")] = torch.empty((B, max(self.W, 1)), dtype=torch.int32,
                                                device=device)
            self.out[(d, "nseg")] = torch.empty(B, dtype=torch.int32, device=device)
            self.out[(d, "replay")] = torch.empty(B, dtype=torch.int64, device=device)
        self.s_in, self.s_run, self.s_out = (torch.cuda.Stream(device=device) for _ in range(3))
        self.ev_in = [torch.cuda.Event() for _ in range(self.chunks)]
        self.ev_run = [torch.cuda.Event() for _ in range(self.chunks)]

    def host_buffers(self):
        """Pinned host tensors shaped like the outputs."""
        return {k: torch_empty_pinned_like(v) for k, v in self.out.items()}

    def _canonical(self, host_in):
        return shared_inputs(host_in, self.IN_KEYS)

    def bytes_per_run(self, host_in=None):
        """Bytes copied host->device and device->host by one run with these inputs."""
        canon = self._canonical(host_in)
        h2d = sum(self.dev[k].numel() * self.dev[k].element_size()
                  for k in self.IN_KEYS if canon[k] == k)
        d2h = sum(v.numel() * v.element_size() for v in self.out.values())
        return h2d, d2h

    def run(self, host_in: dict, host_out: dict):
        import torch
        canon = self._canonical(host_in)
        cur = torch.cuda.current_stream()
        self.s_in.wait_stream(cur)
        for c in range(self.chunks):
            lo, hi = self.bounds[c], self.bounds[c + 1]
            if hi <= lo:
                continue
            n = hi - lo
            with torch.cuda.stream(self.s_in):
                for k in self.IN_KEYS:
                    if canon[k] == k:
                        self.dev[k][lo:hi].copy_(host_in[k][lo:hi], non_blocking=True)
                self.ev_in[c].record(self.s_in)
            self.s_run.wait_event(self.ev_in[c])
            sr = self.s_run.cuda_stream
            d = {k: self.dev[canon[k]][lo:hi] for k in self.IN_KEYS}
            o = {k: v[lo:hi] for k, v in self.out.items()}
            for dr, (ck, xk) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
                fn = dc_schedule_forward_batch if dr == FWD else dc_schedule_backward_batch
                _check(fn(n, self.L, d[ck], d[xk], d["dt"], o[(dr, "makespan")],
                          o[(dr, "bits")], o[(dr, "nseg")], None, self.workspace,
                          self.ws_bytes, sr), "schedule (host pipeline)")
                _check(dc_eval_timeline_batch(n, self.L, dr, d[ck], d[xk], d["dt"],
                                              o[(dr, "bits")], o[(dr, "replay")], sr),
                       "dc_eval_timeline_batch (host pipeline)")
            self.ev_run[c].record(self.s_run)
            self.s_out.wait_event(self.ev_run[c])
            with torch.cuda.stream(self.s_out):
                for k, v in o.items():
                    host_out[k][lo:hi].copy_(v, non_blocking=True)
        cur.wait_stream(self.s_out)
        cur.wait_stream(self.s_run)


def torch_empty_pinned_like(t):
    import torch
    return torch.empty(t.shape, dtype=t.dtype).pin_memory()
