"""DynaComm CPU oracle -- TEST INFRASTRUCTURE ONLY.

A plain C statement of the paper's scheduling path (the recurrences Eq. 8 and
Eq. 9 of Algorithms 3 and 4, with their choice among equal optima, the cost function f_m of Sec. III-B written from Eq. 1-7,
brute force over the 0-1 program, the seeded profile generator standing in
for the profiler of Sec. IV-A, and the paper's competing greedy schedulers,
Algorithms 1 and 2), wrapped with ctypes and numpy.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this package. It shares no code with the CUDA library in
``paper_2101_07968_gb300`` and neither imports the other.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dynacomm_oracle.c")
_SRC_GREEDY = os.path.join(_HERE, "greedy_oracle.c")
_HDR = os.path.join(_HERE, "dynacomm_oracle.h")
# DC_ORACLE_LIB names a library built from planted-mistake copies of these
# sources; only tests/test_oracle_mutations.py sets it, in child processes
_LIB_OVERRIDE = os.environ.get("DC_ORACLE_LIB")
_LIB = _LIB_OVERRIDE or os.path.join(_HERE, "liboracle.so")

LAYERS_FIXED, LAYERS_UNIFORM, LAYERS_LOGUNIFORM = 0, 1, 2
DIST_UNIFORM, DIST_LOGUNIFORM = 0, 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C99, -O2, pthreads)."""
    if _LIB_OVERRIDE:
        return _LIB_OVERRIDE
    stale = force or not os.path.exists(_LIB) or any(
        os.path.getmtime(p) > os.path.getmtime(_LIB) for p in (_SRC, _SRC_GREEDY, _HDR))
    if stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-std=gnu99", "-O2", "-fPIC", "-shared", "-Wall",
                               "-o", tmp, _SRC, _SRC_GREEDY, "-lm", "-lpthread"])
        os.replace(tmp, _LIB)
    return _LIB


class _Cfg(ctypes.Structure):
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


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        i64, i32, u64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_uint64
        vp = ctypes.c_void_p
        _lib.orc_dp_forward.restype = i64
        _lib.orc_dp_forward.argtypes = [i32, vp, vp, i64, vp, vp]
        _lib.orc_dp_backward.restype = i64
        _lib.orc_dp_backward.argtypes = [i32, vp, vp, i64, vp, vp]
        _lib.orc_replay_forward.restype = i64
        _lib.orc_replay_forward.argtypes = [i32, vp, vp, i64, vp]
        _lib.orc_replay_backward.restype = i64
        _lib.orc_replay_backward.argtypes = [i32, vp, vp, i64, vp]
        _lib.orc_brute.restype = i64
        _lib.orc_brute.argtypes = [i32, i32, vp, vp, i64, vp, vp]
        _lib.orc_dp_backward_1d.restype = i64
        _lib.orc_dp_backward_1d.argtypes = [i32, vp, vp, i64]
        _lib.orc_schedule_batch.restype = None
        _lib.orc_schedule_batch.argtypes = [i32, i64, i32, vp, vp, vp, vp, vp, vp, vp, i32]
        _lib.orc_replay_batch.restype = None
        _lib.orc_replay_batch.argtypes = [i32, i64, i32, vp, vp, vp, vp, vp, i32]
        _lib.orc_splitmix64.restype = u64
        _lib.orc_splitmix64.argtypes = [u64, u64]
        _lib.orc_uniform_int.restype = i64
        _lib.orc_uniform_int.argtypes = [i64, i64, u64]
        _lib.orc_loguniform.restype = i64
        _lib.orc_loguniform.argtypes = [i64, i64, u64]
        _lib.orc_instance_draws.restype = None
        _lib.orc_instance_draws.argtypes = [ctypes.POINTER(_Cfg), i64, vp, vp, vp]
        _lib.orc_layer_draw.restype = i64
        _lib.orc_layer_draw.argtypes = [ctypes.POINTER(_Cfg), i64, i32, i32]
        _lib.orc_greedy_forward.restype = None
        _lib.orc_greedy_forward.argtypes = [i32, vp, vp, i64, vp]
        _lib.orc_greedy_backward.restype = None
        _lib.orc_greedy_backward.argtypes = [i32, vp, vp, i64, vp]
        _lib.orc_greedy_batch.restype = None
        _lib.orc_greedy_batch.argtypes = [i32, i64, i32, vp, vp, vp, vp, vp, i32]
        _lib.orc_profile_gen.restype = i32
        _lib.orc_profile_gen.argtypes = [ctypes.POINTER(_Cfg), vp, vp, vp, vp, vp]
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _i64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int64)


def words(L: int) -> int:
    """Packed decision words per instance, ceil((L-1)/32)."""
    return (L - 1 + 31) // 32


# ---------------------------------------------------------------- one instance
def dp(direction: int, comp, xfer, dt: int):
    """Algorithm 3 (direction 0: comp=fc, xfer=pt) or 4 (1: comp=bc, xfer=gt).

    Returns (makespan, decision d[0..L] as uint8, nseg)."""
    comp, xfer = _i64(comp), _i64(xfer)
    L = comp.shape[0]
    d = np.zeros(L + 1, dtype=np.uint8)
    s = ctypes.c_int32(0)
    if direction == 0:
        v = lib().orc_dp_forward(L, _p(xfer), _p(comp), int(dt), _p(d), ctypes.byref(s))
    else:
        v = lib().orc_dp_backward(L, _p(comp), _p(xfer), int(dt), _p(d), ctypes.byref(s))
    return int(v), d, int(s.value)


def replay(direction: int, comp, xfer, dt: int, d) -> int:
    """f_m of Sec. III-B for decision d[0..L] (entries 1..L-1 used)."""
    comp, xfer = _i64(comp), _i64(xfer)
    L = comp.shape[0]
    d = np.ascontiguousarray(d, dtype=np.uint8)
    assert d.shape[0] == L + 1
    if direction == 0:
        return int(lib().orc_replay_forward(L, _p(xfer), _p(comp), int(dt), _p(d)))
    return int(lib().orc_replay_backward(L, _p(comp), _p(xfer), int(dt), _p(d)))


def brute(direction: int, comp, xfer, dt: int, with_table: bool = False):
    """Brute force over all 2^(L-1) decisions: (optimum, fewest segments among
    optimal decisions[, opt table (L+1)x(L+1) of sub-problem optima])."""
    comp, xfer = _i64(comp), _i64(xfer)
    L = comp.shape[0]
    s = ctypes.c_int32(0)
    tab = np.zeros((L + 1) * (L + 1), dtype=np.int64) if with_table else None
    v = lib().orc_brute(direction, L, _p(comp), _p(xfer), int(dt), ctypes.byref(s),
                        _p(tab) if with_table else None)
    if with_table:
        return int(v), int(s.value), tab.reshape(L + 1, L + 1)
    return int(v), int(s.value)


def dp_backward_1d(bc, gt, dt: int) -> int:
    bc, gt = _i64(bc), _i64(gt)
    return int(lib().orc_dp_backward_1d(bc.shape[0], _p(bc), _p(gt), int(dt)))


# ------------------------------------------------------------------- batches
def schedule_batch(direction: int, comp, xfer, dt, nthreads: int = 1):
    """Returns dict(makespan [B] int64, bits [B,W] uint32, nseg [B] int32, status [B] int32)."""
    comp, xfer, dt = _i64(comp), _i64(xfer), _i64(dt)
    B, L = comp.shape
    W = words(L)
    out = dict(makespan=np.zeros(B, np.int64), bits=np.zeros((B, W), np.uint32),
               nseg=np.zeros(B, np.int32), status=np.zeros(B, np.int32))
    lib().orc_schedule_batch(direction, B, L, _p(comp), _p(xfer), _p(dt), _p(out["makespan"]),
                             _p(out["bits"]), _p(out["nseg"]), _p(out["status"]), int(nthreads))
    return out


def replay_batch(direction: int, comp, xfer, dt, bits, nthreads: int = 1) -> np.ndarray:
    comp, xfer, dt = _i64(comp), _i64(xfer), _i64(dt)
    B, L = comp.shape
    bits = np.ascontiguousarray(bits, dtype=np.uint32).reshape(B, words(L))
    out = np.zeros(B, np.int64)
    lib().orc_replay_batch(direction, B, L, _p(comp), _p(xfer), _p(dt), _p(bits), _p(out),
                           int(nthreads))
    return out


def greedy_forward(pt, fc, dt: int) -> np.ndarray:
    """Algorithm 1 (iBatch forward greedy): decision p[0..L] (uint8)."""
    pt, fc = _i64(pt), _i64(fc)
    L = len(pt)
    p = np.zeros(L + 1, np.uint8)
    lib().orc_greedy_forward(L, _p(pt), _p(fc), int(dt), _p(p))
    return p


def greedy_backward(bc, gt, dt: int) -> np.ndarray:
    """Algorithm 2 (iPart backward greedy): decision g[0..L] (uint8)."""
    bc, gt = _i64(bc), _i64(gt)
    L = len(bc)
    g = np.zeros(L + 1, np.uint8)
    lib().orc_greedy_backward(L, _p(bc), _p(gt), int(dt), _p(g))
    return g


def greedy_batch(direction: int, comp, xfer, dt, nthreads: int = 1) -> dict:
    """Algorithm 1 (direction 0) or 2 (direction 1) over a batch: dict(bits [B,W]
    uint32, makespan [B] int64 = f_m of the decision, -status on a bad instance)."""
    comp, xfer, dt = _i64(comp), _i64(xfer), _i64(dt)
    B, L = comp.shape
    out = dict(bits=np.zeros((B, words(L)), np.uint32), makespan=np.zeros(B, np.int64))
    lib().orc_greedy_batch(direction, B, L, _p(comp), _p(xfer), _p(dt), _p(out["bits"]),
                           _p(out["makespan"]), int(nthreads))
    return out


def bits_to_decision(bits_row, L: int) -> np.ndarray:
    d = np.zeros(L + 1, np.uint8)
    for l in range(1, L):
        d[l] = (int(bits_row[(l - 1) // 32]) >> ((l - 1) % 32)) & 1
    return d


# ----------------------------------------------------------------- generator
def _cfg_struct(cfg: dict, keep: list) -> _Cfg:
    c = _Cfg()
    c.L = int(cfg["L"])
    c.layer_mode = int(cfg["layer_mode"])
    c.batch = int(cfg["batch"])
    c.inst0 = int(cfg.get("inst0", 0))
    c.seed = int(cfg["seed"])
    if cfg["layer_mode"] == LAYERS_FIXED:
        fp, ff = _i64(cfg["fixed_params"]), _i64(cfg["fixed_flops"])
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


def profile_gen(cfg: dict):
    """Returns dict(fc, pt, bc, gt [batch, L] int64, dt [batch] int64)."""
    keep: list = []
    c = _cfg_struct(cfg, keep)
    B, L = c.batch, c.L
    out = {k: np.zeros((B, L), np.int64) for k in ("fc", "pt", "bc", "gt")}
    out["dt"] = np.zeros(B, np.int64)
    rc = lib().orc_profile_gen(ctypes.byref(c), _p(out["fc"]), _p(out["pt"]), _p(out["bc"]),
                               _p(out["gt"]), _p(out["dt"]))
    if rc != 0:
        raise ValueError("bad profile config")
    return out


def instance_draws(cfg: dict, i: int):
    keep: list = []
    c = _cfg_struct(cfg, keep)
    r, b, d = (np.zeros(1, np.int64) for _ in range(3))
    lib().orc_instance_draws(ctypes.byref(c), int(i), _p(r), _p(b), _p(d))
    return int(r[0]), int(b[0]), int(d[0])


def layer_draw(cfg: dict, i: int, field: int, layer: int) -> int:
    keep: list = []
    c = _cfg_struct(cfg, keep)
    return int(lib().orc_layer_draw(ctypes.byref(c), int(i), int(field), int(layer)))


def splitmix64(seed: int, ctr: int) -> int:
    return int(lib().orc_splitmix64(seed, ctr))


def uniform_int(lo: int, hi: int, r: int) -> int:
    return int(lib().orc_uniform_int(lo, hi, r))


def loguniform(lo: int, hi: int, r: int) -> int:
    return int(lib().orc_loguniform(lo, hi, r))
