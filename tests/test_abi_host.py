"""Host-side checks of the C ABI (no GPU): the library builds for sm_103a,
exports every function include/dynacomm.h declares, and rejects bad arguments
before launching anything."""
import ctypes
import os
import re

import pytest

from paper_2101_07968_gb300 import build as libbuild
from paper_2101_07968_gb300 import dynacomm as dc
from paper_2101_07968_gb300 import workloads as wl

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                      "include", "dynacomm.h")


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return dc.lib()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dc_[a-z0-9_]+)\s*\(", text)))


def test_header_symbols_exported(lib):
    names = _declared()
    assert len(names) >= 7
    raw = ctypes.CDLL(dc.LIB_PATH)
    for n in names:
        assert hasattr(raw, n), n
    assert sorted(dc.exported_names()) == names


def test_status_strings(lib):
    for s in range(9):
        assert dc.dc_status_string(s) and dc.dc_status_string(s) != "unknown status"
    assert dc.dc_status_string(99) == "unknown status"


def test_workspace_query(lib):
    assert dc.dc_schedule_workspace_bytes(-1, 8) == 0
    assert dc.dc_schedule_workspace_bytes(10, 0) == 0
    assert dc.dc_schedule_workspace_bytes(10, 4097) == 0
    assert dc.dc_schedule_workspace_bytes(1000, 16) >= 256 + 4000
    # 17 <= L <= 256: work list plus per-thread traceback slots, one per lane of
    # the launched CTAs: as many as the batch's tiles need, up to about one
    # resident wave (then fixed, so only the work list grows)
    mid = dc.dc_schedule_workspace_bytes(1000, 54)
    assert mid >= 256 + 4000 and mid == dc.dc_schedule_workspace_bytes(1000, 54)
    assert dc.dc_schedule_workspace_bytes(2000, 54) > mid + 4000
    big = dc.dc_schedule_workspace_bytes(200_000, 54)
    assert abs(dc.dc_schedule_workspace_bytes(300_000, 54) - big - 400_000) < 256
    # above L = 64 the listed instances also get DP-table slots
    assert dc.dc_schedule_workspace_bytes(1000, 65) > dc.dc_schedule_workspace_bytes(1000, 64)
    # long L: one DP-table slot per concurrently solved instance
    one = dc.dc_schedule_workspace_bytes(1, 1024)
    assert one >= 1024 * 1025 // 2 * 8
    assert dc.dc_schedule_workspace_bytes(16384, 1024) > one
    assert dc.dc_schedule_workspace_bytes(16384, 1024) <= 5 * 2**30


def test_kernel_launch_count(lib):
    """Two passes per schedule call; long deep-chain batches split their first
    pass into launches of about 90 ms of work (at least two resident waves)."""
    f = dc.dc_schedule_kernel_launches
    assert f(0, 16) == 0 and f(10, 0) == 0 and f(10, 4097) == 0
    assert f(1_000_000, 16) == 2 and f(262_144, 54) == 2 and f(10, 256) == 2
    assert f(1, 1024) == 2 and f(2000, 1024) == 2
    deep = f(16384, 1024)
    assert 3 <= deep <= 12          # 280 ms of work at the measured rate, split
    assert f(32768, 1024) >= deep   # more work, at least as many launches


FAKE = 0x1000  # never dereferenced: every case below fails its host check first


@pytest.mark.parametrize("fn", ["dc_schedule_forward_batch", "dc_schedule_backward_batch"])
def test_schedule_host_checks(lib, fn):
    f = getattr(dc, fn)
    big = 1 << 30
    assert f(5, 0, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, big) == dc.DC_ERR_BAD_SHAPE
    assert f(5, 4097, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, big) == dc.DC_ERR_BAD_SHAPE
    assert f(-1, 8, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, big) == dc.DC_ERR_BAD_SHAPE
    assert f(2**32, 8, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, big) == dc.DC_ERR_BAD_SHAPE
    assert f(0, 8, None, None, None, None, None, None, None, None, 0) == dc.DC_OK
    assert f(5, 8, None, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, big) == dc.DC_ERR_NULL
    assert f(5, 8, FAKE, FAKE, FAKE, None, FAKE, None, None, FAKE, big) == dc.DC_ERR_NULL
    assert f(5, 8, FAKE, FAKE, FAKE, FAKE, None, None, None, FAKE, big) == dc.DC_ERR_NULL
    need = dc.dc_schedule_workspace_bytes(5, 8)
    assert f(5, 8, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, None, need) == dc.DC_ERR_WORKSPACE
    assert f(5, 8, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, need - 1) == dc.DC_ERR_WORKSPACE
    need = dc.dc_schedule_workspace_bytes(50, 300)
    assert f(50, 300, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, need - 8) == \
        dc.DC_ERR_WORKSPACE


def test_eval_host_checks(lib):
    f = dc.dc_eval_timeline_batch
    assert f(5, 8, 2, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(5, 0, 0, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(0, 8, 0, None, None, None, None, None) == dc.DC_OK
    assert f(5, 8, 1, FAKE, FAKE, FAKE, None, FAKE) == dc.DC_ERR_NULL
    assert f(5, 8, 1, FAKE, None, FAKE, FAKE, FAKE) == dc.DC_ERR_NULL


def test_profile_gen_host_checks(lib):
    cfg = wl.with_batch(wl.config("tiny"), 10)
    for key, val, code in (("L", 0, dc.DC_ERR_BAD_CONFIG), ("L", 4097, dc.DC_ERR_BAD_CONFIG),
                           ("rate_lo", 0, dc.DC_ERR_BAD_CONFIG),
                           ("bw_hi", 2**31, dc.DC_ERR_BAD_CONFIG),
                           ("dt_lo", -1, dc.DC_ERR_BAD_CONFIG),
                           ("bwd_flops_mult", 17, dc.DC_ERR_BAD_CONFIG),
                           ("bits_per_param", 0, dc.DC_ERR_BAD_CONFIG),
                           ("layer_mode", 7, dc.DC_ERR_BAD_CONFIG),
                           ("batch", -1, dc.DC_ERR_BAD_CONFIG)):
        bad = dict(cfg)
        bad[key] = val
        assert dc.dc_profile_gen(bad, FAKE, FAKE, FAKE, FAKE, FAKE) == code, key
    fixed = wl.config("alexnet")
    bad = dict(fixed)
    bad["L"] = 1025
    bad["fixed_params"] = list(range(1025))
    bad["fixed_flops"] = list(range(1025))
    assert dc.dc_profile_gen(bad, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_CONFIG
    assert dc.dc_profile_gen(wl.with_batch(cfg, 0), None, None, None, None, None) == dc.DC_OK
    assert dc.dc_profile_gen(cfg, None, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_NULL


def test_roof_probe_host_checks(lib):
    f = dc.dc_roof_int_probe
    assert f(2, 1, 32, 4, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(0, 1, 33, 4, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(0, 1, 32, 3, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(0, 1, 32, 4, None) == dc.DC_ERR_NULL


def test_binding_refuses_host_tensors(lib):
    import torch
    with pytest.raises(ValueError):
        dc._ptr(torch.zeros(3, dtype=torch.int64))


@pytest.mark.parametrize("fn", ["dc_greedy_forward_batch", "dc_greedy_backward_batch"])
def test_greedy_host_checks(lib, fn):
    f = getattr(dc, fn)
    assert f(5, 0, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(5, 4097, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(-1, 8, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(2**32, 8, FAKE, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_BAD_SHAPE
    assert f(0, 8, None, None, None, None, None) == dc.DC_OK
    assert f(5, 8, None, FAKE, FAKE, FAKE, FAKE) == dc.DC_ERR_NULL
    assert f(5, 8, FAKE, FAKE, FAKE, None, FAKE) == dc.DC_ERR_NULL
    assert f(5, 8, FAKE, FAKE, FAKE, FAKE, None) == dc.DC_ERR_NULL


def test_generated_host_checks(lib):
    f = dc.dc_schedule_generated_batch
    q = dc.dc_schedule_generated_workspace_bytes
    assert q(1000, 16) >= 256 + 8 * 1000 and q(1000, 17) == 0 and q(-1, 8) == 0 and q(5, 0) == 0
    cfg = wl.with_batch(wl.config("vgg16"), 1000)
    need = q(1000, 16)
    bad = dict(cfg)
    bad["rate_lo"] = 0
    assert f(bad, FAKE, FAKE, None, None, FAKE, need) == dc.DC_ERR_BAD_CONFIG
    deep = wl.with_batch(wl.config("deepchain"), 10)
    assert f(deep, FAKE, FAKE, None, None, FAKE, 1 << 30) == dc.DC_ERR_BAD_SHAPE
    assert f(wl.with_batch(cfg, 0), None, None, None, None, None, 0) == dc.DC_OK
    assert f(cfg, None, FAKE, None, None, FAKE, need) == dc.DC_ERR_NULL
    assert f(cfg, FAKE, None, None, None, FAKE, need) == dc.DC_ERR_NULL
    assert f(cfg, FAKE, FAKE, None, None, None, need) == dc.DC_ERR_WORKSPACE
    assert f(cfg, FAKE, FAKE, None, None, FAKE, need - 1) == dc.DC_ERR_WORKSPACE


def test_time_next_pass_arguments(lib):
    """The timing request takes both events or neither; the checks run on the
    host (no event is touched until a schedule call uses the request)."""
    assert dc.dc_time_next_pass(None, FAKE) == dc.DC_ERR_NULL
    assert dc.dc_time_next_pass(FAKE, None) == dc.DC_ERR_NULL
    assert dc.dc_time_next_pass(None, None) == dc.DC_OK  # withdraws nothing pending
