"""The workspace-free entry point against the workspace one, on the GPU.

dc_schedule_batch_static exists for callers that cannot allocate device memory
where they schedule (a runtime whose allocator owns all device memory, or a
scheduler running in the idle window between a push and the next pull, where a
cudaMalloc could synchronise the device). Its scratch is a fixed array inside
the library, shared by all calls, so this file runs last and checks two calls in
a row: the second must not see the first one's leftovers.
"""
import numpy as np
import pytest

from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build, dynacomm
    build.build()
    dynacomm.lib()
    return dynacomm


def _outputs(torch, B, W):
    return dict(makespan=torch.empty(B, dtype=torch.int64, device="cuda"),
                bits=torch.empty((B, max(W, 1)), dtype=torch.int32, device="cuda"),
                nseg=torch.empty(B, dtype=torch.int32, device="cuda"),
                status=torch.empty(B, dtype=torch.int32, device="cuda"))


@pytest.mark.parametrize("name,batch", [("vgg16", 200_003), ("tiny", 4096)])
def test_static_scratch_matches_workspace_entry(dc, name, batch):
    import torch
    cfg = wl.with_batch(wl.config(name), batch)
    prof = dc.profile_gen(cfg)
    B, L, W = batch, cfg["L"], dc.words(cfg["L"])
    # a poisoned instance and two 64-bit ones, so that the shared work list is used
    prof["pt"][7, 0] = 1 << 34
    prof["gt"][11, 3] = 1 << 34
    prof["fc"][13, 1] = -1
    for d, (c, x) in ((dc.FWD, ("fc", "pt")), (dc.BWD, ("bc", "gt"))):
        ref = dc.schedule(d, prof[c], prof[x], prof["dt"])
        torch.cuda.synchronize()
        ref = {k: v.cpu().numpy() for k, v in ref.items()}
        for call in range(2):
            out = _outputs(torch, B, W)
            st = dc.dc_schedule_batch_static(d, B, L, prof[c], prof[x], prof["dt"],
                                             out["makespan"], out["bits"], out["nseg"],
                                             out["status"])
            assert st == dc.DC_OK, dc.dc_status_string(st)
            torch.cuda.synchronize()
            for k in ("makespan", "nseg", "status"):
                assert np.array_equal(out[k].cpu().numpy(), ref[k]), (name, d, call, k)
            g = out["bits"].cpu().numpy()[:, :W]
            assert np.array_equal(g, ref["bits"][:, :W]), (name, d, call, "bits")
        if d == dc.FWD:
            assert ref["status"][13] == dc.DC_ERR_NEGATIVE and ref["status"][7] == dc.DC_OK
        else:
            assert ref["status"][11] == dc.DC_OK


def test_static_scratch_null_status_and_nseg(dc):
    """With nseg and status NULL, a failed instance reports -status in its
    makespan; every other output equals the workspace entry's, on two calls in a
    row through the shared scratch."""
    import torch
    cfg = wl.with_batch(wl.config("vgg16"), 50_000)
    prof = dc.profile_gen(cfg)
    B, L, W = cfg["batch"], cfg["L"], dc.words(cfg["L"])
    prof["pt"][7, 0] = 1 << 34   # 64-bit instance: the work list is used
    prof["fc"][13, 1] = -1       # negative cost
    prof["dt"][21] = 1 << 51     # L * dt beyond 2^52
    for d, (c, x) in ((dc.FWD, ("fc", "pt")), (dc.BWD, ("bc", "gt"))):
        ref = dc.schedule(d, prof[c], prof[x], prof["dt"])
        torch.cuda.synchronize()
        ref = {k: v.cpu().numpy() for k, v in ref.items()}
        for call in range(2):
            out = _outputs(torch, B, W)
            st = dc.dc_schedule_batch_static(d, B, L, prof[c], prof[x], prof["dt"],
                                             out["makespan"], out["bits"], None, None)
            assert st == dc.DC_OK, dc.dc_status_string(st)
            torch.cuda.synchronize()
            got = out["makespan"].cpu().numpy()
            assert np.array_equal(got, ref["makespan"]), (d, call)
            assert np.array_equal(out["bits"].cpu().numpy()[:, :W], ref["bits"][:, :W])
            if d == dc.FWD:
                assert got[13] == -dc.DC_ERR_NEGATIVE
            assert got[21] == -dc.DC_ERR_RANGE


def test_static_scratch_limits(dc):
    import torch
    big = dc.DC_STATIC_MAX_BATCH + 1
    z = torch.empty(1, dtype=torch.int64, device="cuda")
    assert dc.dc_schedule_batch_static(0, big, 8, z, z, z, z, z, None, None) == \
        dc.DC_ERR_WORKSPACE
    assert dc.dc_schedule_batch_static(0, 10, 17, z, z, z, z, z, None, None) == \
        dc.DC_ERR_BAD_SHAPE
    assert dc.dc_schedule_batch_static(2, 10, 8, z, z, z, z, z, None, None) == \
        dc.DC_ERR_BAD_SHAPE
    assert dc.dc_schedule_batch_static(0, 0, 8, None, None, None, None, None, None, None) == \
        dc.DC_OK
