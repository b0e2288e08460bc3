"""dc_time_next_pass on the GPU: the events it asks for bracket the first pass of
the next schedule call (dense, looped and deep-chain kernels), inside the call's
own time, and leave every output as it is without the request; the request is
used up by that one call."""
import numpy as np
import pytest

from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build as libbuild
    from paper_2101_07968_gb300 import dynacomm as dc
    libbuild.build()
    dc.lib()
    return dc


def _events(torch, n):
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
    for e in evs:
        e.record()  # creates the CUDA events
    torch.cuda.synchronize()
    return evs


@pytest.mark.parametrize("L, B", [(8, 5000), (16, 40_013), (54, 3000), (300, 200)])
def test_first_pass_events(dc, L, B):
    import torch
    comp, xfer, dt = wl.random_instances(77 + L, B, L)
    c, x, d = (torch.from_numpy(a).cuda() for a in (comp, xfer, dt))
    sch = dc.Scheduler(B, L)
    ref = {k: v.clone() for k, v in sch.run(0, c, x, d).items()}
    call0, k0, k1, call1 = _events(torch, 4)
    for direction in (0, 1):
        call0.record()
        assert dc.dc_time_next_pass(k0, k1) == dc.DC_OK
        out = sch.run(direction, c, x, d)
        call1.record()
        torch.cuda.synchronize()
        first = k0.elapsed_time(k1)
        call = call0.elapsed_time(call1)
        assert 0.0 < first <= call, (first, call)
        # the request is used up: a second call records nothing into k0/k1
        k1_before = k1.elapsed_time(call1)
        sch.run(direction, c, x, d)
        torch.cuda.synchronize()
        assert k1.elapsed_time(call1) == pytest.approx(k1_before)
    out = sch.run(0, c, x, d)
    torch.cuda.synchronize()
    for k in ("makespan", "bits", "nseg", "status"):
        assert torch.equal(out[k], ref[k]), k


def test_request_used_up_by_a_failing_call(dc):
    """A schedule call that fails its host checks still uses up the request: the
    next, valid call records nothing into the events."""
    import torch
    comp, xfer, dt = wl.random_instances(5, 300, 16)
    c, x, d = (torch.from_numpy(a).cuda() for a in (comp, xfer, dt))
    sch = dc.Scheduler(300, 16)
    k0, k1, after = _events(torch, 3)
    assert dc.dc_time_next_pass(k0, k1) == dc.DC_OK
    o = sch.out[0]
    bad = dc.dc_schedule_forward_batch(300, 16, c, x, d, o["makespan"], o["bits"], o["nseg"],
                                       o["status"], sch.workspace, 0)  # workspace too short
    assert bad == dc.DC_ERR_WORKSPACE
    after.record()
    torch.cuda.synchronize()
    before = k1.elapsed_time(after)
    sch.run(0, c, x, d)
    torch.cuda.synchronize()
    assert k1.elapsed_time(after) == pytest.approx(before)
