"""Generate-and-solve (dc_schedule_generated_batch) against the unfused path:
dc_profile_gen, then dc_schedule_forward_batch and dc_schedule_backward_batch on
the profiles it wrote. Every output bit-exact; a sample also against the oracle
directly. Configurations cover the fixed CNN shapes, per-instance layer draws,
short L, latencies large enough that every instance takes the 64-bit list pass,
batches that mix 32-bit and listed instances (some listed in one direction
only, through large latencies or large compute), and optima deeper than the
kept traceback columns.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
NTHREADS = os.cpu_count() or 1


@pytest.fixture(scope="module")
def dc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build, dynacomm
    build.build()
    dynacomm.lib()
    return dynacomm


def _configs():
    tiny = wl.config("tiny")
    out = [("tiny", tiny), ("alexnet", wl.config("alexnet")), ("vgg16", wl.config("vgg16")),
           ("draws16", wl.lsweep_config(16, 100_003))]
    for L in (1, 2, 5):
        c = wl.with_batch(tiny, 5_001)
        c["L"] = L
        out.append((f"tiny_L{L}", c))
    big = wl.with_batch(tiny, 20_011, inst0=777)
    big.update(dt_lo=10 ** 9, dt_hi=10 ** 12)  # bounds above 2^31: the list pass
    out.append(("huge_dt", big))
    # bounds on both sides of 2^31 - 1: 32-bit and listed instances side by side,
    # and a few listed in the backward direction only (its compute is larger)
    mixed = wl.with_batch(tiny, 20_011, inst0=555)
    mixed.update(dt_lo=2 * 10 ** 8, dt_hi=4 * 10 ** 8)
    out.append(("mixed_dt", mixed))
    # the same through large compute at ordinary latencies: optima of 2-5 segments
    # on both sides of the bound, compute costs above 2^31 / L (the 64-bit prefix)
    heavy = wl.with_batch(tiny, 20_011, inst0=999)
    heavy.update(flops_lo=10 ** 9, flops_hi=10 ** 12, rate_lo=10 ** 3, rate_hi=10 ** 4)
    out.append(("mixed_wide", heavy))
    # optima of up to 8 segments: those deeper than the kept columns are listed
    deep = wl.with_batch(tiny, 20_011, inst0=333)
    deep.update(flops_lo=10 ** 9, flops_hi=10 ** 11, rate_lo=10 ** 3, rate_hi=10 ** 4)
    out.append(("deep_s", deep))
    return out


@pytest.mark.parametrize("name,cfg", _configs(), ids=[n for n, _ in _configs()])
def test_fused_equals_unfused(dc, name, cfg):
    import torch
    B, L = cfg["batch"], cfg["L"]
    W = dc.words(L)
    fused = dc.GeneratedScheduler(cfg).run()
    prof = dc.profile_gen(cfg)
    torch.cuda.synchronize()
    for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        ref = dc.schedule(d, prof[c], prof[x], prof["dt"])
        torch.cuda.synchronize()
        for k in ("makespan", "nseg", "status"):
            assert torch.equal(fused[k][d], ref[k]), (name, d, k)
        if W:
            assert torch.equal(fused["bits"][d][:, :W], ref["bits"][:, :W]), (name, d, "bits")
    # a sample straight against the oracle
    n = min(B, 3000)
    po = oracle.profile_gen(wl.with_batch(cfg, n, inst0=cfg.get("inst0", 0)))
    for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        exp = oracle.schedule_batch(d, po[c], po[x], po["dt"], nthreads=NTHREADS)
        assert np.array_equal(fused["makespan"][d][:n].cpu().numpy(), exp["makespan"])
        assert np.array_equal(fused["nseg"][d][:n].cpu().numpy(), exp["nseg"])
        if W:
            assert np.array_equal(fused["bits"][d][:n, :W].cpu().numpy().view(np.uint32), exp["bits"])
        if name == "deep_s":  # some tracebacks need more than the kept columns 1..4
            assert int(exp["nseg"].max()) > 5
    if name == "huge_dt":  # the list pass ran: some bound exceeds 2^31
        assert int((L * po["dt"] + po["fc"].sum(1)).max()) > 2 ** 31
    if name in ("mixed_dt", "mixed_wide"):  # the batch holds all three kinds of instance
        f = {k: prof[k].cpu().numpy() for k in ("fc", "pt", "bc", "gt", "dt")}

        def wide(c, x):  # the capped bound of the shifted 32-bit form
            tc = f[c].sum(1)
            return L * f["dt"] + tc + np.minimum(f[x], tc[:, None]).sum(1) > 2 ** 31 - 1

        wf, wb = wide("fc", "pt"), wide("bc", "gt")
        assert (~wf & ~wb).any() and (wf & wb).any() and (wb & ~wf).any()


def test_fused_errors(dc):
    import torch
    cfg = wl.config("deepchain")  # L = 1024: above the fused path's 16
    assert dc.dc_schedule_generated_workspace_bytes(16, 1024) == 0
    ws = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    z = torch.empty(2 * 16 * 40, dtype=torch.int64, device="cuda")
    st = dc.dc_schedule_generated_batch(wl.with_batch(cfg, 16), z, z, None, None, ws, ws.numel())
    assert st == dc.DC_ERR_BAD_SHAPE
    small = wl.with_batch(wl.config("vgg16"), 1000)
    need = dc.dc_schedule_generated_workspace_bytes(1000, 16)
    assert need >= 256 + 8 * 1000
    st = dc.dc_schedule_generated_batch(small, z, z, None, None, ws, need - 1)
    assert st == dc.DC_ERR_WORKSPACE
