"""The checked build (-DDC_CHECKED) on the GPU: every kernel family with its
index checks compiled in, on inputs that reach each of them (short L, looped L,
the CTA-per-instance work list, the deep-chain kernel with 1 and 8 warps per
instance, the forward E form, faults), gives outputs bit-identical to the
normal build's and records no failed check. The checks count a failure and skip
the access instead of trapping, so a wrong index shows up here as a count.

Run the whole GPU suite against the checked build with
`python -m paper_2101_07968_gb300.build --checked` and then
`DC_CHECKED=1 python -m pytest tests -m gpu`; this file then also reads the
counters that the suite left behind.
"""
import os

import numpy as np
import pytest

from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
FWD, BWD = 0, 1


@pytest.fixture(scope="module")
def libs():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build, dynacomm
    normal = build.build()
    checked = build.build(checked=True)
    yield dynacomm, normal, checked
    dynacomm._lib = None
    dynacomm.LIB_PATH = normal if os.environ.get("DC_CHECKED") != "1" else checked


def _use(dc, path):
    dc._lib = None
    dc.LIB_PATH = path
    dc.lib()


def _cases():
    yield "vgg16", wl.with_batch(wl.config("vgg16"), 20_000)
    yield "resnet50", wl.with_batch(wl.config("resnet50"), 4_000)
    yield "deep1", wl.with_batch(wl.config("deepchain"), 2_000)   # one warp per instance
    yield "deep8", wl.with_batch(wl.config("deepchain"), 40)      # eight warps per instance


def _solve(dc, prof, L):
    import torch
    out = {}
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        r = dc.schedule(d, prof[c], prof[x], prof["dt"])
        W = dc.words(L)
        rep = dc.eval_timeline(d, prof[c], prof[x], prof["dt"], r["bits"][:, :max(W, 1)].contiguous())
        torch.cuda.synchronize()
        out[d] = {k: v.cpu().numpy() for k, v in r.items()}
        out[d]["replay"] = rep.cpu().numpy()
    return out


def test_counters_left_by_the_checked_suite(libs):
    """Under DC_CHECKED=1 the whole suite ran on the checked build: no check failed."""
    dc, normal, checked = libs
    if os.environ.get("DC_CHECKED") != "1":
        pytest.skip("the suite ran on the normal build")
    _use(dc, checked)
    fails = dc.checked_failures()
    assert all(c == 0 for c, _ in fails.values()), fails


def test_checked_build_matches_and_records_nothing(libs):
    import torch
    dc, normal, checked = libs
    inputs = []
    _use(dc, normal)
    for name, cfg in _cases():
        prof = dc.profile_gen(cfg)
        prof = {k: v.clone() for k, v in prof.items()}
        if name in ("vgg16", "resnet50"):  # a few faults and 64-bit instances
            prof["pt"][5, 0] = 1 << 40
            prof["fc"][9, 1] = -1
            prof["dt"][13] = 1 << 51
        inputs.append((name, cfg["L"], prof))
    # instances with a large total compute: the 32/64-bit templates of the work list
    comp, xfer, dt = wl.random_instances(7, 300, 300, 0, 1 << 26, 0, 1 << 20)
    t = lambda a: torch.from_numpy(a).cuda()
    inputs.append(("wide300", 300, {"fc": t(comp), "bc": t(comp), "pt": t(xfer), "gt": t(xfer),
                                     "dt": t(dt)}))
    want = {name: _solve(dc, prof, L) for name, L, prof in inputs}
    _use(dc, checked)
    dc.checked_failures(reset=True)
    for name, L, prof in inputs:
        got = _solve(dc, prof, L)
        for d in (FWD, BWD):
            for k, v in want[name][d].items():
                assert np.array_equal(got[d][k], v), (name, d, k)
    fails = dc.checked_failures()
    assert all(c == 0 for c, _ in fails.values()), fails
