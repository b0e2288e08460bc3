"""A whole step captured as a CUDA graph (dynacomm.StepGraph, the two directions on
parallel branches with their own workspaces) gives, replay after replay, exactly
the eager path's profiles, decisions, makespans and replays."""
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


@pytest.mark.parametrize("name,batch", [("tiny", 4096), ("vgg16", 20_011), ("resnet50", 3_001),
                                        ("alexnet", 1), ("deepchain", 300)])
def test_step_graph_equals_eager(dc, name, batch):
    import torch
    cfg = wl.with_batch(wl.config(name), batch, inst0=7)
    g = dc.StepGraph(cfg)
    prof = dc.profile_gen(cfg)
    torch.cuda.synchronize()
    for _ in range(2):
        g.graph.replay()
        torch.cuda.synchronize()
        for k in prof:
            assert torch.equal(g.prof[k], prof[k]), k
        for d, (c, x) in ((dc.FWD, ("fc", "pt")), (dc.BWD, ("bc", "gt"))):
            ref = dc.schedule(d, prof[c], prof[x], prof["dt"])
            torch.cuda.synchronize()
            for k in ("makespan", "nseg", "status", "bits"):
                assert torch.equal(g.sched.out[d][k], ref[k]), (d, k)
            assert torch.equal(g.replay_out[d], ref["makespan"]), d
