"""GPU greedy schedulers (Algorithm 1 forward, Algorithm 2 backward) against the
oracle's greedy schedulers, through the C ABI: every decision word and
every makespan bit-exact, faults included.

The oracle enumerates every pair and position (Algorithm 2 costs O(L^3) there,
plus a replay per candidate), so the CNN batches are checked on samples and the
decisions of the whole batch are replayed instead.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
FWD, BWD = 0, 1
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


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _gpu(dc, d, comp, xfer, dt):
    import torch
    B, L = comp.shape
    out = dc.greedy(d, _dev(comp), _dev(xfer), _dev(dt))
    torch.cuda.synchronize()
    W = dc.words(L)
    bits = out["bits"].cpu().numpy().view(np.uint32)[:, :W] if W else np.zeros((B, 0), np.uint32)
    return out["makespan"].cpu().numpy(), bits


def _check(dc, d, comp, xfer, dt, label):
    mk, bits = _gpu(dc, d, comp, xfer, dt)
    exp = oracle.greedy_batch(d, comp, xfer, dt, nthreads=NTHREADS)
    bad = np.nonzero((mk != exp["makespan"]) | (bits != exp["bits"]).any(axis=1))[0]
    assert bad.size == 0, (f"{label}: {bad.size} mismatches, first {bad[0]}: gpu {mk[bad[0]]} "
                           f"{bits[bad[0]]} oracle {exp['makespan'][bad[0]]} {exp['bits'][bad[0]]}")
    return mk, bits


@pytest.mark.parametrize("L", [1, 2, 3, 5, 8, 16, 17, 33, 54, 64, 65, 100])
@pytest.mark.parametrize("kind", ["tie", "uni", "skew"])
def test_greedy_random_parity(dc, L, kind):
    B = {True: 600, False: 150}[L <= 17] + 11
    gen = {"tie": wl.tie_heavy_instances, "uni": wl.random_instances,
           "skew": wl.skewed_instances}[kind]
    comp, xfer, dt = gen(7000 + 13 * L + len(kind), B, L)
    for d in (FWD, BWD):
        _check(dc, d, comp, xfer, dt, f"greedy L={L} {kind} dir={d}")


def test_greedy_faults(dc):
    L, B = 12, 64
    comp, xfer, dt = wl.random_instances(3, B, L, 0, 100_000, 0, 10_000)
    comp[3, 4] = -1
    dt[7] = -2
    xfer[9, 0] = 1 << 52
    comp[11, :] = (1 << 52) // L
    for d in (FWD, BWD):
        mk, bits = _check(dc, d, comp, xfer, dt, f"greedy faults dir={d}")
        assert list(mk[[3, 7, 9, 11]]) == [-3, -3, -4, -4]
        assert not bits[[3, 7, 9, 11]].any()


@pytest.mark.parametrize("name,sample", [("tiny", 4096), ("alexnet", 20000), ("vgg16", 20000),
                                         ("resnet50", 400)])
def test_greedy_configs(dc, name, sample):
    """A sample bit-exact with the oracle; every decision of the batch replays to
    its makespan; no greedy decision beats the DP."""
    import torch
    cfg = wl.config(name)
    prof = {k: v for k, v in dc.profile_gen(cfg).items()}
    torch.cuda.synchronize()
    for d, (c, x) in ((FWD, ("fc", "pt")), (BWD, ("bc", "gt"))):
        out = dc.greedy(d, prof[c], prof[x], prof["dt"])
        dp = dc.schedule(d, prof[c], prof[x], prof["dt"])
        W = dc.words(cfg["L"])
        rep = dc.eval_timeline(d, prof[c], prof[x], prof["dt"], out["bits"][:, :W].contiguous())
        torch.cuda.synchronize()
        assert torch.equal(rep, out["makespan"])
        assert bool((dp["makespan"] <= out["makespan"]).all())
        idx = slice(0, sample)
        h = {k: prof[k][idx].cpu().numpy() for k in (c, x, "dt")}
        exp = oracle.greedy_batch(d, h[c], h[x], h["dt"], nthreads=NTHREADS)
        assert np.array_equal(out["makespan"][idx].cpu().numpy(), exp["makespan"])
        assert np.array_equal(out["bits"][idx, :W].cpu().numpy().view(np.uint32), exp["bits"])
