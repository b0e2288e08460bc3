"""The barrier discipline checked by running the kernels with their block size
permuted (compute-sanitizer's race check is closed on this machine).

DC_BLOCK_WARPS=1|2|4|8 makes the looped kernel (17 <= L <= 256), the deep-chain
kernel (L > 256) and the CTA-per-instance kernel of the work lists run with that
many warps per CTA. A missing __syncwarp / __syncthreads, or an index that
assumes one block size, shows up as outputs that change with it: every output
word must be identical for every block size, and equal to the oracle's.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
FWD, BWD = 0, 1
WARPS = (1, 2, 4, 8)


@pytest.fixture(scope="module")
def dc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build, dynacomm
    build.build()
    dynacomm.lib()
    return dynacomm


def _run(dc, d, comp, xfer, dt):
    import torch
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    out = dc.schedule(d, t(comp), t(xfer), t(dt))
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _wide(seed, B, L):
    """Skewed instances, a third of them with values beyond 32 bits, so that the
    work list (the CTA-per-instance kernel) has instances to solve."""
    comp, xfer, dt = wl.skewed_instances(seed, B, L)
    rng = np.random.default_rng(seed)
    wide = np.arange(B) % 3 == 0
    comp[wide] = comp[wide] * 3 + rng.integers(1 << 26, 1 << 32, size=(int(wide.sum()), L))
    xfer[wide] = xfer[wide] + rng.integers(1 << 20, 1 << 34, size=(int(wide.sum()), L))
    return comp, xfer, dt


CASES = [
    ("looped L=54", lambda: wl.skewed_instances(501, 700, 54)),
    ("looped L=100 + list", lambda: _wide(502, 300, 100)),
    ("looped L=200", lambda: wl.tie_heavy_instances(503, 200, 200)),
    ("deep L=300 + list", lambda: _wide(504, 120, 300)),
    ("deep L=600", lambda: wl.skewed_instances(505, 60, 600)),
]


@pytest.mark.parametrize("name,make", CASES, ids=[c[0] for c in CASES])
def test_outputs_do_not_depend_on_the_block_size(dc, monkeypatch, name, make):
    comp, xfer, dt = make()
    for d in (FWD, BWD):
        monkeypatch.delenv("DC_BLOCK_WARPS", raising=False)
        ref = _run(dc, d, comp, xfer, dt)
        exp = oracle.schedule_batch(d, comp, xfer, dt, nthreads=os.cpu_count() or 1)
        W = dc.words(comp.shape[1])
        assert np.array_equal(ref["makespan"], exp["makespan"]), (name, d)
        assert np.array_equal(ref["bits"].view(np.uint32)[:, :W], exp["bits"]), (name, d)
        for w in WARPS:
            monkeypatch.setenv("DC_BLOCK_WARPS", str(w))
            got = _run(dc, d, comp, xfer, dt)
            for k in ("makespan", "bits", "nseg", "status"):
                assert np.array_equal(got[k], ref[k]), (name, d, w, k)
    monkeypatch.delenv("DC_BLOCK_WARPS", raising=False)
