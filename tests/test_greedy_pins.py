"""Pins of the oracle's competing greedy schedulers (Algorithms 1 and 2).

The greedy algorithms have no closed form; they are pinned by hand-worked
examples (tests/golden/greedy_worked.txt, worked by hand from the greedy rules
of Sec. II-C), by a second, independent oracle (oracle/pyref.py, explicit
candidate lists and its own replay), by special cases whose outcome the
algorithms fix, and by
the optimality of the DP (no greedy decision beats Algorithms 3/4).
"""
import os

import numpy as np
import pytest

import oracle
from oracle import pyref
from paper_2101_07968_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "greedy_worked.txt")


def _golden():
    rows = []
    for line in open(GOLDEN):
        if not line.strip() or line.startswith("#"):
            continue
        head, comp, xfer, bits, mk = [p.split() for p in line.split("|")]
        rows.append((head[0], int(head[1]), int(head[2]), [int(v) for v in comp],
                     [int(v) for v in xfer], [int(v) for v in bits], int(mk[0])))
    return rows


@pytest.mark.parametrize("case", range(4))
def test_worked_examples(case):
    d, L, dt, comp, xfer, bits, mk = _golden()[case]
    direction = 0 if d == "forward" else 1
    dec = (oracle.greedy_forward(xfer, comp, dt) if direction == 0
           else oracle.greedy_backward(comp, xfer, dt))
    assert list(dec[1:L]) == bits
    out = oracle.greedy_batch(direction, np.array([comp]), np.array([xfer]), np.array([dt]))
    assert out["makespan"][0] == mk


@pytest.mark.parametrize("L", range(1, 11))
@pytest.mark.parametrize("kind", ["tie", "uni", "skew"])
def test_two_oracles_agree(L, kind):
    gen = {"tie": wl.tie_heavy_instances, "uni": wl.random_instances,
           "skew": wl.skewed_instances}[kind]
    comp, xfer, dt = gen(97 * L + len(kind), 120, L)
    for i in range(len(dt)):
        c, x, d = [int(v) for v in comp[i]], [int(v) for v in xfer[i]], int(dt[i])
        assert list(oracle.greedy_forward(x, c, d)) == pyref.forward_bits(pyref.greedy_forward(x, c, d), L)
        g = oracle.greedy_backward(c, x, d)
        D = pyref.greedy_backward(c, x, d)
        assert list(g) == pyref.backward_bits(D, L)
        assert oracle.replay_batch(1, comp[i:i + 1], xfer[i:i + 1], dt[i:i + 1],
                                   _pack(g, L))[0] == pyref.backward_time(c, x, d, D)


def _pack(d, L):
    W = (L - 1 + 31) // 32
    w = np.zeros((1, W), np.uint32)
    for l in range(1, L):
        if d[l]:
            w[0, (l - 1) // 32] |= np.uint32(1 << ((l - 1) % 32))
    return w


def test_short_models():
    """L = 1: the single segment; L = 2: both algorithms end at layer by layer."""
    assert list(oracle.greedy_forward([5], [7], 3)) == [0, 0]
    assert list(oracle.greedy_backward([5], [7], 3)) == [0, 0]
    comp, xfer, dt = wl.random_instances(4, 200, 2, 0, 1000, 0, 1000)
    for i in range(200):
        assert oracle.greedy_forward(xfer[i], comp[i], dt[i])[1] == 1
        assert oracle.greedy_backward(comp[i], xfer[i], dt[i])[1] == 1


def test_huge_latency():
    """dt above every compute sum: every pair and position meets the overlap
    condition. Forward: the largest first-segment compute is D1 = L-1, so D_f =
    [0, L-1, L]. Backward: each candidate's chain ends at once (D = [L+1, n, 1]),
    and Algorithm 2 keeps the single break with the least f_m, lowest n first."""
    for L in (3, 5, 8):
        comp, xfer, _ = wl.random_instances(8 + L, 100, L, 1, 1000, 0, 0)
        dt = np.full(100, 10 ** 9, np.int64)
        for i in range(100):
            p = oracle.greedy_forward(xfer[i], comp[i], dt[i])
            assert list(p[1:L]) == [0] * (L - 2) + [1]
            g = oracle.greedy_backward(comp[i], xfer[i], dt[i])
            best, best_r = None, None
            for n in range(2, L + 1):  # position n breaks after the last L+1-n layers
                d = np.zeros(L + 1, np.uint8)
                d[L + 1 - n] = 1
                t = oracle.replay_batch(1, comp[i:i + 1], xfer[i:i + 1], dt[i:i + 1], _pack(d, L))[0]
                if best is None or t < best:
                    best, best_r = t, L + 1 - n
            exp = [0] * (L + 1)
            exp[best_r] = 1
            assert list(g) == exp


@pytest.mark.parametrize("name", ["tiny", "vgg16", "resnet50"])
def test_dp_never_worse_than_greedy(name):
    """Algorithms 3/4 are optimal (Sec. IV-B3): no greedy decision has a smaller
    makespan, and the greedy makespan is f_m of its own decision."""
    cfg = wl.with_batch(wl.config(name), 400)
    prof = oracle.profile_gen(cfg)
    for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        gr = oracle.greedy_batch(d, prof[c], prof[x], prof["dt"], nthreads=4)
        dp = oracle.schedule_batch(d, prof[c], prof[x], prof["dt"], nthreads=4)
        assert (dp["makespan"] <= gr["makespan"]).all()
        rep = oracle.replay_batch(d, prof[c], prof[x], prof["dt"], gr["bits"], nthreads=4)
        assert np.array_equal(rep, gr["makespan"])
