"""A second, independent oracle for the two dynamic programs, in pure Python.

TEST INFRASTRUCTURE ONLY (same import rule as the C oracle). It exists to
cross-check the C oracle on small, tie-heavy inputs, where the exact boundaries
depend on which of several optima is returned rather than on the optimum alone.

It is written differently from the C oracle on purpose: top-down, as a
memoised recursion over sub-problems (m layers, n segments) of Sec. IV-B1, with
every sum taken directly over its index range as Eq. 8 / Eq. 9 print it (no
prefix arrays), and the choice among equal optima made by comparing (value,
index) pairs: the smallest value wins and, on a tie, the smallest index -- the
lowest split k within a cell and the lowest segment count n overall, which is
what the paper's algorithms return (their improvement tests are strict).
Use for L up to about 30.
"""
from __future__ import annotations

import sys
from functools import lru_cache


def _solve(L, last_segment_end):
    """Least finishing time over cuts of all L processed layers, the cut that
    attains it and its segment count. last_segment_end(m, n, k, before) is the
    finishing time of processed layers k+1..m sent as the n-th segment, once the
    first k layers finished (in n-1 segments) at `before`."""
    sys.setrecursionlimit(max(sys.getrecursionlimit(), 10 * L + 100))

    @lru_cache(maxsize=None)
    def best(m, n):
        """(X(m, n), lowest minimising k), or None when m layers cannot form n segments."""
        if n == 0:
            return (0, None) if m == 0 else None
        if m < n:
            return None
        options = []
        for k in range(m):  # the n-th segment holds processed layers k+1..m
            sub = best(k, n - 1)
            if sub is not None:
                options.append((last_segment_end(m, n, k, sub[0]), k))
        return min(options)

    value, s = min((best(L, n)[0], n) for n in range(1, L + 1))
    cut = [0] * (L + 1)
    m, n = L, s
    while n > 0:
        k = best(m, n)[1]
        if 1 <= k <= L - 1:
            cut[k] = 1
        m, n = k, n - 1
    return value, cut, s


def forward(pt, fc, dt):
    """Eq. 8. pt, fc: per-layer lists (layer l at index l-1).

    Returns (T_forward, p as a list of L+1 ints, number of segments)."""
    L = len(pt)

    def end(m, n, k, before):
        arrived = n * dt + sum(pt[l - 1] for l in range(1, m + 1))
        return max(before, arrived) + sum(fc[l - 1] for l in range(k + 1, m + 1))

    return _solve(L, end)


def backward(bc, gt, dt):
    """Eq. 9. bc, gt: per-layer lists in layer order 1..L; sub-problems hold the
    LAST m layers, so g[k] = 1 is a break after the last k layers."""
    L = len(bc)

    def end(m, n, k, before):
        computed = sum(bc[l - 1] for l in range(L - m + 1, L + 1))
        pushed = sum(gt[l - 1] for l in range(L - m + 1, L - k + 1))
        return max(before, computed) + dt + pushed

    return _solve(L, end)


# ---------------------------------------------------------------------------
# The competing greedy schedulers (Algorithms 1 and 2), written again with
# explicit candidate lists and key tuples. Readings (same as the C oracle's
# G1-G5): ties keep the first candidate in enumeration order; an empty
# Options set takes the largest slack; Algorithm 1's first pair orders S2 by
# (max first compute, min first transfer, min slack, enumeration order); the
# estimated total execution time of Algorithm 2 is the backward makespan.

def _rsum(v, a, b):
    """v over layers a..b (1-based, inclusive)."""
    return sum(v[l - 1] for l in range(a, b + 1))


def _pick_min(cands, key):
    """First candidate with the smallest key (enumeration order on ties)."""
    best = None
    for c in cands:
        if best is None or key(c) < key(best):
            best = c
    return best


def greedy_forward(pt, fc, dt):
    """Algorithm 1: returns the decomposition decision D_f = [0, ..., L]."""
    L = len(pt)
    if L < 2:
        return [0, L]
    pairs = [(a, b) for a in range(1, L) for b in range(a + 1, L + 1)]
    slack = lambda a, b: dt + _rsum(pt, a + 1, b) - _rsum(fc, 1, a)
    s2 = [(a, b) for (a, b) in pairs if slack(a, b) >= 0]
    if s2:
        d1, d2 = _pick_min(s2, lambda q: (-_rsum(fc, 1, q[0]), dt + _rsum(pt, 1, q[0]),
                                          slack(*q)))
    else:
        d1, d2 = _pick_min(pairs, lambda q: -slack(*q))
    D = [0, d1, d2]
    n, m = d1, d2
    while m < L:
        cover = _rsum(fc, n + 1, m)
        gap = lambda x: dt + _rsum(pt, m + 1, x) - cover
        xs = list(range(m + 1, L + 1))
        options = [x for x in xs if gap(x) >= 0]
        j = _pick_min(options, gap) if options else _pick_min(xs, lambda x: -gap(x))
        n, m = m, j
        D.append(m)
    return D


def backward_time(bc, gt, dt, positions):
    """Backward makespan of a decomposition [L+1, q1, q2, ..., 1]: segment i
    holds layers q_{i-1}-1 down to q_i; its push waits for its own compute and
    for the previous push (Eq. 2, Eq. 7) and costs dt plus its gradients."""
    L = len(bc)
    link = 0
    for hi, lo in zip(positions[:-1], positions[1:]):
        done = _rsum(bc, lo, L)  # layers L..lo computed back to back
        link = max(link, done) + dt + _rsum(gt, lo, hi - 1)
    return link


def greedy_backward(bc, gt, dt):
    """Algorithm 2: returns the decomposition decision D_b = [L+1, ..., 1]."""
    L = len(bc)
    if L < 2:
        return [L + 1, 1]
    candidates = []
    for n in range(2, L + 1):
        D = [L + 1, n]
        k, m = 1, n
        while True:
            link = k * dt + _rsum(gt, m, L)
            gap = lambda x: link - _rsum(bc, x, m - 1)
            xs = list(range(1, m))
            options = [x for x in xs if gap(x) >= 0]
            j = _pick_min(options, gap) if options else _pick_min(xs, lambda x: -gap(x))
            D.append(j)
            m, k = j, k + 1
            if m == 1:
                break
        candidates.append(D)
    return _pick_min(candidates, lambda D: backward_time(bc, gt, dt, D))


def forward_bits(D, L):
    """p[1..L-1] of a forward decision D_f."""
    p = [0] * (L + 1)
    for q in D[1:-1]:
        p[q] = 1
    return p


def backward_bits(D, L):
    """g[1..L-1] of a backward decision D_b: position q breaks after the last
    L+1-q layers."""
    g = [0] * (L + 1)
    for q in D[1:-1]:
        g[L + 1 - q] = 1
    return g
