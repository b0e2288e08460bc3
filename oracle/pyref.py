"""Second, independent transcription of Algorithms 3 and 4 in pure Python.

TEST INFRASTRUCTURE ONLY (same import rule as the C oracle). It exists to
cross-check the C oracle on tie-heavy small inputs, where the exact boundaries
depend on the listings' tie-break rules rather than on the optimum alone. Sums
are taken directly over their index ranges as Eq. 8 / Eq. 9 print them, with no
prefix arrays, so the two transcriptions share neither code nor structure.
Use for L up to about 30.
"""
from __future__ import annotations

INF = float("inf")


def forward(pt, fc, dt):
    """Algorithm 3 with Eq. 8. pt, fc: per-layer lists (layer l at index l-1).

    Returns (T_forward, p as a list of L+1 ints, number of enabled positions)."""
    L = len(pt)
    F = [[INF] * (L + 1) for _ in range(L + 1)]
    path = [[-1] * (L + 1) for _ in range(L + 1)]
    F[0][0] = 0
    for m in range(1, L + 1):
        for n in range(1, m + 1):
            for k in range(0, m):
                if F[k][n - 1] == INF:
                    continue
                pull_done = n * dt + sum(pt[l - 1] for l in range(1, m + 1))
                t_lst = max(F[k][n - 1], pull_done)
                cost = t_lst + sum(fc[l - 1] for l in range(k + 1, m + 1))
                if F[m][n] <= cost:
                    continue
                F[m][n] = cost
                path[m][n] = k
    best, steps = INF, -1
    for k in range(1, L + 1):
        if best <= F[L][k]:
            continue
        best, steps = F[L][k], k
    p = [0] * (L + 1)
    cur = L
    for k in range(1, steps + 1):
        tmp = path[cur][steps - k + 1]
        if 1 <= tmp <= L - 1:
            p[tmp] = 1
        cur = tmp
    return best, p, steps


def backward(bc, gt, dt):
    """Algorithm 4 with Eq. 9. bc, gt: per-layer lists in layer order 1..L."""
    L = len(bc)
    B = [[INF] * (L + 1) for _ in range(L + 1)]
    path = [[-1] * (L + 1) for _ in range(L + 1)]
    B[0][0] = 0
    for m in range(1, L + 1):
        for n in range(1, m + 1):
            for k in range(0, m):
                if B[k][n - 1] == INF:
                    continue
                comp_done = sum(bc[l - 1] for l in range(L - m + 1, L + 1))
                t_lst = max(B[k][n - 1], comp_done)
                cost = t_lst + dt + sum(gt[l - 1] for l in range(L - m + 1, L - k + 1))
                if B[m][n] <= cost:
                    continue
                B[m][n] = cost
                path[m][n] = k
    best, steps = INF, -1
    for k in range(1, L + 1):
        if best <= B[L][k]:
            continue
        best, steps = B[L][k], k
    g = [0] * (L + 1)
    cl = 1
    for k in range(1, steps + 1):
        tmp = path[L - cl + 1][steps - k + 1]
        if 1 <= tmp <= L - 1:
            g[tmp] = 1
        cl = L - tmp + 1
    return best, g, steps


# ---------------------------------------------------------------------------
# The competing greedy schedulers (Algorithms 1 and 2), transcribed again with
# explicit candidate lists and key tuples. Readings (same as the C oracle's
# G1-G5): ties keep the first candidate of the listing's enumeration; an empty
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
