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
