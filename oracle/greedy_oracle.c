/*
 * The paper's competing greedy schedulers: TEST INFRASTRUCTURE, like the rest of
 * this directory (only tests/, __graft_entry__.smoke() and bench.py's baseline
 * legs load it; it shares nothing with the CUDA library).
 *
 *  - iBatch's greedy parameter scheduling, forward (Algorithm 1, Sec. II-C);
 *  - iPart's greedy gradient scheduling, backward (Algorithm 2, Sec. II-C).
 *
 * Both are built from one greedy rule, written here from what the section
 * states rather than from the listings' layout: the transfer of the next
 * segment should just cover the compute it overlaps. A candidate position's
 * SLACK is the overlapping transfer time less the compute time; the rule picks
 * the candidate with the least non-negative slack (the tightest cover).
 * Readings where the paper leaves a choice open:
 *   G1 ties keep the first candidate in enumeration order (x ascending for the
 *      next position, the second position n ascending for Algorithm 2's
 *      candidates);
 *   G2 when no candidate has a non-negative slack, the one with the largest
 *      slack (the closest to covering) is taken, G1 on ties;
 *   G3 the first two forward positions 1 <= D1 < D2 <= L: among the pairs whose
 *      slack is non-negative, the largest first-segment compute, then the least
 *      first transfer, then the least slack, then G1; with no such pair, G2
 *      over all pairs; later positions follow the rule while m < L;
 *   G4 iBatch's second, reverse-order forward greedy is not given in the paper:
 *      the forward greedy is Algorithm 1 alone;
 *   G5 Algorithm 2 keeps, among its candidates, the one whose estimated total
 *      execution time is least; that estimate is f_m (the backward replay); for
 *      L = 1 there is no candidate and the decision is the single segment.
 * Decisions use the layout of the rest of the oracle: p[l] (forward) and g[r]
 * (backward, r = number of last layers before the break) for 1 <= l, r <= L-1.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "dynacomm_oracle.h"

/* S[l] = v[1] + ... + v[l] over 1-based layers, S[0] = 0 */
static void layer_prefix(int32_t L, const int64_t *v, int64_t *S)
{
    S[0] = 0;
    for (int32_t l = 1; l <= L; l++) S[l] = S[l - 1] + v[l - 1];
}

/* The greedy rule over candidates 0..count-1 with the given slacks: the least
 * non-negative slack, else (G2) the largest; the first on ties (G1). */
static int32_t greedy_pick(const int64_t *slack, int32_t count)
{
    int32_t pick = -1;
    for (int32_t c = 0; c < count; c++)
        if (slack[c] >= 0 && (pick < 0 || slack[c] < slack[pick])) pick = c;
    if (pick >= 0) return pick;
    pick = 0;
    for (int32_t c = 1; c < count; c++)
        if (slack[c] > slack[pick]) pick = c;
    return pick;
}

void orc_greedy_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt, uint8_t *p)
{
    for (int32_t l = 0; l <= L; l++) p[l] = 0;
    if (L < 2) return;
    int64_t *PT = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + 1));
    int64_t *FC = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + 1));
    int64_t *slack = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + 1));
    layer_prefix(L, pt, PT);
    layer_prefix(L, fc, FC);

    /* G3: the first segment 1..a and the second a+1..b. The second pull
     * (dt + its parameters) overlaps the first segment's compute. */
    int32_t a_best = 0, b_best = 0, have = 0;
    for (int32_t a = 1; a < L; a++)
        for (int32_t b = a + 1; b <= L; b++) {
            const int64_t s = dt + (PT[b] - PT[a]) - FC[a];
            if (s < 0) continue;
            int better = !have;
            if (have) {
                const int64_t s0 = dt + (PT[b_best] - PT[a_best]) - FC[a_best];
                if (FC[a] != FC[a_best])
                    better = FC[a] > FC[a_best]; /* largest first compute */
                else if (PT[a] != PT[a_best])
                    better = PT[a] < PT[a_best]; /* least first transfer dt + PT[a] */
                else
                    better = s < s0; /* least slack */
            }
            if (better) {
                a_best = a;
                b_best = b;
                have = 1;
            }
        }
    if (!have) { /* G2 over every pair */
        int64_t s_best = 0;
        for (int32_t a = 1; a < L; a++)
            for (int32_t b = a + 1; b <= L; b++) {
                const int64_t s = dt + (PT[b] - PT[a]) - FC[a];
                if (!have || s > s_best) {
                    a_best = a;
                    b_best = b;
                    s_best = s;
                    have = 1;
                }
            }
    }
    p[a_best] = 1;
    if (b_best < L) p[b_best] = 1;

    /* later positions: the segment n+1..m computes while the next pull m+1..x
     * travels; x ranges over m+1..L */
    int32_t n = a_best, m = b_best;
    while (m < L) {
        const int32_t count = L - m;
        for (int32_t c = 0; c < count; c++) {
            const int32_t x = m + 1 + c;
            slack[c] = dt + (PT[x] - PT[m]) - (FC[m] - FC[n]);
        }
        const int32_t x = m + 1 + greedy_pick(slack, count);
        n = m;
        m = x;
        if (m < L) p[m] = 1;
    }
    free(PT);
    free(FC);
    free(slack);
}

/* One backward candidate of Algorithm 2: the first push carries layers q..L
 * (q = the second decomposition position, 2 <= q <= L); then, while layers
 * 1..m-1 remain, the k-th push's link time so far (k*dt plus the gradients of
 * layers m..L) overlaps the compute of layers x..m-1, and the rule picks x
 * among 1..m-1. Writes the decision into g (breaks after the last L+1-q and
 * L+1-x layers). */
static void backward_chain(int32_t L, const int64_t *BC, const int64_t *GT, int64_t dt,
                           int32_t q, int64_t *slack, uint8_t *g)
{
    memset(g, 0, (size_t)L + 1);
    g[L + 1 - q] = 1;
    int32_t m = q;
    for (int64_t k = 1; m != 1; k++) {
        const int64_t link = k * dt + (GT[L] - GT[m - 1]);
        const int32_t count = m - 1;
        for (int32_t c = 0; c < count; c++) {
            const int32_t x = 1 + c;
            slack[c] = link - (BC[m - 1] - BC[x - 1]);
        }
        const int32_t x = 1 + greedy_pick(slack, count);
        if (x > 1) g[L + 1 - x] = 1;
        m = x;
    }
}

void orc_greedy_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt, uint8_t *g)
{
    for (int32_t r = 0; r <= L; r++) g[r] = 0;
    if (L < 2) return;
    int64_t *BC = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + 1));
    int64_t *GT = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + 1));
    int64_t *slack = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + 1));
    uint8_t *cand = (uint8_t *)malloc((size_t)L + 1);
    layer_prefix(L, bc, BC);
    layer_prefix(L, gt, GT);
    int64_t t_best = 0;
    for (int32_t q = 2; q <= L; q++) { /* G5, G1: the least f_m, the first q on ties */
        backward_chain(L, BC, GT, dt, q, slack, cand);
        const int64_t t = orc_replay_backward(L, bc, gt, dt, cand);
        if (q == 2 || t < t_best) {
            t_best = t;
            memcpy(g, cand, (size_t)L + 1);
        }
    }
    free(BC);
    free(GT);
    free(slack);
    free(cand);
}
