/*
 * The paper's competing greedy schedulers: TEST INFRASTRUCTURE, like the rest of
 * this directory (only tests/, __graft_entry__.smoke() and bench.py's baseline
 * legs load it; it shares nothing with the CUDA library).
 *
 *  - greedy parameter scheduling of iBatch, forward (Algorithm 1, Sec. II-C);
 *  - greedy gradient scheduling of iPart, backward (Algorithm 2, Sec. II-C).
 *
 * Plain transcriptions in the listings' order: every pair or position is
 * enumerated, every condition and key evaluated with direct range sums.
 * Readings where the listings leave a choice open:
 *   G1 ties: "choose the one with minimum ..." keeps the first candidate in the
 *      listing's enumeration order (x ascending; n ascending);
 *   G2 an empty Options set (no position meets the overlap condition) takes the
 *      position whose slack -- the condition's left side less its right side --
 *      is largest, the one closest to meeting it (G1 on ties);
 *   G3 Algorithm 1 steps 1-4: pairs 1 <= D1 < D2 <= L; among the pairs meeting
 *      the condition: maximum first-segment compute, then minimum first
 *      transfer, then the loop's own key (minimum slack), then G1; with no pair
 *      meeting it, G2 over all pairs; the loop runs while m < L;
 *   G4 iBatch's second, reverse-order forward greedy is not given in the paper:
 *      the forward greedy is Algorithm 1 alone;
 *   G5 Algorithm 2's "estimated total execution time" is f_m (the backward
 *      replay); for L = 1 (no candidate) the decision is the single segment.
 * Decisions use the layout of the rest of the oracle: p[l] (forward) and g[r]
 * (backward, r = number of last layers before the break) for 1 <= l, r <= L-1.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "dynacomm_oracle.h"

/* v[a] + ... + v[b] over 1-based layers (0 when a > b) */
static int64_t range_sum(const int64_t *v, int32_t a, int32_t b)
{
    int64_t s = 0;
    for (int32_t l = a; l <= b; l++) s += v[l - 1];
    return s;
}

void orc_greedy_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt, uint8_t *p)
{
    for (int32_t l = 0; l <= L; l++) p[l] = 0;
    if (L < 2) return;

    /* steps 1-4: the first two decomposition positions */
    int found = 0;
    int32_t d1b = 0, d2b = 0;
    int64_t kc = 0, kx = 0, ks = 0;
    for (int32_t d1 = 1; d1 < L; d1++) {
        for (int32_t d2 = d1 + 1; d2 <= L; d2++) {
            int64_t comp1 = range_sum(fc, 1, d1);
            int64_t slack = dt + range_sum(pt, d1 + 1, d2) - comp1;
            if (slack < 0) continue; /* not in S2 */
            int64_t xfer1 = dt + range_sum(pt, 1, d1);
            int better = !found || comp1 > kc || (comp1 == kc && xfer1 < kx) ||
                         (comp1 == kc && xfer1 == kx && slack < ks);
            if (better) {
                found = 1;
                d1b = d1;
                d2b = d2;
                kc = comp1;
                kx = xfer1;
                ks = slack;
            }
        }
    }
    if (!found) { /* G2 over all pairs */
        int first = 1;
        for (int32_t d1 = 1; d1 < L; d1++) {
            for (int32_t d2 = d1 + 1; d2 <= L; d2++) {
                int64_t slack = dt + range_sum(pt, d1 + 1, d2) - range_sum(fc, 1, d1);
                if (first || slack > ks) {
                    first = 0;
                    d1b = d1;
                    d2b = d2;
                    ks = slack;
                }
            }
        }
    }
    p[d1b] = 1;
    if (d2b < L) p[d2b] = 1;

    /* steps 5-17 */
    int32_t n = d1b, m = d2b;
    while (m < L) {
        int64_t comp = range_sum(fc, n + 1, m);
        int32_t j = -1;
        int64_t best = 0;
        for (int32_t x = m + 1; x <= L; x++) {
            int64_t slack = dt + range_sum(pt, m + 1, x) - comp;
            if (slack >= 0 && (j < 0 || slack < best)) {
                j = x;
                best = slack;
            }
        }
        if (j < 0) { /* G2 */
            for (int32_t x = m + 1; x <= L; x++) {
                int64_t slack = dt + range_sum(pt, m + 1, x) - comp;
                if (j < 0 || slack > best) {
                    j = x;
                    best = slack;
                }
            }
        }
        n = m;
        m = j;
        if (m < L) p[m] = 1;
    }
}

void orc_greedy_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt, uint8_t *g)
{
    for (int32_t r = 0; r <= L; r++) g[r] = 0;
    if (L < 2) return;
    uint8_t *cand = (uint8_t *)malloc((size_t)L + 1);
    int have = 0;
    int64_t best_t = 0;
    for (int32_t n = 2; n <= L; n++) {
        memset(cand, 0, (size_t)L + 1);
        /* decomposition position q (2 <= q <= L) breaks between layers q and
         * q-1, after the last L+1-q layers */
        cand[L + 1 - n] = 1;
        int32_t m = n;
        int64_t k = 1;
        do {
            int64_t link = k * dt + range_sum(gt, m, L);
            int32_t j = -1;
            int64_t best = 0;
            for (int32_t x = 1; x <= m - 1; x++) {
                int64_t slack = link - range_sum(bc, x, m - 1);
                if (slack >= 0 && (j < 0 || slack < best)) {
                    j = x;
                    best = slack;
                }
            }
            if (j < 0) { /* G2 */
                for (int32_t x = 1; x <= m - 1; x++) {
                    int64_t slack = link - range_sum(bc, x, m - 1);
                    if (j < 0 || slack > best) {
                        j = x;
                        best = slack;
                    }
                }
            }
            if (j > 1) cand[L + 1 - j] = 1;
            m = j;
            k += 1;
        } while (m != 1);
        int64_t t = orc_replay_backward(L, bc, gt, dt, cand);
        if (!have || t < best_t) {
            have = 1;
            best_t = t;
            memcpy(g, cand, (size_t)L + 1);
        }
    }
    free(cand);
}
