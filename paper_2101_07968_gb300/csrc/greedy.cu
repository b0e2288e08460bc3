// The paper's competing schedulers as batched kernels (Sec. II-C): greedy
// parameter scheduling of iBatch (Algorithm 1, forward) and greedy gradient
// scheduling of iPart (Algorithm 2, backward), one instance per thread.
//
// Readings where the listings leave a choice open (the same as the oracle's):
//  * ties in "choose the one with minimum ..." keep the first candidate of the
//    listing's enumeration (positions ascending, Algorithm 2's n ascending);
//  * an empty Options set takes the position with the largest slack (the
//    condition's left side less its right side), the one closest to meeting it;
//  * Algorithm 1's first pair (D1, D2): among the pairs meeting the condition,
//    maximum first-segment compute, then minimum first transfer, then minimum
//    slack; with none meeting it, the largest slack; the loop runs while m < L;
//  * Algorithm 2's "estimated total execution time" is f_m, the backward replay.
//
// Prefix sums are non-decreasing, which makes each choice a short monotone scan
// instead of the listings' enumerations:
//  * forward: D1 is valid iff dt + P[L] - P[D1] >= FC[D1] (take D2 = L), a prefix
//    of [1, L-1]; its largest FC is at the last valid D1 and the smallest P among
//    equal FC at the first D1 of that plateau (a lower D1 never has a larger
//    minimum slack). D2, and every later step, is the first x whose transfer
//    covers the compute (minimum slack), else the first x reaching P[L];
//  * backward: the positions x meeting k*dt + GT[m..L] >= BC[x..m-1] form a
//    suffix [x*, m-1]; the minimum slack is at x*, found by one downward scan;
//    with none, the largest slack is at m-1, extended down over zero-compute
//    layers (ties keep the lowest x).
// Segment boundaries come in time order, so f_m is accumulated on the fly
// (forward: end_s = max(end_{s-1}, s*dt + P[b_s]) + FC[b_s] - FC[b_{s-1}];
// backward: link = max(link, BC[q..L]) + dt + GT of the segment).
#include "common.cuh"

namespace dc {
namespace {

__device__ __forceinline__ int instance_check(int L, const int64_t *c, const int64_t *x, int64_t dt,
                                              uint64_t &sc, uint64_t &sx)
{
    bool neg = dt < 0, big = (dt >> 52) != 0;
    sc = 0;
    sx = 0;
    for (int l = 0; l < L; ++l) {
        const int64_t cv = __ldg(c + l), xv = __ldg(x + l);
        neg |= (cv < 0) | (xv < 0);
        big |= ((cv | xv) >> 52) != 0;
        sc += uint64_t(cv);
        sx += uint64_t(xv);
    }
    if (neg) return DC_ERR_NEGATIVE;
    if (big || exceeds_range(L, dt, sc, sx)) return DC_ERR_RANGE;
    return DC_OK;
}

__device__ __forceinline__ void set_bit(uint32_t *w, int l) { w[(l - 1) >> 5] |= 1u << ((l - 1) & 31); }

// Algorithm 1. fc, pt: the instance's rows (layer l at index l-1).
__device__ void greedy_fwd(int L, const int64_t *fc, const int64_t *pt, int64_t dt, int64_t Ptot,
                           uint32_t *bits, int64_t *makespan)
{
    if (L < 2) {  // one segment
        *makespan = dt + __ldg(pt) + __ldg(fc);
        return;
    }
    // steps 1-4: D1 (and the prefix sums at it)
    int d1 = 0, plateau = 1;
    int64_t P = 0, FC = 0, P1 = 0, FC1 = 0, plateauP = 0, plateauFC = 0;
    for (int d = 1; d < L; ++d) {
        const int64_t f = __ldg(fc + d - 1);
        if (d == 1 || f != 0) {  // FC grows: a new plateau starts at d
            plateau = d;
            plateauP = P + __ldg(pt + d - 1);
            plateauFC = FC + f;
        }
        P += __ldg(pt + d - 1);
        FC += f;
        if (dt + Ptot - P < FC) break;  // valid D1 form a prefix
        d1 = plateau;
        P1 = plateauP;
        FC1 = plateauFC;
    }
    int64_t Pm, FCm;
    int m;
    if (d1 > 0) {
        // D2: the first x > D1 with dt + P[x] - P[D1] >= FC[D1] (exists: x = L)
        Pm = P1;
        FCm = FC1;
        m = d1;
        do {
            ++m;
            Pm += __ldg(pt + m - 1);
            FCm += __ldg(fc + m - 1);
        } while (dt + Pm - P1 < FC1);
    } else {
        // no pair meets the condition: the largest slack is D1 = 1 and D2 the
        // first x > 1 with P[x] = P[L]
        d1 = 1;
        P1 = __ldg(pt);
        FC1 = __ldg(fc);
        Pm = P1;
        FCm = FC1;
        m = 1;
        do {
            ++m;
            Pm += __ldg(pt + m - 1);
            FCm += __ldg(fc + m - 1);
        } while (Pm < Ptot);
    }
    // f_m over the segments fixed so far: [1, D1], [D1+1, D2]
    int64_t end = dt + P1 + FC1;
    end = max(end, 2 * dt + Pm) + (FCm - FC1);
    int s = 2;
    set_bit(bits, d1);
    int n = d1;
    int64_t FCn = FC1;
    while (m < L) {
        set_bit(bits, m);
        const int64_t cover = FCm - FCn;
        // the first x > m whose transfer covers `cover`; else the first x with
        // P[x] = P[L] (largest slack)
        int j = m, jg = -1;
        int64_t Px = Pm, FCx = FCm, Pg = 0, FCg = 0;
        bool ok = false;
        while (j < L) {
            ++j;
            Px += __ldg(pt + j - 1);
            FCx += __ldg(fc + j - 1);
            if (jg < 0 && Px == Ptot) {
                jg = j;
                Pg = Px;
                FCg = FCx;
            }
            if (dt + Px - Pm >= cover) {
                ok = true;
                break;
            }
        }
        if (!ok) {
            j = jg;
            Px = Pg;
            FCx = FCg;
        }
        ++s;
        end = max(end, int64_t(s) * dt + Px) + (FCx - FCm);
        n = m;
        FCn = FCm;
        m = j;
        Pm = Px;
        FCm = FCx;
    }
    (void)n;
    *makespan = end;
}

// One chain of Algorithm 2 from second position n; returns its f_m and, when
// `bits` is given, sets its decision there. BCs, GTs: sums of bc, gt over
// layers n..L.
__device__ int64_t greedy_bwd_chain(int L, const int64_t *bc, const int64_t *gt, int64_t dt,
                                    int n, int64_t BCs, int64_t GTs, uint32_t *bits)
{
    // segment 1 holds layers L..n
    int64_t link = BCs + dt + GTs;  // f_m so far
    if (bits) set_bit(bits, L + 1 - n);
    int m = n;
    int64_t k = 1;
    while (m > 1) {
        const int64_t limit = k * dt + GTs;  // the listing's link estimate
        // x* = the lowest x in [1, m-1] with BC[x..m-1] <= limit
        int64_t s = 0, g = 0;
        int x = m;
        while (x > 1) {
            const int64_t b = __ldg(bc + x - 2);
            if (s + b > limit) break;
            s += b;
            g += __ldg(gt + x - 2);
            --x;
        }
        if (x == m) {  // none: the largest slack, x = m-1 and the zero-compute layers below
            s = __ldg(bc + m - 2);
            g = __ldg(gt + m - 2);
            x = m - 1;
            while (x > 1 && __ldg(bc + x - 2) == 0) {
                g += __ldg(gt + x - 2);
                --x;
            }
        }
        // segment m-1..x
        BCs += s;
        GTs += g;
        link = max(link, BCs) + dt + g;
        if (bits && x > 1) set_bit(bits, L + 1 - x);
        m = x;
        k += 1;
    }
    return link;
}

// Algorithm 2. bc, gt: the instance's rows in layer order 1..L.
__device__ void greedy_bwd(int L, const int64_t *bc, const int64_t *gt, int64_t dt, int64_t BCtot,
                           int64_t GTtot, uint32_t *bits, int64_t *makespan)
{
    if (L < 2) {
        *makespan = BCtot + dt + GTtot;
        return;
    }
    int best_n = 2;
    int64_t best = 0, BCs = BCtot, GTs = GTtot;
    for (int n = 2; n <= L; ++n) {
        BCs -= __ldg(bc + n - 2);  // layers n..L
        GTs -= __ldg(gt + n - 2);
        const int64_t t = greedy_bwd_chain(L, bc, gt, dt, n, BCs, GTs, nullptr);
        if (n == 2 || t < best) {
            best = t;
            best_n = n;
        }
    }
    BCs = BCtot;
    GTs = GTtot;
    for (int n = 2; n <= best_n; ++n) {
        BCs -= __ldg(bc + n - 2);
        GTs -= __ldg(gt + n - 2);
    }
    greedy_bwd_chain(L, bc, gt, dt, best_n, BCs, GTs, bits);
    *makespan = best;
}

template <bool FWD>
__global__ void __launch_bounds__(128) greedy_kernel(int64_t batch, int L,
                                                     const int64_t *__restrict__ comp,
                                                     const int64_t *__restrict__ xfer,
                                                     const int64_t *__restrict__ dt,
                                                     int64_t *__restrict__ makespan,
                                                     uint32_t *__restrict__ bits)
{
    const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= batch) return;
    const int W = words_for(L);
    uint32_t *w = bits + i * W;
    for (int q = 0; q < W; ++q) w[q] = 0u;
    const int64_t *c = comp + i * L, *x = xfer + i * L;
    const int64_t dti = __ldg(dt + i);
    uint64_t sc, sx;
    const int st = instance_check(L, c, x, dti, sc, sx);
    if (st != DC_OK) {
        makespan[i] = -int64_t(st);
        return;
    }
    if (FWD)
        greedy_fwd(L, c, x, dti, int64_t(sx), w, makespan + i);
    else
        greedy_bwd(L, c, x, dti, int64_t(sc), int64_t(sx), w, makespan + i);
}

}  // namespace
}  // namespace dc

extern "C" dc_status dc_greedy_forward_batch(int64_t batch, int32_t L, const int64_t *fc,
                                             const int64_t *pt, const int64_t *dt,
                                             int64_t *makespan, uint32_t *bits,
                                             cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_greedy_forward_batch");
    if (batch < 0 || L < 1 || L > DC_L_MAX || batch > int64_t(0xffffffffll)) return DC_ERR_BAD_SHAPE;
    if (batch == 0) return DC_OK;
    if (!fc || !pt || !dt || !makespan || (!bits && dc::words_for(L) > 0)) return DC_ERR_NULL;
    const unsigned grid = unsigned((batch + 127) / 128);
    dc::greedy_kernel<true><<<grid, 128, 0, stream>>>(batch, L, fc, pt, dt, makespan, bits);
    return cudaGetLastError() == cudaSuccess ? DC_OK : DC_ERR_CUDA;
}

extern "C" dc_status dc_greedy_backward_batch(int64_t batch, int32_t L, const int64_t *bc,
                                              const int64_t *gt, const int64_t *dt,
                                              int64_t *makespan, uint32_t *bits,
                                              cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_greedy_backward_batch");
    if (batch < 0 || L < 1 || L > DC_L_MAX || batch > int64_t(0xffffffffll)) return DC_ERR_BAD_SHAPE;
    if (batch == 0) return DC_OK;
    if (!bc || !gt || !dt || !makespan || (!bits && dc::words_for(L) > 0)) return DC_ERR_NULL;
    const unsigned grid = unsigned((batch + 127) / 128);
    dc::greedy_kernel<false><<<grid, 128, 0, stream>>>(batch, L, bc, gt, dt, makespan, bits);
    return cudaGetLastError() == cudaSuccess ? DC_OK : DC_ERR_CUDA;
}
