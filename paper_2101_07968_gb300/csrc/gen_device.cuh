// Device side of the seeded profile generator, shared by the generator kernel
// and the fused generate-and-solve kernel: every value is a pure function of
// (seed, global instance index, field, layer), so any kernel can regenerate any
// instance's rows. Integer-only: SplitMix64 draws, multiply-high uniform
// integers, piecewise-linear log-uniform knots built on the host in double
// precision, and exact ceiling divisions by multiply-high with a per-divisor
// reciprocal.
#pragma once

#include "common.cuh"

namespace dc {

constexpr int kKnots = 512;
constexpr int kFixedMax = 1024;

struct GenParams {
    int64_t batch, inst0;
    uint64_t seed;
    int32_t L, layer_mode, rate_dist, bw_dist, bwd_mult, bits;
    int64_t rate_lo, rate_hi, bw_lo, bw_hi, dt_lo, dt_hi;
    int64_t params_lo, params_hi, flops_lo, flops_hi;
    int64_t rate_knots[kKnots + 1], bw_knots[kKnots + 1];
    // per-layer tables: fixed params/FLOPs, or log-uniform knots of the draws
    int64_t layer0[kFixedMax], layer1[kFixedMax];
};
static_assert(sizeof(GenParams) < 32000, "kernel parameter block limit");

__device__ __forceinline__ uint64_t splitmix(uint64_t seed, uint64_t ctr)
{
    uint64_t z = seed + (ctr + 1) * 0x9e3779b97f4a7c15ull;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t counter(int64_t gi, int field, int layer)
{
    return (uint64_t(gi) << 20) | (uint64_t(field) << 12) | uint64_t(layer);
}

__device__ __forceinline__ int64_t uniform_int(int64_t lo, int64_t hi, uint64_t r)
{
    return lo + int64_t(__umul64hi(r, uint64_t(hi - lo) + 1u));
}

template <typename Tab>
__device__ __forceinline__ int64_t loguniform(const Tab &knots, uint64_t r)
{
    const int j = int(r >> 55);
    const uint64_t f = (r >> 23) & 0xffffffffull;
    const int64_t t0 = knots[j], t1 = knots[j + 1];
    return t0 + int64_t((uint64_t(t1 - t0) * f) >> 32);
}

// Exact ceil(a / d) for 0 <= a < 2^62 and 1 <= d < 2^31 with m = floor((2^64-1)/d)
// precomputed once per divisor: q = mulhi(a, m) is floor(a/d) or one less,
// because a*m/2^64 >= a/d - a*(1 + ((2^64-1) mod d))/(d*2^64) > a/d - 1/4; one
// remainder step makes it exact.
__device__ __forceinline__ void floor_div(uint64_t a, uint64_t d, uint64_t m, uint64_t &q,
                                          uint64_t &r)
{
    q = __umul64hi(a, m);
    r = a - q * d;
    if (r >= d) {
        ++q;
        r -= d;
    }
}

__device__ __forceinline__ uint64_t ceil_div(uint64_t a, uint64_t d, uint64_t m)
{
    uint64_t q = __umul64hi(a, m);
    uint64_t r = a - q * d;
    if (r >= d) {
        ++q;
        r -= d;
    }
    return q + (r != 0 ? 1u : 0u);
}

// Host: config checks, and the generator's parameter block for a valid config.
dc_status check_profile_cfg(const dc_profile_cfg *c);
void fill_gen_params(const dc_profile_cfg *c, GenParams &g);

// Generate-and-solve for 1 <= L <= 16 (dp_fused.cu): outputs [2][batch], forward
// first; workspace: fused_workspace_bytes(batch).
size_t fused_workspace_bytes(int64_t batch);
cudaError_t launch_fused(const GenParams &g, int64_t *makespan, uint32_t *bits, int32_t *nseg,
                         int32_t *status, void *workspace, cudaStream_t stream);

// Rate, bandwidth and latency of global instance gi, with the reciprocals of
// rate and bandwidth for ceil_div.
struct InstanceDraws {
    uint64_t rate, mrate, bw, mbw;
    int64_t dt;
};

template <typename Tab>
__device__ __forceinline__ InstanceDraws instance_draws(const GenParams &g, const Tab &rate_knots,
                                                        const Tab &bw_knots, int64_t gi)
{
    const uint64_t r_rate = splitmix(g.seed, counter(gi, 0, 0));
    const uint64_t r_bw = splitmix(g.seed, counter(gi, 1, 0));
    const int64_t rate = g.rate_dist == DC_DIST_LOGUNIFORM ? loguniform(rate_knots, r_rate)
                                                           : uniform_int(g.rate_lo, g.rate_hi, r_rate);
    const int64_t bw = g.bw_dist == DC_DIST_LOGUNIFORM ? loguniform(bw_knots, r_bw)
                                                       : uniform_int(g.bw_lo, g.bw_hi, r_bw);
    InstanceDraws d;
    d.rate = uint64_t(rate);
    d.mrate = ~uint64_t(0) / uint64_t(rate);
    d.bw = uint64_t(bw);
    d.mbw = ~uint64_t(0) / uint64_t(bw);
    d.dt = uniform_int(g.dt_lo, g.dt_hi, splitmix(g.seed, counter(gi, 2, 0)));
    return d;
}

// Parameters and FLOPs of layer l (0-based) of global instance gi.
template <typename Tab>
__device__ __forceinline__ void layer_draws(const GenParams &g, const Tab &l0, const Tab &l1,
                                            int64_t gi, int l, int64_t &params, int64_t &flops)
{
    if (g.layer_mode == DC_LAYERS_FIXED) {
        params = l0[l];
        flops = l1[l];
    } else {
        const uint64_t rp = splitmix(g.seed, counter(gi, 3, l));
        const uint64_t rf = splitmix(g.seed, counter(gi, 4, l));
        if (g.layer_mode == DC_LAYERS_LOGUNIFORM) {
            params = loguniform(l0, rp);
            flops = loguniform(l1, rf);
        } else {
            params = uniform_int(g.params_lo, g.params_hi, rp);
            flops = uniform_int(g.flops_lo, g.flops_hi, rf);
        }
    }
}

// Forward compute, backward compute and transfer cost (pt = gt) of one layer.
__device__ __forceinline__ void layer_costs(const GenParams &g, const InstanceDraws &d,
                                            int64_t params, int64_t flops, int64_t &fc,
                                            int64_t &bc, int64_t &xfer)
{
    xfer = int64_t(ceil_div(uint64_t(g.bits) * 1000u * uint64_t(params), d.bw, d.mbw));
    if (g.bwd_mult == 2) {
        // flops = q*rate + r (0 <= r < rate): ceil(flops/rate) = q + (r > 0) and
        // ceil(2*flops/rate) = 2q + ceil(2r/rate) = 2q + (r > 0) + (2r > rate)
        uint64_t q, r;
        floor_div(uint64_t(flops), d.rate, d.mrate, q, r);
        const uint64_t up = r != 0 ? 1u : 0u;
        fc = int64_t(q + up);
        bc = int64_t(2 * q + up + (2 * r > d.rate ? 1u : 0u));
    } else {
        fc = int64_t(ceil_div(uint64_t(flops), d.rate, d.mrate));
        bc = int64_t(ceil_div(uint64_t(g.bwd_mult) * uint64_t(flops), d.rate, d.mrate));
    }
}

}  // namespace dc
