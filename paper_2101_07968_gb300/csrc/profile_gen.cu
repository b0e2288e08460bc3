// Seeded synthetic profile generator (stand-in for the real-time profiler of
// Sec. IV-A, which derives pt, fc, bc, gt and dt from a framework's profiler).
//
// Every value is a pure function of (seed, global instance index, field, layer),
// so any sub-range of a batch can be generated on its own. Integer-only on the
// device: SplitMix64 draws, multiply-high uniform integers, piecewise-linear
// log-uniform knots built on the host in double precision, and exact ceiling
// divisions by multiply-high with a per-instance reciprocal.
#include <cmath>

#include "common.cuh"

namespace dc {
namespace {

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

__device__ __forceinline__ int64_t loguniform(const int64_t *knots, uint64_t r)
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

// Warp-level tiles of 32 consecutive instances. Phase 1: lane j draws rate,
// bandwidth and latency of instance j and forms the two division magic numbers
// (32 instances' 64-bit divisions run side by side). Phase 2: the warp walks the
// tile's 32*L (instance, layer) elements 32 at a time, so the four output rows
// are written coalesced. Only __syncwarp between the phases.
constexpr int kGenWarps = 8;

__global__ void __launch_bounds__(32 * kGenWarps)
    gen_kernel(const __grid_constant__ GenParams g, int64_t *__restrict__ fc,
               int64_t *__restrict__ pt, int64_t *__restrict__ bc, int64_t *__restrict__ gt,
               int64_t *__restrict__ dt)
{
    __shared__ int64_t s_rate[kKnots + 1], s_bw[kKnots + 1];
    __shared__ int64_t s_l0[kFixedMax], s_l1[kFixedMax];
    __shared__ uint64_t s_inst[kGenWarps][4][32];  // rate, magic(rate), bw, magic(bw)
    const int L = g.L, t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nl = g.layer_mode == DC_LAYERS_FIXED ? L
                   : (g.layer_mode == DC_LAYERS_LOGUNIFORM ? kKnots + 1 : 0);
    for (int j = t; j <= kKnots; j += blockDim.x) {
        s_rate[j] = g.rate_knots[j];
        s_bw[j] = g.bw_knots[j];
    }
    for (int j = t; j < nl; j += blockDim.x) {
        s_l0[j] = g.layer0[j];
        s_l1[j] = g.layer1[j];
    }
    __syncthreads();
    uint64_t(*si)[32] = s_inst[warp];
    const int step_i = 32 / L, step_l = 32 % L;  // advance of (instance, layer) per 32 elements
    const int64_t tiles = (g.batch + 31) / 32;
    for (int64_t tile = int64_t(blockIdx.x) * kGenWarps + warp; tile < tiles;
         tile += int64_t(gridDim.x) * kGenWarps) {
        const int64_t i0 = tile * 32;
        const int n_inst = int(g.batch - i0 < 32 ? g.batch - i0 : 32);
        __syncwarp();  // previous tile done with si
        if (lane < n_inst) {
            const int64_t i = i0 + lane, gi = g.inst0 + i;
            const uint64_t r_rate = splitmix(g.seed, counter(gi, 0, 0));
            const uint64_t r_bw = splitmix(g.seed, counter(gi, 1, 0));
            const int64_t rate = g.rate_dist == DC_DIST_LOGUNIFORM
                                     ? loguniform(s_rate, r_rate)
                                     : uniform_int(g.rate_lo, g.rate_hi, r_rate);
            const int64_t bw = g.bw_dist == DC_DIST_LOGUNIFORM
                                   ? loguniform(s_bw, r_bw)
                                   : uniform_int(g.bw_lo, g.bw_hi, r_bw);
            si[0][lane] = uint64_t(rate);
            si[1][lane] = ~uint64_t(0) / uint64_t(rate);
            si[2][lane] = uint64_t(bw);
            si[3][lane] = ~uint64_t(0) / uint64_t(bw);
            dt[i] = uniform_int(g.dt_lo, g.dt_hi, splitmix(g.seed, counter(gi, 2, 0)));
        }
        __syncwarp();
        const int total = n_inst * L;
        int il = lane / L, l = lane - (lane / L) * L;
        for (int e = lane; e < total; e += 32) {
            const int64_t gi = g.inst0 + i0 + il;
            int64_t params, flops;
            if (g.layer_mode == DC_LAYERS_FIXED) {
                params = s_l0[l];
                flops = s_l1[l];
            } else {
                const uint64_t rp = splitmix(g.seed, counter(gi, 3, l));
                const uint64_t rf = splitmix(g.seed, counter(gi, 4, l));
                if (g.layer_mode == DC_LAYERS_LOGUNIFORM) {
                    params = loguniform(s_l0, rp);
                    flops = loguniform(s_l1, rf);
                } else {
                    params = uniform_int(g.params_lo, g.params_hi, rp);
                    flops = uniform_int(g.flops_lo, g.flops_hi, rf);
                }
            }
            const uint64_t rate = si[0][il], mr = si[1][il];
            const uint64_t bw = si[2][il], mb = si[3][il];
            const uint64_t xfer = ceil_div(uint64_t(g.bits) * 1000u * uint64_t(params), bw, mb);
            const int64_t o = i0 * L + e;
            fc[o] = int64_t(ceil_div(uint64_t(flops), rate, mr));
            bc[o] = int64_t(ceil_div(uint64_t(g.bwd_mult) * uint64_t(flops), rate, mr));
            pt[o] = int64_t(xfer);
            gt[o] = int64_t(xfer);
            il += step_i;
            l += step_l;
            if (l >= L) {
                l -= L;
                ++il;
            }
        }
    }
}

int64_t knot(int64_t lo, int64_t hi, int j)
{
    if (j <= 0) return lo;
    if (j >= kKnots) return hi;
    const double x = double(j) / 512.0;
    const double y = std::log(double(hi) / double(lo));
    return int64_t(std::llround(double(lo) * std::exp(x * y)));
}

void knots(int64_t lo, int64_t hi, int64_t *out)
{
    for (int j = 0; j <= kKnots; ++j) out[j] = knot(lo, hi, j);
}

bool in_range(int64_t lo, int64_t hi, int64_t min_lo, int64_t max_hi)
{
    return lo >= min_lo && lo <= hi && hi <= max_hi;
}

}  // namespace

dc_status check_profile_cfg(const dc_profile_cfg *c)
{
    const int64_t cap = int64_t(1) << 40, rcap = (int64_t(1) << 31) - 1;
    if (c->L < 1 || c->L > DC_L_MAX || c->batch < 0 || c->inst0 < 0) return DC_ERR_BAD_CONFIG;
    if (c->inst0 + c->batch > (int64_t(1) << 44)) return DC_ERR_BAD_CONFIG;
    if (c->bwd_flops_mult < 1 || c->bwd_flops_mult > 16) return DC_ERR_BAD_CONFIG;
    if (c->bits_per_param < 1 || c->bits_per_param > 64) return DC_ERR_BAD_CONFIG;
    if (!in_range(c->rate_lo, c->rate_hi, 1, rcap) || !in_range(c->bw_lo, c->bw_hi, 1, rcap))
        return DC_ERR_BAD_CONFIG;
    if (!in_range(c->dt_lo, c->dt_hi, 0, cap)) return DC_ERR_BAD_CONFIG;
    if (c->rate_dist < 0 || c->rate_dist > 1 || c->bw_dist < 0 || c->bw_dist > 1)
        return DC_ERR_BAD_CONFIG;
    if (c->layer_mode == DC_LAYERS_FIXED) {
        if (c->L > kFixedMax) return DC_ERR_BAD_CONFIG;
        if (!c->fixed_params || !c->fixed_flops) return DC_ERR_NULL;
        for (int l = 0; l < c->L; ++l)
            if (!in_range(c->fixed_params[l], c->fixed_params[l], 0, cap) ||
                !in_range(c->fixed_flops[l], c->fixed_flops[l], 0, cap))
                return DC_ERR_BAD_CONFIG;
    } else if (c->layer_mode == DC_LAYERS_UNIFORM || c->layer_mode == DC_LAYERS_LOGUNIFORM) {
        const int64_t min_lo = c->layer_mode == DC_LAYERS_LOGUNIFORM ? 1 : 0;
        if (!in_range(c->params_lo, c->params_hi, min_lo, cap) ||
            !in_range(c->flops_lo, c->flops_hi, min_lo, cap))
            return DC_ERR_BAD_CONFIG;
    } else {
        return DC_ERR_BAD_CONFIG;
    }
    return DC_OK;
}

cudaError_t launch_gen(const dc_profile_cfg *c, int64_t *fc, int64_t *pt, int64_t *bc,
                       int64_t *gt, int64_t *dt, cudaStream_t stream)
{
    static thread_local GenParams g;  // 25 KB: kept off the caller's stack
    g.batch = c->batch;
    g.inst0 = c->inst0;
    g.seed = c->seed;
    g.L = c->L;
    g.layer_mode = c->layer_mode;
    g.rate_dist = c->rate_dist;
    g.bw_dist = c->bw_dist;
    g.bwd_mult = c->bwd_flops_mult;
    g.bits = c->bits_per_param;
    g.rate_lo = c->rate_lo;
    g.rate_hi = c->rate_hi;
    g.bw_lo = c->bw_lo;
    g.bw_hi = c->bw_hi;
    g.dt_lo = c->dt_lo;
    g.dt_hi = c->dt_hi;
    g.params_lo = c->params_lo;
    g.params_hi = c->params_hi;
    g.flops_lo = c->flops_lo;
    g.flops_hi = c->flops_hi;
    if (c->rate_dist == DC_DIST_LOGUNIFORM) knots(c->rate_lo, c->rate_hi, g.rate_knots);
    if (c->bw_dist == DC_DIST_LOGUNIFORM) knots(c->bw_lo, c->bw_hi, g.bw_knots);
    if (c->layer_mode == DC_LAYERS_FIXED) {
        for (int l = 0; l < c->L; ++l) {
            g.layer0[l] = c->fixed_params[l];
            g.layer1[l] = c->fixed_flops[l];
        }
    } else if (c->layer_mode == DC_LAYERS_LOGUNIFORM) {
        knots(c->params_lo, c->params_hi, g.layer0);
        knots(c->flops_lo, c->flops_hi, g.layer1);
    }
    const int64_t tiles = (c->batch + 31) / 32;
    int64_t blocks = (tiles + kGenWarps - 1) / kGenWarps;
    if (blocks > 152 * 8) blocks = 152 * 8;
    gen_kernel<<<unsigned(blocks), 32 * kGenWarps, 0, stream>>>(g, fc, pt, bc, gt, dt);
    return cudaGetLastError();
}

}  // namespace dc
