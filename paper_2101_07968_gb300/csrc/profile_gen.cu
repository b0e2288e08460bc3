// Seeded synthetic profile generator (stand-in for the real-time profiler of
// Sec. IV-A, which derives pt, fc, bc, gt and dt from a framework's profiler).
//
// Every value is a pure function of (seed, global instance index, field, layer),
// so any sub-range of a batch can be generated on its own. Integer-only on the
// device: SplitMix64 draws, multiply-high uniform integers, piecewise-linear
// log-uniform knots built on the host in double precision, and exact ceiling
// divisions by multiply-high with a per-instance reciprocal.
#include <cmath>

#include "gen_device.cuh"

namespace dc {
namespace {

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
            const int64_t i = i0 + lane;
            const InstanceDraws d = instance_draws(g, s_rate, s_bw, g.inst0 + i);
            si[0][lane] = d.rate;
            si[1][lane] = d.mrate;
            si[2][lane] = d.bw;
            si[3][lane] = d.mbw;
            dt[i] = d.dt;
        }
        __syncwarp();
        const int total = n_inst * L;
        int il = lane / L, l = lane - (lane / L) * L;
        for (int e = lane; e < total; e += 32) {
            int64_t params, flops;
            layer_draws(g, s_l0, s_l1, g.inst0 + i0 + il, l, params, flops);
            InstanceDraws d;
            d.rate = si[0][il];
            d.mrate = si[1][il];
            d.bw = si[2][il];
            d.mbw = si[3][il];
            int64_t f, b, x;
            layer_costs(g, d, params, flops, f, b, x);
            const int64_t o = i0 * L + e;
            fc[o] = f;
            bc[o] = b;
            pt[o] = x;
            gt[o] = x;
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

void fill_gen_params(const dc_profile_cfg *c, GenParams &g)
{
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
}

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
    fill_gen_params(c, g);
    const int64_t tiles = (c->batch + 31) / 32;
    int64_t blocks = (tiles + kGenWarps - 1) / kGenWarps;
    if (blocks > 152 * 8) blocks = 152 * 8;
    gen_kernel<<<unsigned(blocks), 32 * kGenWarps, 0, stream>>>(g, fc, pt, bc, gt, dt);
    return cudaGetLastError();
}

}  // namespace dc
