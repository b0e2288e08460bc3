// Generate-and-solve for 1 <= L <= 16 (dc_schedule_generated_batch): the short-L
// passes of dp_small.cu with each tile's rows drawn inside the kernel by the
// profile generator's device functions instead of being read from memory.
#include "dp_small.cuh"

namespace dc {
namespace {

// ---------------------------------------------------------------------------
// Generate and solve in one pass (no profile round trip through HBM): each lane
// draws its instance's rows with the profile generator's own device functions
// into its row of the staging area, then the tile is solved as in dp_small.cu.
// Both directions come from one draw of the rows (fused_pair_kernel): the forward
// and backward U, V rows are derived from the staged rows and saved in the lane's
// slice, and one copy of the solve, with the direction as a runtime argument,
// runs once per direction (two unrolled copies overflow the instruction cache).
// Each direction has its own list pass, which regenerates the listed instances'
// rows.
// workspace: [0, 256) the two list counters and the tile ticket,
// [256, 256 + 8 batch) the two lists, then the generator's tables
inline size_t fused_tables_offset(int64_t batch) { return (256 + 8 * size_t(batch) + 255) / 256 * 256; }

struct FusedOut {
    int64_t *makespan[2];
    uint32_t *bits[2];
    int32_t *nseg[2], *status[2];
    uint32_t *wide_count[2], *wide_list[2];
    uint32_t *ticket;  // tiles handed out (zero before the launch)
};

// The generator's lookup tables, copied once per call from the parameter block
// into the workspace: lanes index them with their own draws, which global loads
// serve in parallel where the parameter (constant) path serialises them.
struct GenTables {
    int64_t rate[kKnots + 1], bw[kKnots + 1], l0[kFixedMax], l1[kFixedMax];
};

__global__ void __launch_bounds__(256) copy_tables_kernel(const __grid_constant__ GenParams g,
                                                          GenTables *t)
{
    for (int j = threadIdx.x; j <= kKnots; j += blockDim.x) {
        t->rate[j] = g.rate_knots[j];
        t->bw[j] = g.bw_knots[j];
    }
    for (int j = threadIdx.x; j < kFixedMax; j += blockDim.x) {
        t->l0[j] = g.layer0[j];
        t->l1[j] = g.layer1[j];
    }
}

// Shared memory of a warp of the pair pass, per lane (lane-interleaved words):
// the backward U, V at [0, 2(L+1)), then the table, whose first 2(L+1) words hold
// the forward U, V until the forward solve loads them; the tile's staged rows
// (compute forward, compute backward, transfer, at the padded stride) overlap it
// all, being read before any of it is written.
template <int L>
struct Pair32 {
    static constexpr int kUV = 2 * (L + 1);
    static constexpr int kTab = Tab32<L>::kWords > kUV ? Tab32<L>::kWords : kUV;
    static constexpr int kSlotBytes = 32 * (kUV + kTab) * 4;
    static constexpr int kRowsBytes = 3 * 32 * Tab32<L>::kStride * 8;
    static constexpr int kBytes = kRowsBytes > kSlotBytes ? kRowsBytes : kSlotBytes;
};

// Both directions of each instance from one draw of its rows.
template <int L>
__global__ void __launch_bounds__(32, DC_SMALL_MINB)
    fused_pair_kernel(const __grid_constant__ GenParams g, const GenTables *t, const FusedOut o)
{
    using K = Tab32<L>;
    using P = Pair32<L>;
    constexpr int W = (L - 1 + 31) / 32;
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x;
    int64_t *stF = reinterpret_cast<int64_t *>(smem) + lane * K::kStride;
    int64_t *stB = stF + 32 * K::kStride;
    int64_t *stX = stB + 32 * K::kStride;
    int32_t *uvb = reinterpret_cast<int32_t *>(smem) + lane;  // backward U, V
    int32_t *lw = uvb + 32 * P::kUV;                           // table; forward U, V first
    const int64_t tiles = (g.batch + 31) / 32;
    pdl_trigger();
    auto solve_tile = [&](int64_t tile) {
        const int64_t i = tile * 32 + lane;
        const bool active = i < g.batch;
        const int64_t gi = g.inst0 + i;
        InstanceDraws d = {};
        if (active) d = instance_draws(g, t->rate, t->bw, gi);
        __syncwarp();  // every lane is done with the area (the previous tile's table)
        if (active) {
            // rolled from kSplitMinL on: unrolled, the generator's divisions and the
            // DP overflow the instruction cache
#pragma unroll (L >= kSplitMinL ? 1 : L)
            for (int l = 0; l < L; ++l) {
                int64_t params, flops, f, b, x;
                layer_draws(g, t->l0, t->l1, gi, l, params, flops);
                layer_costs(g, d, params, flops, f, b, x);
                stF[l] = f;
                stB[l] = b;
                stX[l] = x;
            }
        }
        const int64_t dti = active ? d.dt : 0;
        uint64_t xraw[2];
        bool wide[2];
        int st[2];
        {
            int32_t Uf[L + 1], Vf[L + 1], Ub[L + 1], Vb[L + 1];
            row_uv<L, true>(stF, stX, dti, Uf, Vf, xraw[0], wide[0], st[0]);
            row_uv<L, false>(stB, stX, dti, Ub, Vb, xraw[1], wide[1], st[1]);
            __syncwarp();  // rows read: the lanes' slices may be written
#pragma unroll
            for (int m = 0; m <= L; ++m) {
                lw[32 * m] = Uf[m];
                lw[32 * (L + 1 + m)] = Vf[m];
                uvb[32 * m] = Ub[m];
                uvb[32 * (L + 1 + m)] = Vb[m];
            }
        }
        if (!active) return;
#pragma unroll 1
        for (int dir = 0; dir < 2; ++dir) {
            const bool fwd = dir == 0;
            const int32_t *uv = fwd ? lw : uvb;
            int32_t U[L + 1], V[L + 1];
#pragma unroll
            for (int m = 0; m <= L; ++m) {
                U[m] = uv[32 * m];
                V[m] = uv[32 * (L + 1 + m)];
            }
            if (st[dir] != DC_OK) {
                write_failure(st[dir], i, W, o.makespan[dir], o.bits[dir], o.nseg[dir],
                              o.status[dir]);
            } else if (wide[dir] || !solve_uv<L>(fwd, U, V, int32_t(dti), xraw[dir], lw, i,
                                                 o.makespan[dir], o.bits[dir], o.nseg[dir],
                                                 o.status[dir])) {
                const uint32_t at = atomicAdd(o.wide_count[dir], 1u);
                if (DC_CHECK(int64_t(at) < g.batch)) o.wide_list[dir][at] = uint32_t(i);
            }
        }
    };
    if constexpr (L >= kSplitMinL) {
        // tiles from a ticket, the next claimed while this one is solved
        auto claim = [&]() {
            uint32_t v = 0;
            if (lane == 0) v = atomicAdd(o.ticket, 1u);
            return v;
        };
        int64_t tile = int64_t(__shfl_sync(0xffffffffu, claim(), 0));
        while (tile < tiles) {
            const uint32_t next_raw = claim();
            solve_tile(tile);
            tile = int64_t(__shfl_sync(0xffffffffu, next_raw, 0));
        }
    } else {
        for (int64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x) solve_tile(tile);
    }
}

// 64-bit pass over one direction's list, rows regenerated.
template <int L, bool FWD>
__global__ void __launch_bounds__(32)
    fused_list_kernel(const __grid_constant__ GenParams g, const GenTables *t, const FusedOut o)
{
    constexpr int dir = FWD ? 0 : 1;
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x;
    uint64_t *lw = reinterpret_cast<uint64_t *>(smem) + lane;
    pdl_wait();  // the passes ahead of this one have finished
    const int64_t count = int64_t(*o.wide_count[dir]);
    for (int64_t j = int64_t(blockIdx.x) * 32 + lane; j - lane < count; j += int64_t(gridDim.x) * 32) {
        if (j >= count) continue;
        const int64_t i = int64_t(o.wide_list[dir][j]);
        const int64_t gi = g.inst0 + i;
        const InstanceDraws d = instance_draws(g, t->rate, t->bw, gi);
        uint64_t Pc[L + 1], Px[L + 1], xraw;
        bool neg = false, big = false;  // checked by the dense pass
        row_prefix<L, FWD>(
            [&](int col, int64_t &cv, int64_t &xv) {
                int64_t params, flops, f, b, x;
                layer_draws(g, t->l0, t->l1, gi, col, params, flops);
                layer_costs(g, d, params, flops, f, b, x);
                cv = FWD ? f : b;
                xv = x;
            },
            Pc, Px, xraw, neg, big);
        solve<L, FWD, uint64_t, L>(Pc, Px, d.dt, xraw - Px[L], lw, i, o.makespan[dir],
                                   o.bits[dir], o.nseg[dir], o.status[dir]);
    }
}

template <int L, bool FWD>
cudaError_t launch_fused_list(const GenParams &g, const GenTables *t, const FusedOut &o,
                              cudaStream_t stream)
{
    using K64 = Small<L, uint64_t, L>;
    static DeviceCache attr;  // the list kernel's shared-memory limit, raised once per device
    int done = 0;
    cudaError_t ae = attr.get(done, [](int &v) {
        v = 1;
        return cudaFuncSetAttribute(fused_list_kernel<L, FWD>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, K64::kTableBytes);
    });
    if (ae != cudaSuccess) return ae;
    int64_t lgrid = (g.batch + 31) / 32;
    if (lgrid > int64_t(sm_count()) * 4) lgrid = int64_t(sm_count()) * 4;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(unsigned(lgrid));
    lc.blockDim = dim3(32);
    lc.dynamicSmemBytes = K64::kTableBytes;
    lc.stream = stream;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, fused_list_kernel<L, FWD>, g, t, o);
}

template <int L>
cudaError_t launch_fused_L(const GenParams &g, const GenTables *t, const FusedOut &o,
                           cudaStream_t stream)
{
    static DeviceCache resident;  // single-warp CTAs of the pair kernel per SM
    int per_sm = 0;
    cudaError_t le = resident.get(per_sm, [](int &n) {
        cudaError_t e = cudaFuncSetAttribute(fused_pair_kernel<L>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             Pair32<L>::kBytes);
        if (e != cudaSuccess) return e;
        return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fused_pair_kernel<L>, 32,
                                                             Pair32<L>::kBytes);
    });
    if (le != cudaSuccess) return le;
    const int64_t tiles = (g.batch + 31) / 32;
    int64_t grid = int64_t(sm_count()) * per_sm;
    if (grid > tiles) grid = tiles;
    fused_pair_kernel<L><<<unsigned(grid), 32, Pair32<L>::kBytes, stream>>>(g, t, o);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    e = launch_fused_list<L, true>(g, t, o, stream);
    if (e != cudaSuccess) return e;
    return launch_fused_list<L, false>(g, t, o, stream);
}

}  // namespace

size_t fused_workspace_bytes(int64_t batch) { return fused_tables_offset(batch) + sizeof(GenTables); }

// Generate-and-solve for 1 <= L <= 16: outputs [2][batch] (forward first).
cudaError_t launch_fused(const GenParams &g, int64_t *makespan, uint32_t *bits, int32_t *nseg,
                         int32_t *status, void *workspace, cudaStream_t stream)
{
    const int64_t B = g.batch;
    const int W = words_for(g.L);
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    FusedOut o;
    for (int d = 0; d < 2; ++d) {
        o.makespan[d] = makespan + d * B;
        o.bits[d] = bits + d * B * W;
        o.nseg[d] = nseg ? nseg + d * B : nullptr;
        o.status[d] = status ? status + d * B : nullptr;
        o.wide_count[d] = reinterpret_cast<uint32_t *>(ws) + d;
        o.wide_list[d] = reinterpret_cast<uint32_t *>(ws + 256) + d * B;
    }
    o.ticket = reinterpret_cast<uint32_t *>(ws) + 2;
    cudaError_t e = cudaMemsetAsync(ws, 0, 3 * sizeof(uint32_t), stream);
    if (e != cudaSuccess) return e;
    GenTables *t = reinterpret_cast<GenTables *>(ws + fused_tables_offset(B));
    copy_tables_kernel<<<1, 256, 0, stream>>>(g, t);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
#define DC_FUSED_CASE(LL) \
    case LL: return launch_fused_L<LL>(g, t, o, stream);
    switch (g.L) {
        DC_FUSED_CASE(1) DC_FUSED_CASE(2) DC_FUSED_CASE(3) DC_FUSED_CASE(4)
        DC_FUSED_CASE(5) DC_FUSED_CASE(6) DC_FUSED_CASE(7) DC_FUSED_CASE(8)
        DC_FUSED_CASE(9) DC_FUSED_CASE(10) DC_FUSED_CASE(11) DC_FUSED_CASE(12)
        DC_FUSED_CASE(13) DC_FUSED_CASE(14) DC_FUSED_CASE(15) DC_FUSED_CASE(16)
        default: return cudaErrorInvalidValue;
    }
#undef DC_FUSED_CASE
}

}  // namespace dc

DC_CHECKED_EXPORT(dp_fused)
