// Thread-per-instance DynaComm DP for 1 <= L <= 16 (Eq. 8 / Algorithm 3 and
// Eq. 9 / Algorithm 4), fully unrolled at compile time for each L.
//
// Both directions are one template after reindexing the layers into processing
// order (forward: layer 1 first; backward: layer L first):
//   X[m][n] = min_{k} max(X[k][n-1], R(m,n)) - S[k]  + S[m] + c
// forward : R(m,n) = n*dt + sum of the first m pt,  S = prefix of fc, c = 0
// backward: R(m,n) = sum of the last m bc,          S = prefix of gt (last m), c = dt
// with k in [n-1, m-1] (only those X[k][n-1] are finite) and k = 0 for n = 1.
//
// Design (GB300):
//  * one instance per thread, 32 instances per warp, no inter-thread traffic in
//    the fill; the DP column lives in registers with compile-time indices;
//  * the 32-bit pass solves the shifted form (see the block before fill_e in
//    dp_small.cuh): a transition is one add-then-max and two candidates fold
//    into one 3-input min, 1.5 integer-ALU instructions on GB300;
//  * the fill keeps only the minimum VALUE per cell; the traceback recovers
//    Path[m][n] as the lowest k whose candidate equals the cell, which is the k
//    Algorithm 3/4 keeps with its strict-improvement test. A step compares all
//    of its candidates at once (bit mask, lowest set bit), and every step runs
//    the same code (column 1 is read as U less a constant, the other kept
//    columns from the table), so the lanes of a warp at different depths do not
//    split into separate paths. The pass keeps only columns 1..kKeepCols: the
//    traceback of an s-segment optimum reads columns 1..s-1 only, and s is small
//    in practice (2-5 on CNN-shaped profiles); an instance whose s needs a
//    deeper column is re-solved by the 64-bit pass, which keeps every column;
//  * a row whose costs all fit 32 bits (compute below 2^31 / L) gets its prefix
//    sums in 32-bit arithmetic (fast_uv); other rows take the 64-bit prefix,
//    which also classifies bad input;
//  * transfer costs are first capped at the instance's total compute, which
//    changes no decision (see row_prefix); the shifted 32-bit form is exact
//    whenever the capped bound L*dt + sum(capped xfer) + sum(comp) is below
//    2^31. Other instances (and the deep ones above) are appended to a work list
//    that a 64-bit instantiation of the literal template solves afterwards; that
//    pass is launched early and waits in hardware for this one (programmatic
//    dependent launch);
//  * persistent single-warp CTAs walk 32-instance tiles. A tile's rows arrive by
//    cp.async (coalesced 16-byte copies of cost pairs for even L) at a row
//    stride at which every lane reads its own row without bank conflicts
//    (stage_stride); the prefix sums then leave them in registers. Short rows
//    (L < kSplitMinL) stage in the warp's table area, which keeps a warp small
//    (many resident warps) while the next tile is prefetched into L2; longer
//    rows stage beside the table, so that the next tile's copies are in flight
//    while this one is solved, and take their tiles from a ticket (see the
//    kernel).
#include "dp_small.cuh"

namespace dc {
namespace {

// Resident single-warp CTAs per SM the registers must allow: the split design
// is held to 12 by its shared memory, so its registers may grow to that.
__host__ __device__ constexpr int dense_min_ctas(int L) { return L >= kSplitMinL ? 12 : DC_SMALL_MINB; }

// 32-bit pass over the whole batch; persistent single-warp CTAs.
//  * shared design (L < kSplitMinL): a tile's rows are staged in the warp's table
//    area, so a warp holds only max(rows, table) of shared memory and many warps
//    fit an SM; while a tile is solved its successor is prefetched into L2. Tiles
//    are dealt statically (warp w takes w, w + grid, ...): short tiles, for which
//    one atomic per tile on a shared ticket would cost more than the balance gains.
//  * split design (L >= kSplitMinL): the staging lies beside the table, and the
//    copies of the warp's next tile (rows and dt) are issued as soon as this
//    tile's rows are read, so they land while it is solved. Tiles come from an
//    atomic ticket, claimed one tile ahead: warps on a crowded sub-partition
//    progress more slowly than others, and a static deal would leave the SMs
//    emptying out behind the slowest warps.
template <int L, bool FWD>
__global__ void __launch_bounds__(32, dense_min_ctas(L))
    small_dense_kernel(int64_t batch, const int64_t *__restrict__ comp,
                       const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
                       int64_t *__restrict__ makespan, uint32_t *__restrict__ bits,
                       int32_t *__restrict__ nseg, int32_t *__restrict__ status,
                       uint32_t *__restrict__ wide_count, uint32_t *__restrict__ wide_list,
                       bool pairs)
{
    using K = Tab32<L>;
    constexpr int W = (L - 1 + 31) / 32;
    constexpr bool kSplit = L >= kSplitMinL;
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x;
    int32_t *lw = reinterpret_cast<int32_t *>(smem) + lane;
    int64_t *stC = reinterpret_cast<int64_t *>(smem + (kSplit ? K::kBytes : 0));
    int64_t *stX = stC + 32 * K::kStride;
    int64_t *stD = stX + 32 * K::kStride;  // the tile's dt (split design)
    uint32_t *ticket = wide_count + 1;     // tiles handed out (zero before the launch)

    const int64_t tiles = (batch + 31) / 32;
    pdl_trigger();  // the list pass may be scheduled as soon as CTAs of this one exit
    auto rows_of = [&](int64_t t) { return int(batch - t * 32 < 32 ? batch - t * 32 : 32); };
    auto claim = [&]() {
        uint32_t v = 0;
        if (lane == 0) v = atomicAdd(ticket, 1u);
        return v;
    };
    // the solve of one tile's rows, held by each lane in U, V
    auto finish = [&](int64_t i, const int32_t (&U)[L + 1], const int32_t (&V)[L + 1],
                      int64_t dti, uint64_t xraw, bool wide, int st) {
        if (st != DC_OK) {
            write_failure(st, i, W, makespan, bits, nseg, status);
        } else if (wide ||
                   !solve_uv<L>(FWD, U, V, int32_t(dti), xraw, lw, i, makespan, bits, nseg, status)) {
            // 64-bit values, or a traceback deeper than the kept columns: work list
            const uint32_t at = atomicAdd(wide_count, 1u);
            if (DC_CHECK(int64_t(at) < batch)) wide_list[at] = uint32_t(i);
        }
    };

    if constexpr (kSplit) {
        auto stage = [&](int64_t t) {
            const int64_t b = t * 32;
            const int r = rows_of(t);
            if (lane < r) cp_async8(stD + lane, dt + b + lane);
            stage_tile<L>(stC, stX, comp, xfer, b, r, lane, pairs);  // commits the group
        };
        int64_t tile = int64_t(__shfl_sync(0xffffffffu, claim(), 0));
        if (tile >= tiles) return;
        stage(tile);
        uint32_t next_raw = claim();  // claimed a tile ahead: its copies go out mid-tile
        while (tile < tiles) {
            const int64_t i = tile * 32 + lane;
            const bool active = lane < rows_of(tile);
            cp_async_wait_all();
            __syncwarp();
            const int64_t dti = active ? stD[lane] : 0;
            int32_t U[L + 1], V[L + 1];
            uint64_t xraw;
            bool wide;
            int st;
            row_uv<L, FWD>(stC + lane * K::kStride, stX + lane * K::kStride, dti, U, V, xraw,
                           wide, st);
            __syncwarp();  // the staging is read: the next tile's copies may land there
            const int64_t next = int64_t(__shfl_sync(0xffffffffu, next_raw, 0));
            if (next < tiles) {
                stage(next);
                next_raw = claim();
            }
            tile = next;
            if (active) finish(i, U, V, dti, xraw, wide, st);
        }
    } else {
        int64_t tile = blockIdx.x;
        if (tile >= tiles) return;
        for (; tile < tiles; tile += gridDim.x) {
            const int64_t base = tile * 32;
            const int rows = rows_of(tile);
            __syncwarp();  // every lane is done with the table: stage the tile's rows there
            stage_tile<L>(stC, stX, comp, xfer, base, rows, lane, pairs);
            if (tile + gridDim.x < tiles) {  // the warp's next tile into L2, one 128-byte line per lane and array
                const int64_t nbase = (tile + gridDim.x) * 32;
                if (lane * 16 < rows_of(tile + gridDim.x) * L) {
                    asm volatile("prefetch.global.L2 [%0];" ::"l"(comp + nbase * L + lane * 16));
                    asm volatile("prefetch.global.L2 [%0];" ::"l"(xfer + nbase * L + lane * 16));
                }
            }
            const int64_t i = base + lane;
            const bool active = lane < rows;
            const int64_t dti = active ? __ldg(dt + i) : 0;
            cp_async_wait_all();
            __syncwarp();
            int32_t U[L + 1], V[L + 1];
            uint64_t xraw;
            bool wide;
            int st;
            row_uv<L, FWD>(stC + lane * K::kStride, stX + lane * K::kStride, dti, U, V, xraw,
                           wide, st);
            __syncwarp();  // rows read: the lanes' table slices may be written
            if (active) finish(i, U, V, dti, xraw, wide, st);
        }
    }
}

// 64-bit pass over the work list, every column kept.
template <int L, bool FWD>
__global__ void __launch_bounds__(32)
    small_list_kernel(const int64_t *__restrict__ comp, const int64_t *__restrict__ xfer,
                      const int64_t *__restrict__ dt, int64_t *__restrict__ makespan,
                      uint32_t *__restrict__ bits, int32_t *__restrict__ nseg,
                      int32_t *__restrict__ status, const uint32_t *__restrict__ wide_count,
                      const uint32_t *__restrict__ wide_list)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const int lane = threadIdx.x;
    uint64_t *lw = reinterpret_cast<uint64_t *>(smem) + lane;
    pdl_wait();  // the dense pass has finished its list
    const int64_t count = int64_t(*wide_count);
    for (int64_t j = int64_t(blockIdx.x) * 32 + lane; j - lane < count; j += int64_t(gridDim.x) * 32) {
        if (j >= count) continue;
        const int64_t i = int64_t(wide_list[j]);
        const int64_t *crow = comp + i * L;
        const int64_t *xrow = xfer + i * L;
        const int64_t dti = __ldg(dt + i);
        uint64_t Pc[L + 1], Px[L + 1], xraw;
        bool neg = false, big = false;  // checked by the dense pass
        row_prefix<L, FWD>(
            [&](int col, int64_t &cv, int64_t &xv) {
                cv = __ldg(crow + col);
                xv = __ldg(xrow + col);
            },
            Pc, Px, xraw, neg, big);
        solve<L, FWD, uint64_t, L>(Pc, Px, dti, xraw - Px[L], lw, i, makespan, bits, nseg,
                                   status);
    }
}

}  // namespace

int sm_count()
{
    static DeviceCache sms;
    int n = 0;
    const cudaError_t e = sms.get(n, [](int &v) {
        int dev = 0;
        cudaError_t r = cudaGetDevice(&dev);
        if (r == cudaSuccess) r = cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        return r;
    });
    return e == cudaSuccess ? n : 152;
}

namespace {

template <int L, bool FWD>
cudaError_t launch_dir(int64_t batch, const int64_t *comp, const int64_t *xfer,
                       const int64_t *dt, int64_t *makespan, uint32_t *bits, int32_t *nseg,
                       int32_t *status, uint32_t *wide_count, uint32_t *wide_list,
                       const PassEvents &pe, cudaStream_t stream)
{
    using K64 = Small<L, uint64_t, L>;
    constexpr int kSmem = L >= kSplitMinL ? Tab32<L>::kSplitBytes : Tab32<L>::kSharedBytes;
    static DeviceCache resident;  // single-warp CTAs of the dense kernel per SM
    int per_sm = 0;
    cudaError_t le = resident.get(per_sm, [](int &n) {
        cudaError_t e = cudaFuncSetAttribute(small_dense_kernel<L, FWD>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(small_list_kernel<L, FWD>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, K64::kTableBytes);
        if (e != cudaSuccess) return e;
        return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, small_dense_kernel<L, FWD>, 32,
                                                             kSmem);
    });
    if (le != cudaSuccess) return le;
    const int64_t tiles = (batch + 31) / 32;
    int64_t grid = int64_t(sm_count()) * per_sm;
    if (grid > tiles) grid = tiles;
    if (pe.start) {
        const cudaError_t re = cudaEventRecord(pe.start, stream);
        if (re != cudaSuccess) return re;
    }
    small_dense_kernel<L, FWD><<<unsigned(grid), 32, kSmem, stream>>>(
        batch, comp, xfer, dt, makespan, bits, nseg, status, wide_count, wide_list,
        ((reinterpret_cast<uintptr_t>(comp) | reinterpret_cast<uintptr_t>(xfer)) & 15u) == 0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (pe.stop) {
        e = cudaEventRecord(pe.stop, stream);
        if (e != cudaSuccess) return e;
    }
    // the list length is known on the device only: persistent warps (4 per SM)
    // walk it, and the surplus exits at once
    int64_t lgrid = (batch + 31) / 32;
    if (lgrid > int64_t(sm_count()) * 4) lgrid = int64_t(sm_count()) * 4;
    // launched early (programmatic dependent launch): its CTAs wait in hardware
    // until the dense pass completes, so the launch overlaps that pass's tail
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(unsigned(lgrid));
    lc.blockDim = dim3(32);
    lc.dynamicSmemBytes = K64::kTableBytes;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, small_list_kernel<L, FWD>, comp, xfer, dt, makespan, bits,
                              nseg, status, static_cast<const uint32_t *>(wide_count),
                              static_cast<const uint32_t *>(wide_list));
}

}  // namespace

cudaError_t launch_small(bool forward, int64_t batch, int L, const int64_t *comp,
                         const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                         uint32_t *bits, int32_t *nseg, int32_t *status,
                         uint32_t *wide_count, uint32_t *wide_list, const PassEvents &pe,
                         cudaStream_t stream)
{
#define DC_SMALL_CASE(LL)                                                                     \
    case LL:                                                                                  \
        return forward ? launch_dir<LL, true>(batch, comp, xfer, dt, makespan, bits, nseg,   \
                                              status, wide_count, wide_list, pe, stream)     \
                       : launch_dir<LL, false>(batch, comp, xfer, dt, makespan, bits, nseg,  \
                                               status, wide_count, wide_list, pe, stream);
    switch (L) {
        DC_SMALL_CASE(1) DC_SMALL_CASE(2) DC_SMALL_CASE(3) DC_SMALL_CASE(4)
        DC_SMALL_CASE(5) DC_SMALL_CASE(6) DC_SMALL_CASE(7) DC_SMALL_CASE(8)
        DC_SMALL_CASE(9) DC_SMALL_CASE(10) DC_SMALL_CASE(11) DC_SMALL_CASE(12)
        DC_SMALL_CASE(13) DC_SMALL_CASE(14) DC_SMALL_CASE(15) DC_SMALL_CASE(16)
        default: return cudaErrorInvalidValue;
    }
#undef DC_SMALL_CASE
}

}  // namespace dc

DC_CHECKED_EXPORT(dp_small)
