// Thread-per-instance DynaComm DP for 17 <= L <= 256 (Eq. 8 / Algorithm 3 and
// Eq. 9 / Algorithm 4), 32-bit arithmetic, runtime loops.
//
// Same processing-order template as the other kernels:
//   X[m][n] = min_{k in [n-1, m-1]} max(X[k][n-1], R(m,n)) - S[k] + S[m] + c,
// solved in the shifted form of the short-L kernel: values relative to the
// start of the cell's last transfer, so that a transition is one 32-bit
// add-then-max and the minimum runs on 3-input mins (1.5 integer-ALU
// instructions per transition):
//   forward : B[m][n] + Q[m] = min_k max(G[k] + Q[m], A[k]),  A[k] = B[k][n-1] + P[k],
//   backward: F[m][n] - dt = min_k max(U[m] + NGT[k], F[k][n-1]),  F = X - dt - S[m],
// with G[k] = FC[L] - FC[k], Q[m] = dt + P[m], U = BC - dt (backward),
// NGT[k] = -(transfer prefix), A[m][1] = FC[L] + P[m], F[m][1] = BC[m]; both are
// min_k max(U[m] + V[k], C[k]) with a row constant U (Q forward) that is the
// same in every column and the previous column C in the max operand. The
// makespan is min_n B[L][n] + n*dt + P[L] (forward) or min_n F[L][n] + dt + S[L]
// (backward), plus the capped-off transfer. Every candidate differs from Eq.
// 8/9's by a constant of its cell, so every argmin is the same.
//
// Design (GB300):
//  * one instance per thread; the lane's two per-layer arrays and its current
//    column live in its slice of shared memory, lane-interleaved so that a
//    warp's accesses never conflict (U[v] at word 32*v + lane; the column and V
//    as 64-bit pairs at 32*v + lane, one load per candidate k);
//  * register blocking: a column is filled in blocks of kB = 8 consecutive rows
//    held in registers; every (column, V) pair read from shared memory feeds kB
//    transitions. A full block's own triangle (row bot+j takes k < bot+j) is
//    unrolled without branches; only a column's lowest, partial block takes the
//    general path. Rows are visited top-down so that the column is
//    updated in place: a block reads only rows below its own top, which still
//    hold column n-1;
//  * transfer costs capped at the total compute (exact, as in the short-L
//    kernel); the shifted values fit in signed 32 bits whenever the capped bound
//    L*dt + sum(comp) + sum(capped xfer) is below 2^31;
//  * value-only fill with deferred argmin, as in the short-L kernel: columns
//    2..8 (L <= 64) or 2..16 are written to a per-thread slot of the caller's
//    workspace (coalesced across the warp) and the traceback re-derives each
//    Path[m][n] as the lowest k whose candidate equals the cell. Instances whose
//    optimum needs a deeper column, or whose values need more than 31 bits, are
//    put on a work list that the CTA-per-instance kernel solves afterwards;
//  * persistent CTAs claim 32-instance tiles from an atomic ticket, so the
//    long, uneven per-tile work balances across the GPU. The lane slices take
//    3*(L+1) words per lane and limit the resident warps, so for long rows 2, 4
//    or 8 warps share a tile (same slices, less shared memory per warp): the
//    column's row blocks are dealt to them in a snake, each warp keeps its
//    results in registers until all have read column n-1 (a CTA barrier), then
//    all write column n and meet at a second barrier. The tile's instances are
//    dealt to the warps (32/NW each) for the row reads and the tracebacks, so
//    no warp waits while another does them alone;
//  * the traceback skips the candidates that cannot match: U[m] + V[k] is
//    non-increasing in k and bounds the candidate from below, so a binary
//    search over V finds the first k with U[m] + V[k] <= the cell, and the scan
//    of the kept column starts there.
#include "common.cuh"

namespace dc {
namespace {

constexpr int kB = 8;  // rows per register block
constexpr int kQ = 4;  // row blocks of a column per warp, at most (L <= 32 * warps)

// warps sharing a tile: the lane slices take 3*(L+1) words per lane and limit
// the resident warps, so longer rows spread a tile over more warps (measured
// faster from L = 41 on)
__host__ __device__ inline int mid_warps(int L) { return L <= 40 ? 1 : L <= 64 ? 2 : L <= 128 ? 4 : 8; }

// last column kept for the traceback (a traceback of s segments reads columns
// 1..s-1): 8 up to L = 64, 16 beyond (deeper optima are more common there)
__host__ __device__ inline int mid_keep_last(int L)
{
    const int keep = L <= 64 ? 8 : 16;
    return L - 1 < keep ? L - 1 : keep;
}
// stored cell (m, n), 2 <= n <= keep_last
__host__ __device__ inline int mid_cell(int L, int m, int n)
{
    return (n - 2) * L - (n - 2) * (n - 1) / 2 + (m - n);
}
__host__ __device__ inline int mid_cells(int L)
{
    const int c = mid_keep_last(L);
    return c >= 2 ? mid_cell(L, L, c) + 1 : 0;
}
// traceback slots (one per lane of a launched CTA): about one resident wave of
// CTAs (kMidSlots up to L = 64), and no more than the batch's tiles need
__host__ __device__ inline int64_t mid_slots(int64_t batch, int L)
{
    const int nw = mid_warps(L);
    const int64_t wave = nw <= 2 ? kMidSlots : int64_t(152) * 32 * (nw == 4 ? 4 : 2);
    const int64_t need = (batch + 31) / 32 * 32;
    return need < wave ? need : wave;
}

// Rows -> the lane slices: U (Q forward, BC - dt backward) at 32*v, and the
// (column, V) pairs with column 1 in .x and V (G forward, NGT backward) in .y.
// Checks the input; returns false when this kernel does not solve the instance
// (an input error, whose outputs it writes, or values beyond 31 bits, which it
// lists for the CTA-per-instance kernel).
template <bool FWD>
__device__ __forceinline__ bool mid_prefix(int64_t batch, int64_t i, int L, const int64_t *__restrict__ comp,
                                           const int64_t *__restrict__ xfer, int64_t dti,
                                           uint32_t *lw, int2 *pv, int64_t *makespan,
                                           uint32_t *bits, int32_t *nseg, int32_t *status,
                                           uint32_t *list_count, uint32_t *list, uint64_t &px,
                                           int32_t &fcL)
{
    const int W = words_for(L);
    // transfer costs capped at the total compute (exact: same decisions, makespan
    // lower by sum(xfer) - sum(capped xfer), added back at the end)
    const int64_t *crow = comp + i * L, *xrow = xfer + i * L;
    bool neg = dti < 0, big = (dti >> 52) != 0;
    uint64_t tc = 0;
    px = 0;
    for (int l = 0; l < L; ++l) {
        const int64_t cv = __ldg(crow + l), xv = __ldg(xrow + l);
        neg |= (cv < 0) | (xv < 0);
        big |= ((cv | xv) >> 52) != 0;
        tc += uint64_t(cv);
        px += uint64_t(xv);
    }
    if (neg || big || exceeds_range(L, dti, tc, px)) {
        const int st = neg ? DC_ERR_NEGATIVE : DC_ERR_RANGE;
        makespan[i] = -int64_t(st);
        if (nseg) nseg[i] = 0;
        if (status) status[i] = st;
        for (int w = 0; w < W; ++w) bits[i * W + w] = 0u;
        return false;
    }
    // wrapping 32-bit arithmetic: the values are used only when the range check passes
    uint64_t pc = 0, pxc = 0;
    const uint32_t dtu = uint32_t(dti), tcu = uint32_t(tc);
    lw[0] = FWD ? dtu : 0u - dtu;
    pv[0].y = FWD ? int32_t(tcu) : 0;
    for (int r = 1; r <= L; ++r) {
        const int col = FWD ? r - 1 : L - r;
        const uint64_t cv = uint64_t(__ldg(crow + col)), xv = uint64_t(__ldg(xrow + col));
        pc += cv;
        pxc += xv < tc ? xv : tc;
        const uint32_t u = FWD ? dtu + uint32_t(pxc) : uint32_t(pc) - dtu;
        lw[32 * r] = u;
        pv[32 * r] = make_int2(int32_t(FWD ? tcu + u - dtu : u + dtu),  // column 1: A or F
                               int32_t(FWD ? tcu - uint32_t(pc) : 0u - uint32_t(pxc)));
    }
    if (pc + pxc + uint64_t(L) * uint64_t(dti) > kShiftedLimit) {
        {
            const uint32_t at = atomicAdd(list_count, 1u);
            if (DC_CHECK(int64_t(at) < batch)) list[at] = uint32_t(i);
        }
        return false;
    }
    fcL = int32_t(tcu);
    return true;
}

// Minima of the rows bot..top (top - bot < kB) of column n over their candidates
// k in [n-1, m-1]: best[j] for row bot + j. Reads column n-1 (pv .x) and V (.y);
// writes nothing.
template <bool FWD>
__device__ __forceinline__ void mid_block(const int2 *pv, const int32_t *U, int n, int top,
                                          int bot, int32_t (&best)[kB])
{
    int32_t Ur[kB];
#pragma unroll
    for (int j = 0; j < kB; ++j) {
        const int m = bot + j <= top ? bot + j : top;
        Ur[j] = U[32 * m];
        best[j] = 0x7fffffff;
    }
    // k below the block, four then two at a time: every row of the block takes
    // them; one 64-bit load brings a (column, V) pair
    auto cand = [&](int2 p, int j) { return __viaddmax_s32(Ur[j], p.y, p.x); };
    int k = n - 1;
    for (; k + 3 < bot; k += 4) {
        const int2 p0 = pv[32 * k], p1 = pv[32 * (k + 1)];
        const int2 p2 = pv[32 * (k + 2)], p3 = pv[32 * (k + 3)];
#pragma unroll
        for (int j = 0; j < kB; ++j) {
            best[j] = __vimin3_s32(best[j], cand(p0, j), cand(p1, j));
            best[j] = __vimin3_s32(best[j], cand(p2, j), cand(p3, j));
        }
    }
    if (k + 1 < bot) {
        const int2 p0 = pv[32 * k], p1 = pv[32 * (k + 1)];
#pragma unroll
        for (int j = 0; j < kB; ++j) best[j] = __vimin3_s32(best[j], cand(p0, j), cand(p1, j));
        k += 2;
    }
    if (k < bot) {
        const int2 p0 = pv[32 * k];
#pragma unroll
        for (int j = 0; j < kB; ++j) best[j] = min(best[j], cand(p0, j));
    }
    if (top - bot == kB - 1) {
        // full block, k inside it: row bot+j takes k = bot .. bot+j-1, unrolled
        // without branches, candidates paired into 3-input mins
        int2 q[kB - 1];
#pragma unroll
        for (int t = 0; t < kB - 1; ++t) q[t] = pv[32 * (bot + t)];
#pragma unroll
        for (int j = 1; j < kB; ++j) {
            int t = 0;
#pragma unroll
            for (; t + 1 < j; t += 2) best[j] = __vimin3_s32(best[j], cand(q[t], j), cand(q[t + 1], j));
            if (t < j) best[j] = min(best[j], cand(q[t], j));
        }
        return;
    }
    // partial block (the column's lowest), k inside it
#pragma unroll
    for (int t = 0; t < kB - 1; ++t) {
        const int kk = bot + t;
        if (kk >= top) break;
        const int2 p0 = pv[32 * kk];
#pragma unroll
        for (int j = t + 1; j < kB; ++j) best[j] = min(best[j], cand(p0, j));
    }
}

// Column n's values of rows bot..top (from their minima best[]) into the lane's
// column slot and, for the kept columns, its traceback slot; `last` takes row L's
// minimum.
template <bool FWD>
__device__ __forceinline__ void mid_write(int2 *pv, uint32_t *myslot, int64_t nslots, int L,
                                          int n, int keep, int top, int bot,
                                          const int32_t (&best)[kB], int32_t dt32, int32_t &last)
{
    const int64_t cb = int64_t(mid_cell(L, bot, n)) * nslots;
    // the kept cells of rows bot..top (column n <= keep) lie in the slot's cells
    if (!DC_CHECK(n > keep || (bot >= n && top <= L && mid_cell(L, top, n) < mid_cells(L)))) return;
    if (top - bot == kB - 1) {  // full block
#pragma unroll
        for (int j = 0; j < kB; ++j) {
            const int32_t val = FWD ? best[j] - dt32 : best[j] + dt32;
            pv[32 * (bot + j)].x = val;
            if (n <= keep) myslot[cb + int64_t(j) * nslots] = uint32_t(val);
        }
        if (top == L) last = best[kB - 1];
        return;
    }
#pragma unroll
    for (int j = 0; j < kB; ++j) {
        const int m = bot + j;
        if (m <= top) {
            const int32_t val = FWD ? best[j] - dt32 : best[j] + dt32;
            pv[32 * m].x = val;
            if (n <= keep) myslot[cb + int64_t(j) * nslots] = uint32_t(val);
            if (m == L) last = best[j];
        }
    }
}

// Block b of a column (b = 0 holds row L): rows bot..top.
__device__ __forceinline__ void mid_rows(int L, int n, int b, int &top, int &bot)
{
    top = L - kB * b;
    bot = top - kB + 1 > n ? top - kB + 1 : n;
}

// Block of warp w for its q-th slot when NW warps share a column: a snake over
// the blocks (0, 3, 4, 7 to warp 0 and 1, 2, 5, 6 to warp 1 for NW = 2; rows
// 0..NW-1 left to right, the next NW right to left, and so on), which evens out
// the work of the upper (longer) and lower blocks.
template <int NW>
__device__ __forceinline__ int mid_block_of(int q, int w)
{
    return (q % 2 == 0) ? NW * q + w : NW * q + NW - 1 - w;
}

template <bool FWD, int NW>
__global__ void __launch_bounds__(32 * NW)
    mid_kernel(int64_t batch, int L, const int64_t *__restrict__ comp,
               const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
               int64_t *__restrict__ makespan, uint32_t *__restrict__ bits,
               int32_t *__restrict__ nseg, int32_t *__restrict__ status,
               uint32_t *__restrict__ ticket, uint32_t *__restrict__ list_count,
               uint32_t *__restrict__ list, uint32_t *__restrict__ tb, int64_t nslots)
{
    extern __shared__ uint32_t smem[];
    __shared__ uint32_t s_tile;
    __shared__ int32_t s_dt[32], s_fcL[32], s_go[32], s_best[32], s_s[32];
    __shared__ uint64_t s_px[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int W = words_for(L);
    // lane slices: U[v] at word 32*v + lane (v in [0, L]), then the current column
    // and V as (C[v], V[v]) pairs at 64-bit word 32*v + lane
    uint32_t *lw = smem + lane;
    int2 *pv = reinterpret_cast<int2 *>(smem + 32 * (L + 1)) + lane;
    const int32_t *U = reinterpret_cast<const int32_t *>(lw);
    const int64_t slot = int64_t(blockIdx.x) * 32 + lane;
    uint32_t *myslot = tb + slot;  // cell c at myslot[c * nslots]
    const int keep = mid_keep_last(L);
    const int64_t tiles = (batch + 31) / 32;

    for (;;) {
        if (threadIdx.x == 0) s_tile = atomicAdd(ticket, 1u);
        __syncthreads();
        const uint32_t tile = s_tile;
        if (int64_t(tile) >= tiles) break;
        const int64_t i = int64_t(tile) * 32 + lane;

        // ---- rows -> lane slices: the tile's instances dealt to the warps, 32/NW
        // each (a lane's slice is the same in every warp)
        const bool mine = lane / (32 / NW) == warp;
        if (mine) {
            const int64_t dti = i < batch ? __ldg(dt + i) : 0;
            uint64_t px = 0;
            int32_t fcL = 0;
            const bool go = i < batch && mid_prefix<FWD>(batch, i, L, comp, xfer, dti, lw, pv, makespan,
                                                         bits, nseg, status, list_count, list, px,
                                                         fcL);
            s_dt[lane] = int32_t(dti);
            s_go[lane] = go;
            s_px[lane] = px;
            s_fcL[lane] = fcL;
        }
        if (NW > 1) __syncthreads(); else __syncwarp();
        // every lane runs the fill (lanes without an instance on stale slices:
        // all accesses stay in the lane's own slice and slot), so that the
        // barriers of the split fill are reached by all threads
        const int32_t dt32 = s_dt[lane];
        const int32_t fcL = s_fcL[lane];

        // ---- fill
        int32_t bestV = 0;
        int s = 1;
        if (warp == 0) bestV = FWD ? fcL + dt32 : U[32 * L] + 2 * dt32;
        for (int n = 2; n <= L; ++n) {
            int32_t last = 0;  // row L's minimum: B[L][n] + Q[L] (forward) or F[L][n] - dt
            if constexpr (NW == 1) {
                // rows top-down, so column n overwrites column n-1 in place: a
                // block reads only rows below its own top, which still hold n-1
                for (int top = L; top >= n; top -= kB) {
                    const int bot = top - kB + 1 > n ? top - kB + 1 : n;
                    int32_t best[kB];
                    mid_block<FWD>(pv, U, n, top, bot, best);
                    mid_write<FWD>(pv, myslot, nslots, L, n, keep, top, bot, best, dt32, last);
                }
            } else {
                // NW warps share the column's blocks; a block's rows are read by
                // the blocks above it, so every result waits in registers until
                // all warps have read column n-1
                const int nb = (L - n + kB) / kB;
                int32_t res[kQ][kB];
#pragma unroll
                for (int q = 0; q < kQ; ++q) {
                    const int b = mid_block_of<NW>(q, warp);
                    if (b < nb) {
                        int top, bot;
                        mid_rows(L, n, b, top, bot);
                        mid_block<FWD>(pv, U, n, top, bot, res[q]);
                    }
                }
                __syncthreads();
#pragma unroll
                for (int q = 0; q < kQ; ++q) {
                    const int b = mid_block_of<NW>(q, warp);
                    if (b < nb) {
                        int top, bot;
                        mid_rows(L, n, b, top, bot);
                        mid_write<FWD>(pv, myslot, nslots, L, n, keep, top, bot, res[q], dt32, last);
                    }
                }
                __syncthreads();
            }
            if (warp == 0) {  // row L is in block 0, which warp 0 holds
                // X[L][n] less P[L] (forward: B[L][n] + n dt) or S[L] (backward: F[L][n] + dt)
                const int32_t v = FWD ? last - U[32 * L] + n * dt32 : last + 2 * dt32;
                if (v < bestV) {  // strict: the lowest n wins ties
                    bestV = v;
                    s = n;
                }
            }
        }
        // the tracebacks, dealt to the warps like the rows
        if (warp == 0) {
            s_best[lane] = bestV;
            s_s[lane] = s;
        }
        if (NW > 1) __syncthreads(); else __syncwarp();
        if (!mine || !s_go[lane]) continue;
        bestV = s_best[lane];
        s = s_s[lane];
        const uint64_t px = s_px[lane];
        if (s - 1 > keep && s - 1 >= 2) {  // traceback would need an unkept column
            {
            const uint32_t at = atomicAdd(list_count, 1u);
            if (DC_CHECK(int64_t(at) < batch)) list[at] = uint32_t(i);
        }
            continue;
        }

        // ---- traceback: lowest k whose candidate equals the cell
        // decision words 0 and 1 in registers; words 2.. (L > 65) set in place
        uint32_t word0 = 0u, word1 = 0u;
        for (int w = 2; w < W; ++w) bits[i * W + w] = 0u;
        int err = 0, m = L, n = s;
        int32_t target = FWD ? bestV - s * dt32 + U[32 * L] : bestV - 2 * dt32;  // B[L][s] + Q[L] or F[L][s] - dt
        while (n > 1) {
            const int32_t uu = U[32 * m];
            // U[m] + V[k] is non-increasing in k (V is G forward, the negated
            // transfer prefix backward) and a candidate max(U[m] + V[k], C[k]) is
            // at least U[m] + V[k]: every k before the first with U[m] + V[k] <=
            // target misses, and the scan starts there
            int lo = n - 1, hi = m - 1;
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (uu + pv[32 * mid].y > target)
                    lo = mid + 1;
                else
                    hi = mid;
            }
            // candidates in groups of 8 (loads issued together, lowest match wins)
            int k = -1;
            int32_t fk = 0;
            for (int k0 = lo; k0 < m && k < 0; k0 += 8) {
                int32_t f[8], v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int kk = k0 + u < m ? k0 + u : m - 1;  // stay inside column n-1
                    v[u] = pv[32 * kk].y;
                    if (n - 1 == 1)  // column 1 from U
                        f[u] = FWD ? fcL + U[32 * kk] - dt32 : U[32 * kk] + dt32;
                    else
                        f[u] = DC_CHECK(mid_cell(L, kk, n - 1) < mid_cells(L))
                                   ? int32_t(myslot[int64_t(mid_cell(L, kk, n - 1)) * nslots])
                                   : 0;
                }
#pragma unroll
                for (int u = 8 - 1; u >= 0; --u) {
                    if (k0 + u < m && __viaddmax_s32(uu, v[u], f[u]) == target) {
                        k = k0 + u;
                        fk = f[u];
                    }
                }
            }
            if (k < 0) {
                err = 1;
                break;
            }
            if (k - 1 < 32)
                word0 |= 1u << (k - 1);
            else if (k - 1 < 64)
                word1 |= 1u << (k - 33);
            else
                bits[i * W + ((k - 1) >> 5)] |= 1u << ((k - 1) & 31);
            target = FWD ? fk + dt32 : fk - dt32;  // the cell (k, n-1): B + Q[k] = A + dt, or F - dt
            m = k;
            n -= 1;
        }
        makespan[i] = int64_t(uint64_t(uint32_t(bestV)) + px);
        if (nseg) nseg[i] = s;
        if (status) status[i] = err ? DC_ERR_INTERNAL : DC_OK;
        bits[i * W] = word0;
        if (W > 1) bits[i * W + 1] = word1;
    }
}

template <bool FWD, int NW>
cudaError_t launch_mid_nw(int64_t batch, int L, const int64_t *comp, const int64_t *xfer,
                          const int64_t *dt, int64_t *makespan, uint32_t *bits, int32_t *nseg,
                          int32_t *status, uint32_t *ticket, uint32_t *list_count,
                          uint32_t *list, uint32_t *tb, cudaStream_t stream)
{
    const size_t smem = size_t(3) * (L + 1) * 32 * 4;
    static DeviceCache attr;  // the kernel's shared-memory limit, raised once per device
    int done = 0;
    const cudaError_t ae = attr.get(done, [](int &v) {
        const int most = 3 * (kMidLMax + 1) * 32 * 4;
        v = 1;
        return cudaFuncSetAttribute(mid_kernel<FWD, NW>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, most);
    });
    if (ae != cudaSuccess) return ae;
    const int64_t slots = mid_slots(batch, L);
    const int64_t grid = slots / 32;
    mid_kernel<FWD, NW><<<unsigned(grid), 32 * NW, smem, stream>>>(
        batch, L, comp, xfer, dt, makespan, bits, nseg, status, ticket, list_count, list, tb,
        slots);
    return cudaGetLastError();
}

}  // namespace

size_t mid_scratch_bytes(int64_t batch, int L)
{
    return size_t(mid_slots(batch, L)) * size_t(mid_cells(L)) * 4;
}

cudaError_t launch_mid(bool forward, int64_t batch, int L, const int64_t *comp,
                       const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                       uint32_t *bits, int32_t *nseg, int32_t *status, uint32_t *ticket,
                       uint32_t *list_count, uint32_t *list, uint32_t *tb, cudaStream_t stream)
{
#define DC_MID_LAUNCH(NW)                                                                        \
    return forward ? launch_mid_nw<true, NW>(batch, L, comp, xfer, dt, makespan, bits, nseg,    \
                                             status, ticket, list_count, list, tb, stream)       \
                   : launch_mid_nw<false, NW>(batch, L, comp, xfer, dt, makespan, bits, nseg,   \
                                              status, ticket, list_count, list, tb, stream);
    // warps per tile: the kernel's choice, or the test hook's when its blocks
    // (4 per warp and column) still cover a column's rows
    int nw = mid_warps(L);
    const int f = forced_warps();
    if (f == 1 || (f > 1 && (L + 6) / 8 <= 4 * f)) nw = f;
    switch (nw) {
        case 1: DC_MID_LAUNCH(1)
        case 2: DC_MID_LAUNCH(2)
        case 4: DC_MID_LAUNCH(4)
        default: DC_MID_LAUNCH(8)
    }
#undef DC_MID_LAUNCH
}

}  // namespace dc

DC_CHECKED_EXPORT(dp_mid)
