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
//    the fill; the whole DP runs in registers with compile-time indices;
//  * values are 32-bit whenever the instance bound L*dt + sum(xfer) + sum(comp)
//    is below 2^32 - 1: every DP value and every candidate lies in
//    [0, bound], so the 32-bit fill is exact. Other instances go to a work
//    list solved in 64-bit by the group kernel;
//  * the fill keeps only the minimum VALUE per cell (max, subtract, min per
//    transition). Each finished cell is stored to the lane's slice of shared
//    memory; the traceback then recovers Path[m][n] as the lowest k whose
//    candidate equals the cell, which is exactly the k Algorithm 3/4 keeps
//    with its strict-improvement test;
//  * the warp's rows are loaded with coalesced 64-bit loads into a padded shared
//    buffer (odd row stride: no bank conflicts when each lane reads its row).
#include "common.cuh"

namespace dc {
namespace {

template <int L>
struct Small {
    static constexpr int kCells = L * (L + 1) / 2;
    static constexpr int kOffS = kCells;          // per-lane word offset of S[0..L]
    static constexpr int kOffR = kCells + L + 1;  // per-lane word offset of R[0..L]
    static constexpr int kLaneWords = kCells + 2 * (L + 1);
    static constexpr int kStride = (L % 2 == 0) ? L + 1 : L;  // staging stride, int64 units
    static constexpr int kStageWords = 2 * 32 * kStride * 2;
    static constexpr int kWarpWords =
        (32 * kLaneWords > kStageWords) ? 32 * kLaneWords : kStageWords;
    static constexpr int kWarpBytes = kWarpWords * 4;
    static constexpr int kWarps0 = (48 * 1024) / kWarpBytes;
    static constexpr int kWarps = kWarps0 < 1 ? 1 : (kWarps0 > 8 ? 8 : kWarps0);
    static constexpr int kThreads = 32 * kWarps;
    static constexpr int kSmemBytes = kWarps * kWarpBytes;
};

__host__ __device__ constexpr int cell_of(int L, int m, int n) { return (n - 1) * L - (n - 1) * (n - 2) / 2 + (m - n); }

// The 32-bit fill. lw = this lane's words in shared memory (word w at lw[32*w]).
template <int L, bool FWD>
__device__ __forceinline__ void fill32(const uint32_t (&S)[L + 1], const uint32_t (&Rb)[L + 1],
                                       uint32_t dtv, uint32_t c, uint32_t *lw, uint32_t &T,
                                       int &s)
{
    uint32_t col[L + 1];
    // column n = 1: the only finite predecessor is X[0][0] = 0 and S[0] = 0
#pragma unroll
    for (int m = 1; m <= L; ++m) {
        const uint32_t R = FWD ? dtv + Rb[m] : Rb[m];
        col[m] = R + S[m] + c;
        lw[32 * cell_of(L, m, 1)] = col[m];
    }
    T = col[L];
    s = 1;
#pragma unroll
    for (int n = 2; n <= L; ++n) {
        // rows in descending order so column n overwrites column n-1 in place:
        // row m reads rows k < m, which still hold column n-1.
#pragma unroll
        for (int m = L; m >= n; --m) {
            const uint32_t R = FWD ? uint32_t(n) * dtv + Rb[m] : Rb[m];
            uint32_t best = dmax(col[n - 1], R) - S[n - 1];
#pragma unroll
            for (int k = n; k < m; ++k) best = dmin(best, dmax(col[k], R) - S[k]);
            col[m] = best + S[m] + c;
            lw[32 * cell_of(L, m, n)] = col[m];
        }
        if (col[L] < T) {  // strict: the lowest n wins ties
            T = col[L];
            s = n;
        }
    }
}

template <int L, bool FWD>
__global__ void __launch_bounds__(Small<L>::kThreads)
    small_kernel(int64_t batch, const int64_t *__restrict__ comp,
                 const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
                 int64_t *__restrict__ makespan, uint32_t *__restrict__ bits,
                 int32_t *__restrict__ nseg, int32_t *__restrict__ status,
                 uint32_t *__restrict__ wide_count, uint32_t *__restrict__ wide_list)
{
    using K = Small<L>;
    constexpr int W = (L - 1 + 31) / 32;
    extern __shared__ __align__(16) uint32_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint32_t *region = smem + warp * K::kWarpWords;
    const int64_t base = (int64_t(blockIdx.x) * K::kWarps + warp) * 32;
    if (base >= batch) return;  // warp-uniform
    const int rows = int(batch - base < 32 ? batch - base : 32);
    const int64_t i = base + lane;
    const bool active = lane < rows;

    // ---- coalesced staging of the warp's 32 rows of comp and xfer
    int64_t *stC = reinterpret_cast<int64_t *>(region);
    int64_t *stX = stC + 32 * K::kStride;
    {
        const int64_t *gC = comp + base * L;
        const int64_t *gX = xfer + base * L;
        const int nel = rows * L;
        for (int e = lane; e < nel; e += 32) {
            const int r = e / L, cidx = e - r * L;
            stC[r * K::kStride + cidx] = __ldg(gC + e);
            stX[r * K::kStride + cidx] = __ldg(gX + e);
        }
    }
    const int64_t dti = active ? __ldg(dt + i) : 0;
    __syncwarp();

    // ---- own row, processing order, 64-bit prefix sums and input checks
    uint64_t Pc[L + 1], Px[L + 1];
    bool neg = dti < 0, big = (dti >> 52) != 0;
    Pc[0] = 0;
    Px[0] = 0;
#pragma unroll
    for (int r = 1; r <= L; ++r) {
        const int col = FWD ? r - 1 : L - r;
        const int64_t cv = active ? stC[lane * K::kStride + col] : 0;
        const int64_t xv = active ? stX[lane * K::kStride + col] : 0;
        neg |= (cv < 0) | (xv < 0);
        big |= ((cv | xv) >> 52) != 0;
        Pc[r] = Pc[r - 1] + uint64_t(cv);
        Px[r] = Px[r - 1] + uint64_t(xv);
    }
    __syncwarp();  // every lane is done with the staging area before it is reused

    int st = DC_OK;
    uint64_t bound = 0;
    if (neg) {
        st = DC_ERR_NEGATIVE;
    } else {
        bound = uint64_t(L) * uint64_t(dti) + Pc[L] + Px[L];
        if (big || bound >= uint64_t(kRangeLimit)) st = DC_ERR_RANGE;
    }
    if (!active) return;
    if (st != DC_OK) {
        makespan[i] = -int64_t(st);
        if (nseg) nseg[i] = 0;
        if (status) status[i] = st;
#pragma unroll
        for (int w = 0; w < W; ++w) bits[i * W + w] = 0u;
        return;
    }
    if (bound > kNarrowLimit) {  // needs 64-bit values: hand over to the group kernel
        const uint32_t pos = atomicAdd(wide_count, 1u);
        wide_list[pos] = uint32_t(i);
        return;
    }

    // ---- 32-bit DP
    uint32_t S[L + 1], Rb[L + 1];
#pragma unroll
    for (int m = 0; m <= L; ++m) {
        S[m] = uint32_t(FWD ? Pc[m] : Px[m]);
        Rb[m] = uint32_t(FWD ? Px[m] : Pc[m]);
    }
    const uint32_t dtv = uint32_t(dti);
    const uint32_t c = FWD ? 0u : dtv;
    uint32_t *lw = region + lane;
#pragma unroll
    for (int m = 0; m <= L; ++m) {
        lw[32 * (K::kOffS + m)] = S[m];
        lw[32 * (K::kOffR + m)] = Rb[m];
    }
    uint32_t T;
    int s;
    fill32<L, FWD>(S, Rb, dtv, c, lw, T, s);

    // ---- traceback (Algorithm 3 / 4): from (L, s) step to the lowest k whose
    // candidate equals the cell value, set p_k / g_k, continue at (k, n-1).
    uint32_t word = 0;
    int err = 0;
    int m = L, n = s;
    while (n > 1) {
        const uint32_t R = FWD ? uint32_t(n) * dtv + lw[32 * (K::kOffR + m)]
                               : lw[32 * (K::kOffR + m)];
        const uint32_t target =
            lw[32 * cell_of(L, m, n)] - lw[32 * (K::kOffS + m)] - c;
        const int colbase = cell_of(L, n - 1, n - 1);  // row n-1 of column n-1
        int k = n - 1;
        for (; k < m; ++k) {
            const uint32_t cand =
                dmax(lw[32 * (colbase + k - (n - 1))], R) - lw[32 * (K::kOffS + k)];
            if (cand == target) break;
        }
        if (k >= m) {  // cannot happen: the fill and this check use the same arithmetic
            err = 1;
            break;
        }
        word |= 1u << ((k - 1) & 31);
        m = k;
        n -= 1;
    }
    makespan[i] = int64_t(T);
    if (nseg) nseg[i] = s;
    if (status) status[i] = err ? DC_ERR_INTERNAL : DC_OK;
    if (W > 0) bits[i * W] = word;
}

template <int L>
cudaError_t launch_one(bool forward, int64_t batch, const int64_t *comp, const int64_t *xfer,
                       const int64_t *dt, int64_t *makespan, uint32_t *bits, int32_t *nseg,
                       int32_t *status, uint32_t *wide_count, uint32_t *wide_list,
                       cudaStream_t stream)
{
    using K = Small<L>;
    const int64_t per_block = int64_t(K::kThreads);
    const int64_t blocks = (batch + per_block - 1) / per_block;
    if (blocks > 0x7fffffff) return cudaErrorInvalidValue;
    if (forward)
        small_kernel<L, true><<<unsigned(blocks), K::kThreads, K::kSmemBytes, stream>>>(
            batch, comp, xfer, dt, makespan, bits, nseg, status, wide_count, wide_list);
    else
        small_kernel<L, false><<<unsigned(blocks), K::kThreads, K::kSmemBytes, stream>>>(
            batch, comp, xfer, dt, makespan, bits, nseg, status, wide_count, wide_list);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_small(bool forward, int64_t batch, int L, const int64_t *comp,
                         const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                         uint32_t *bits, int32_t *nseg, int32_t *status,
                         uint32_t *wide_count, uint32_t *wide_list, cudaStream_t stream)
{
#define DC_SMALL_CASE(LL)                                                                    \
    case LL:                                                                                 \
        return launch_one<LL>(forward, batch, comp, xfer, dt, makespan, bits, nseg, status, \
                              wide_count, wide_list, stream);
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
