// CTA-per-instance DynaComm DP for any 1 <= L <= 4096 (Eq. 8 / Algorithm 3 and
// Eq. 9 / Algorithm 4), in 32-bit or 64-bit arithmetic per instance.
//
// Used for L > 64, and for the instances the thread-per-instance kernels list
// (values beyond their 32-bit form, or a traceback deeper than they keep).
// Transfer costs are capped at the total compute first (exact; see the short-L
// kernel).
//
// Same processing-order template as the small kernel:
//   X[m][n] = min_{k in [n-1, m-1]} max(X[k][n-1], R(m,n)) - S[k] + S[m] + c.
// Per instance, the arithmetic is the first that is exact: the shifted signed
// 32-bit form of the short kernels (capped bound below 2^31), the shifted forms
// of this file for wider instances (backward with total compute below 2^31,
// forward below 2^29), the literal template in 32 bits (bound below 2^32), else
// in 64 bits. Column n's (row block, k chunk) tiles are spread over the CTA's
// threads (8 rows x up to 64 candidates per tile, register-blocked), partial row
// minima are combined with shared-memory atomicMin, then the column is
// finalised; columns run in sequence with CTA barriers between them. Every
// finished cell is also written to the instance's DP table (shared memory for
// L <= 64, otherwise a per-CTA slot of the caller's workspace). After the fill,
// warp 0 picks the lowest n minimising X[L][n] and walks the traceback, finding
// each Path[m][n] (the lowest k whose candidate equals the cell) with one ballot
// per 32 candidates.
#include "common.cuh"

namespace dc {
namespace {

struct GroupArgs {
    int64_t batch;
    int L;
    const int64_t *comp, *xfer, *dt;
    int64_t *makespan;
    uint32_t *bits;
    int32_t *nseg, *status;
    const uint32_t *list_count, *list;
    unsigned char *tables;  // nullptr: DP table in shared memory
};

// Shared-memory layout: five arrays of Ls = L + 1 + (L + 1)/32 + 1 entries sized
// for 64-bit values (S, R, two column buffers, per-row partial minima), indexed
// through skew(k) = k + k/32 so that tiles whose k ranges start 64 apart hit
// different banks; then the decision words, a 256-byte scan scratch, and the DP
// table when it stays on chip.
__host__ __device__ inline int group_ls(int L) { return L + 1 + (L + 1) / 32 + 1; }
__device__ __forceinline__ int skew(int k) { return k + (k >> 5); }
__host__ __device__ inline size_t group_arrays_bytes(int L) { return size_t(5) * group_ls(L) * 8; }
__host__ __device__ inline size_t group_bits_bytes(int L)
{
    return (size_t(words_for(L) + 1) * 4 + 15) / 16 * 16;
}
constexpr size_t kScratchBytes = 256;
__host__ __device__ inline size_t group_table_offset(int L)
{
    return group_arrays_bytes(L) + group_bits_bytes(L) + kScratchBytes;
}
inline size_t group_smem_bytes(int L, bool table_in_smem)
{
    return group_table_offset(L) + (table_in_smem ? size_t(tri_cells(L)) * 8 : 0);
}

// Inclusive prefix of v[1..L] in place (v[0] = 0), CTA-wide; each thread owns
// a contiguous chunk, chunk totals are scanned by warp 0.
__device__ void block_prefix_u64(uint64_t *v, int L, uint64_t *scratch /* >= 16 entries */)
{
    const int nt = blockDim.x, t = threadIdx.x;
    const int chunk = (L + nt - 1) / nt;
    const int lo = 1 + t * chunk, hi = min(L, lo + chunk - 1);
    uint64_t acc = 0;
    for (int j = lo; j <= hi; ++j) {
        acc += v[j];
        v[j] = acc;
    }
    const int lane = t & 31, warp = t >> 5, nw = (nt + 31) >> 5;
    uint64_t x = acc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint64_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) scratch[warp] = x;
    __syncthreads();
    if (t == 0) {
        uint64_t run = 0;
        for (int w = 0; w < nw; ++w) {
            const uint64_t tot = scratch[w];
            scratch[w] = run;
            run += tot;
        }
    }
    __syncthreads();
    const uint64_t off = scratch[warp] + x - acc;
    for (int j = lo; j <= hi; ++j) v[j] += off;
    __syncthreads();
}

__device__ __forceinline__ void atomic_min_T(uint32_t *p, uint32_t v) { atomicMin(p, v); }
__device__ __forceinline__ void atomic_min_T(uint64_t *p, uint64_t v)
{
    atomicMin(reinterpret_cast<unsigned long long *>(p), static_cast<unsigned long long>(v));
}

// CTA-wide sums of two per-thread values, returned to every thread.
__device__ void block_sum2_u64(uint64_t &a, uint64_t &b, uint64_t *scratch /* >= 32 */)
{
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        b += __shfl_xor_sync(0xffffffffu, b, o);
    }
    if (lane == 0) {
        scratch[warp] = a;
        scratch[16 + warp] = b;
    }
    __syncthreads();
    a = 0;
    b = 0;
    for (int w = 0; w < nw; ++w) {
        a += scratch[w];
        b += scratch[16 + w];
    }
    __syncthreads();
}

constexpr int kRB = 8;   // rows per tile
constexpr int kKC = 64;  // k per tile

// Tile q of column n (numbering below): rows bot..top, candidates k in [k0, k1).
// Returns false for a tile with no work.
__device__ __forceinline__ bool decode_tile(int q, int L, int n, int nb, int &bot, int &top,
                                            int &k0, int &k1)
{
    int g = int((sqrtf(1.0f + float(q)) - 1.0f) * 0.5f);
    while (4 * (g + 1) * (g + 2) <= q) ++g;
    while (g > 0 && 4 * g * (g + 1) > q) --g;
    const int r = q - 4 * g * (g + 1);
    const int b = 8 * g + r / (g + 1);
    const int j = r % (g + 1);
    if (b >= nb) return false;
    bot = n + kRB * b;
    top = bot + kRB - 1 < L ? bot + kRB - 1 : L;
    k0 = n - 1 + kKC * j;
    if (k0 > top - 1) return false;
    k1 = k0 + kKC < top ? k0 + kKC : top;  // exclusive
    return true;
}

// Column n's work is the set of (row block b, k chunk j) tiles: block b holds
// rows n+8b .. n+8b+7 and needs k in [n-1, top_b - 1], i.e. ceil((8b+8)/64) =
// b/8 + 1 chunks of 64. Tiles are numbered group by group (blocks 8g..8g+7 have
// g+1 chunks each, 4g(g+1) tiles precede group g) and dealt round-robin to the
// CTA's threads; each tile's 8 partial minima are combined with atomicMin.
template <typename T, bool FWD>
__device__ __forceinline__ void fill_tiles(int L, int n, T dtv, const T *S, const T *Rb,
                                           const T *prev, T *best)
{
    const int t = threadIdx.x, nt = blockDim.x;
    const T ndt = T(T(n) * dtv);
    const int nb = (L - n + 1 + kRB - 1) / kRB;
    const int ng = (nb + 7) / 8;
    const int ntiles = 4 * ng * (ng + 1);
    for (int q = t; q < ntiles; q += nt) {
        int bot, top, k0, k1;
        if (!decode_tile(q, L, n, nb, bot, top, k0, k1)) continue;
        T R[kRB], acc[kRB];
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj) {
            const int m = bot + jj <= top ? bot + jj : top;
            R[jj] = FWD ? T(ndt + Rb[skew(m)]) : Rb[skew(m)];
            acc[jj] = T(~T(0));
        }
        const int kf = k1 < bot ? k1 : bot;  // k < bot: every row of the block takes it
        for (int k = k0; k < kf; ++k) {
            const T v = prev[skew(k)], sk = S[skew(k)];
#pragma unroll
            for (int jj = 0; jj < kRB; ++jj) acc[jj] = dmin(acc[jj], T(dmax(v, R[jj]) - sk));
        }
        if (k1 > bot) {  // row bot+jj takes k < bot+jj
#pragma unroll
            for (int u = 0; u < kRB - 1; ++u) {
                const int k = bot + u;
                if (k >= k1) break;
                if (k < k0) continue;
                const T v = prev[skew(k)], sk = S[skew(k)];
#pragma unroll
                for (int jj = u + 1; jj < kRB; ++jj) acc[jj] = dmin(acc[jj], T(dmax(v, R[jj]) - sk));
            }
        }
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj)
            if (bot + jj <= top) atomic_min_T(&best[skew(bot + jj)], acc[jj]);
    }
}

template <typename T, bool FWD>
__device__ void solve(const GroupArgs &a, int64_t i, int64_t dti, uint64_t shift,
                      const uint64_t *P64c, const uint64_t *P64x, unsigned char *arrays,
                      uint32_t *bitsw, T *table)
{
    const int L = a.L, t = threadIdx.x, nt = blockDim.x, Ls = group_ls(L);
    T *S = reinterpret_cast<T *>(arrays);
    T *Rb = S + Ls;
    T *colA = Rb + Ls;
    T *colB = colA + Ls;
    T *best = colB + Ls;
    // P64c / P64x sit in the 64-bit column-buffer bytes, past the typed S and R
    // arrays for either T; the typed columns overwrite them only after this copy.
    for (int m = t; m <= L; m += nt) {
        S[skew(m)] = T(FWD ? P64c[m] : P64x[m]);
        Rb[skew(m)] = T(FWD ? P64x[m] : P64c[m]);
    }
    __syncthreads();

    const T dtv = T(dti);
    const T c = FWD ? T(0) : dtv;
    for (int m = 1 + t; m <= L; m += nt) {  // column 1
        const T R = FWD ? T(dtv + Rb[skew(m)]) : Rb[skew(m)];
        const T v = T(R + S[skew(m)] + c);
        colA[skew(m)] = v;
        best[skew(m)] = T(~T(0));
        if (DC_CHECK(tri_index(L, m, 1) < tri_cells(L))) table[tri_index(L, m, 1)] = v;
    }
    __syncthreads();
    T *prev = colA, *cur = colB;
    for (int n = 2; n <= L; ++n) {
        fill_tiles<T, FWD>(L, n, dtv, S, Rb, prev, best);
        __syncthreads();
        const int64_t cbase = tri_col(L, n) - n;
        for (int m = n + t; m <= L; m += nt) {
            const T v = T(best[skew(m)] + S[skew(m)] + c);
            cur[skew(m)] = v;
            best[skew(m)] = T(~T(0));
            if (DC_CHECK(cbase + m < tri_cells(L))) table[cbase + m] = v;
        }
        __syncthreads();
        T *tmp = prev;
        prev = cur;
        cur = tmp;
    }

    // final pick and traceback by warp 0
    if (t < 32) {
        const int lane = t;
        T bv = T(~T(0));
        int bn = 0x7fffffff;
        for (int n = 1 + lane; n <= L; n += 32) {
            const T v = table[tri_index(L, L, n)];
            if (v < bv) {  // n increases: strict keeps the lowest n in this lane
                bv = v;
                bn = n;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const T ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int on = __shfl_xor_sync(0xffffffffu, bn, o);
            if (ov < bv || (ov == bv && on < bn)) {
                bv = ov;
                bn = on;
            }
        }
        const int s = bn;
        int err = 0;
        int m = L, n = s;
        while (n > 1) {
            const T R = FWD ? T(T(n) * dtv + Rb[skew(m)]) : Rb[skew(m)];
            const T target = T(table[tri_index(L, m, n)] - S[skew(m)] - c);
            const int64_t pbase = tri_col(L, n - 1) - (n - 1);  // + k gives (k, n-1)
            int found = -1;
            for (int k0 = n - 1; k0 < m; k0 += 32) {
                const int k = k0 + lane;
                bool match = false;
                if (k < m) match = T(dmax(table[pbase + k], R) - S[skew(k)]) == target;
                const unsigned bal = __ballot_sync(0xffffffffu, match);
                if (bal) {
                    found = k0 + __ffs(bal) - 1;
                    break;
                }
            }
            if (found < 0) {
                err = 1;
                break;
            }
            if (lane == 0) bitsw[(found - 1) >> 5] |= 1u << ((found - 1) & 31);
            __syncwarp();
            m = found;
            n -= 1;
        }
        if (lane == 0) {
            a.makespan[i] = int64_t(uint64_t(bv) + shift);
            if (a.nseg) a.nseg[i] = s;
            if (a.status) a.status[i] = err ? DC_ERR_INTERNAL : DC_OK;
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// Instances whose capped bound L*dt + sum(comp) + sum(capped xfer) is below 2^31:
// the shifted form of the thread-per-instance kernels, all in signed 32 bits,
// where a transition is one add-then-max and two candidates fold with one
// 3-input min (1.5 integer-ALU instructions per transition):
//   forward : B[m][n] + Q[m] = min_k max(G[k] + Q[m], A[k]),  A[k] = B[k][n-1] + P[k],
//   backward: E[m][n] = min_k max(BC[m] - (n-1)*dt + NGT[k], E[k][n-1]),
// with G[k] = FC[L] - FC[k], Q[m] = dt + P[m] (P = transfer prefix),
// NGT[k] = -(transfer prefix), A[m][1] = FC[L] + P[m], E[m][1] = BC[m]; U = (Q, BC)
// and V = (G, NGT) per direction, and both are min_k max(u[m] + V[k], C[k]). The makespan is min_n (B or E)[L][n] + n*dt plus
// the transfer sum. Each candidate differs from Eq. 8/9's by a constant of its
// row, so every argmin is unchanged. The table holds A (forward) or E.

__device__ __forceinline__ int32_t cand_s32(int32_t col, int32_t u, int32_t v)
{
    return __viaddmax_s32(u, v, col);
}

template <bool FWD>
__device__ __forceinline__ void fill_tiles_s32(int L, int n, int32_t ndt1, const int32_t *U,
                                               const int32_t *V, const int32_t *prev,
                                               int32_t *best)
{
    const int t = threadIdx.x, nt = blockDim.x;
    const int nb = (L - n + 1 + kRB - 1) / kRB;
    const int ng = (nb + 7) / 8;
    const int ntiles = 4 * ng * (ng + 1);
    for (int q = t; q < ntiles; q += nt) {
        int bot, top, k0, k1;
        if (!decode_tile(q, L, n, nb, bot, top, k0, k1)) continue;
        int32_t Ur[kRB], acc[kRB];
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj) {
            const int m = bot + jj <= top ? bot + jj : top;
            Ur[jj] = FWD ? U[skew(m)] : U[skew(m)] - ndt1;
            acc[jj] = 0x7fffffff;
        }
        const int kf = k1 < bot ? k1 : bot;  // k < bot: every row of the block takes it
        int k = k0;
        while (k + 1 < kf) {
            // pairs inside the 32-aligned block of k, where skew(k) is linear in k
            const int kend = min(kf, (k | 31) + 1);
            const int32_t *pc = prev + skew(k), *pv = V + skew(k);
            for (; k + 1 < kend; k += 2, pc += 2, pv += 2) {
                const int32_t c0 = pc[0], v0 = pv[0], c1 = pc[1], v1 = pv[1];
#pragma unroll
                for (int jj = 0; jj < kRB; ++jj)
                    acc[jj] = __vimin3_s32(acc[jj], cand_s32(c0, Ur[jj], v0),
                                           cand_s32(c1, Ur[jj], v1));
            }
            if (k + 1 == kend && kend < kf) {  // a pair across the block boundary
                const int32_t c0 = prev[skew(k)], v0 = V[skew(k)];
                const int32_t c1 = prev[skew(k + 1)], v1 = V[skew(k + 1)];
#pragma unroll
                for (int jj = 0; jj < kRB; ++jj)
                    acc[jj] = __vimin3_s32(acc[jj], cand_s32(c0, Ur[jj], v0),
                                           cand_s32(c1, Ur[jj], v1));
                k += 2;
            }
        }
        if (k < kf) {
            const int32_t c0 = prev[skew(k)], v0 = V[skew(k)];
#pragma unroll
            for (int jj = 0; jj < kRB; ++jj) acc[jj] = min(acc[jj], cand_s32(c0, Ur[jj], v0));
        }
        if (k1 > bot) {  // row bot+jj takes k < bot+jj
#pragma unroll
            for (int u = 0; u < kRB - 1; ++u) {
                const int kk = bot + u;
                if (kk >= k1) break;
                if (kk < k0) continue;
                const int32_t c0 = prev[skew(kk)], v0 = V[skew(kk)];
#pragma unroll
                for (int jj = u + 1; jj < kRB; ++jj)
                    acc[jj] = min(acc[jj], cand_s32(c0, Ur[jj], v0));
            }
        }
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj)
            if (bot + jj <= top) atomicMin(&best[skew(bot + jj)], acc[jj]);
    }
}

template <bool FWD>
__device__ void solve_s32(const GroupArgs &a, int64_t i, int64_t dti, uint64_t xraw,
                          const uint64_t *P64c, const uint64_t *P64x, unsigned char *arrays,
                          uint32_t *bitsw, int32_t *table)
{
    const int L = a.L, t = threadIdx.x, nt = blockDim.x, Ls = group_ls(L);
    // bytes [0, 16Ls): U, V, two columns; [16Ls, 20Ls): partial minima. P64c /
    // P64x occupy bytes [16Ls, 32Ls): only U and V are written before the barrier.
    int32_t *U = reinterpret_cast<int32_t *>(arrays);
    int32_t *V = U + Ls;
    int32_t *colA = V + Ls;
    int32_t *colB = colA + Ls;
    int32_t *best = colB + Ls;
    const int32_t dt = int32_t(dti);
    const int32_t fcL = int32_t(P64c[L]);
    for (int m = t; m <= L; m += nt) {
        U[skew(m)] = FWD ? dt + int32_t(P64x[m]) : int32_t(P64c[m]);
        V[skew(m)] = FWD ? fcL - int32_t(P64c[m]) : -int32_t(P64x[m]);
    }
    __syncthreads();
    for (int m = 1 + t; m <= L; m += nt) {  // column 1
        const int32_t v = FWD ? fcL + U[skew(m)] - dt : U[skew(m)];
        colA[skew(m)] = v;
        best[skew(m)] = 0x7fffffff;
        if (DC_CHECK(tri_index(L, m, 1) < tri_cells(L))) table[tri_index(L, m, 1)] = v;
    }
    __syncthreads();
    int32_t *prev = colA, *cur = colB;
    for (int n = 2; n <= L; ++n) {
        fill_tiles_s32<FWD>(L, n, (n - 1) * dt, U, V, prev, best);
        __syncthreads();
        const int64_t cbase = tri_col(L, n) - n;
        for (int m = n + t; m <= L; m += nt) {
            const int32_t b = best[skew(m)];
            const int32_t v = FWD ? b - dt : b;
            cur[skew(m)] = v;
            best[skew(m)] = 0x7fffffff;
            if (DC_CHECK(cbase + m < tri_cells(L))) table[cbase + m] = v;
        }
        __syncthreads();
        int32_t *tmp = prev;
        prev = cur;
        cur = tmp;
    }

    // final pick and traceback by warp 0
    if (t < 32) {
        const int lane = t;
        // (B or E)[L][n] + n*dt, below 2^31
        const int32_t toB = FWD ? dt - U[skew(L)] : 0;  // A[L][n] + dt - Q[L] = B[L][n]
        int32_t bv = 0x7fffffff;
        int bn = 0x7fffffff;
        for (int n = 1 + lane; n <= L; n += 32) {
            const int32_t v = table[tri_index(L, L, n)] + toB + n * dt;
            if (v < bv) {  // n increases: strict keeps the lowest n in this lane
                bv = v;
                bn = n;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const int32_t ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int on = __shfl_xor_sync(0xffffffffu, bn, o);
            if (ov < bv || (ov == bv && on < bn)) {
                bv = ov;
                bn = on;
            }
        }
        const int s = bn;
        int err = 0;
        int m = L, n = s;
        while (n > 1) {
            const int32_t um = U[skew(m)];
            const int32_t u = FWD ? um : um - (n - 1) * dt;
            const int32_t target = table[tri_index(L, m, n)] + (FWD ? dt : 0);  // B + Q[m] = A + dt
            const int64_t pbase = tri_col(L, n - 1) - (n - 1);  // + k gives (k, n-1)
            int found = -1;
            for (int k0 = n - 1; k0 < m; k0 += 32) {
                const int k = k0 + lane;
                bool match = false;
                if (k < m) match = cand_s32(table[pbase + k], u, V[skew(k)]) == target;
                const unsigned bal = __ballot_sync(0xffffffffu, match);
                if (bal) {
                    found = k0 + __ffs(bal) - 1;
                    break;
                }
            }
            if (found < 0) {
                err = 1;
                break;
            }
            if (lane == 0) bitsw[(found - 1) >> 5] |= 1u << ((found - 1) & 31);
            __syncwarp();
            m = found;
            n -= 1;
        }
        if (lane == 0) {
            a.makespan[i] = int64_t(uint64_t(uint32_t(bv)) + xraw);
            if (a.nseg) a.nseg[i] = s;
            if (a.status) a.status[i] = err ? DC_ERR_INTERNAL : DC_OK;
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// Backward direction in 32 bits for instances whose (capped) bound exceeds 2^32.
// Shift every value by n*dt + GTR[m] (the link's own work):
//   E[m][n] = B[m][n] - n*dt - GTR[m]  lies in [0, BCR[m]]
// and Eq. 9 becomes
//   E[m][n] = min_{k} max(E[k][n-1], BCR[m] - ((n-1)*dt + GTR[k])),  E[m][1] = BCR[m].
// The second term only matters when positive (E >= 0), so (n-1)*dt + GTR[k] may be
// clamped to 2^31 - 1: with total backward compute below 2^31 every quantity fits
// a signed 32-bit word; with NY = -y a transition is one add-then-max and two
// candidates fold with one 3-input min, as in the 32-bit form above. Candidates
// of a cell differ from Eq. 9's by the row constant n*dt + GTR[m], so every
// argmin (and the lowest-k rule) is unchanged; B[L][n] = E[L][n] + n*dt + GTR[L].
constexpr int32_t kYClamp = 0x7fffffff;

__device__ __forceinline__ int32_t yclamp(uint64_t v) { return v < uint64_t(kYClamp) ? int32_t(v) : kYClamp; }

__device__ __forceinline__ void fill_tiles_ebwd(int L, int n, const int32_t *BC, const int32_t *NY,
                                                const int32_t *prev, int32_t *best)
{
    const int t = threadIdx.x, nt = blockDim.x;
    const int nb = (L - n + 1 + kRB - 1) / kRB;
    const int ng = (nb + 7) / 8;
    const int ntiles = 4 * ng * (ng + 1);
    for (int q = t; q < ntiles; q += nt) {
        int bot, top, k0, k1;
        if (!decode_tile(q, L, n, nb, bot, top, k0, k1)) continue;
        int32_t R[kRB], acc[kRB];
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj) {
            const int m = bot + jj <= top ? bot + jj : top;
            R[jj] = BC[skew(m)];
            acc[jj] = 0x7fffffff;
        }
        const int kf = k1 < bot ? k1 : bot;
        int k = k0;
        for (; k + 1 < kf; k += 2) {
            const int32_t v0 = prev[skew(k)], y0 = NY[skew(k)];
            const int32_t v1 = prev[skew(k + 1)], y1 = NY[skew(k + 1)];
#pragma unroll
            for (int jj = 0; jj < kRB; ++jj)
                acc[jj] = __vimin3_s32(acc[jj], __viaddmax_s32(R[jj], y0, v0), __viaddmax_s32(R[jj], y1, v1));
        }
        if (k < kf) {
            const int32_t v0 = prev[skew(k)], y0 = NY[skew(k)];
#pragma unroll
            for (int jj = 0; jj < kRB; ++jj) acc[jj] = min(acc[jj], __viaddmax_s32(R[jj], y0, v0));
        }
        if (k1 > bot) {
#pragma unroll
            for (int u = 0; u < kRB - 1; ++u) {
                const int kk = bot + u;
                if (kk >= k1) break;
                if (kk < k0) continue;
                const int32_t v0 = prev[skew(kk)], y0 = NY[skew(kk)];
#pragma unroll
                for (int jj = u + 1; jj < kRB; ++jj) acc[jj] = min(acc[jj], __viaddmax_s32(R[jj], y0, v0));
            }
        }
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj)
            if (bot + jj <= top) atomicMin(&best[skew(bot + jj)], acc[jj]);
    }
}

__device__ void solve_ebwd(const GroupArgs &a, int64_t i, int64_t dti, uint64_t shift,
                           const uint64_t *P64c, const uint64_t *P64x, unsigned char *arrays,
                           uint32_t *bitsw, int32_t *table)
{
    const int L = a.L, t = threadIdx.x, nt = blockDim.x, Ls = group_ls(L);
    // bytes [0, 8Ls): GTR (64-bit); then BCR, two columns, partial minima, NY (32-bit).
    // P64c / P64x occupy bytes [16Ls, 32Ls): read before anything past 16Ls is written.
    uint64_t *GT = reinterpret_cast<uint64_t *>(arrays);
    int32_t *BC = reinterpret_cast<int32_t *>(arrays + size_t(8) * Ls);
    int32_t *colA = BC + Ls;
    int32_t *colB = colA + Ls;
    int32_t *best = colB + Ls;
    int32_t *NY = best + Ls;
    for (int m = t; m <= L; m += nt) {
        GT[skew(m)] = P64x[m];
        BC[skew(m)] = int32_t(P64c[m]);
    }
    __syncthreads();
    const uint64_t dtv = uint64_t(dti);
    for (int m = 1 + t; m <= L; m += nt) {  // column 1, and Y for column 2
        const int32_t v = BC[skew(m)];
        colA[skew(m)] = v;
        best[skew(m)] = 0x7fffffff;
        if (DC_CHECK(tri_index(L, m, 1) < tri_cells(L))) table[tri_index(L, m, 1)] = v;
        NY[skew(m)] = -yclamp(dtv + GT[skew(m)]);
    }
    __syncthreads();
    int32_t *prev = colA, *cur = colB;
    for (int n = 2; n <= L; ++n) {
        fill_tiles_ebwd(L, n, BC, NY, prev, best);
        __syncthreads();
        const int64_t cbase = tri_col(L, n) - n;
        for (int m = n + t; m <= L; m += nt) {
            const int32_t v = best[skew(m)];
            cur[skew(m)] = v;
            best[skew(m)] = 0x7fffffff;
            if (DC_CHECK(cbase + m < tri_cells(L))) table[cbase + m] = v;
        }
        for (int k = n + t; k <= L; k += nt) NY[skew(k)] = -yclamp(uint64_t(n) * dtv + GT[skew(k)]);
        __syncthreads();
        int32_t *tmp = prev;
        prev = cur;
        cur = tmp;
    }
    if (t < 32) {
        const int lane = t;
        uint64_t bv = ~uint64_t(0);  // E[L][n] + n*dt: B[L][n] less the constant GTR[L]
        int bn = 0x7fffffff;
        for (int n = 1 + lane; n <= L; n += 32) {
            const uint64_t v = uint64_t(table[tri_index(L, L, n)]) + uint64_t(n) * dtv;
            if (v < bv) {
                bv = v;
                bn = n;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const uint64_t ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int on = __shfl_xor_sync(0xffffffffu, bn, o);
            if (ov < bv || (ov == bv && on < bn)) {
                bv = ov;
                bn = on;
            }
        }
        const int s = bn;
        int err = 0, m = L, n = s;
        while (n > 1) {
            const int32_t R = BC[skew(m)];
            const int32_t target = table[tri_index(L, m, n)];
            const int64_t pbase = tri_col(L, n - 1) - (n - 1);
            int found = -1;
            for (int k0 = n - 1; k0 < m; k0 += 32) {
                const int k = k0 + lane;
                bool match = false;
                if (k < m) {
                    const int32_t y = yclamp(uint64_t(n - 1) * dtv + GT[skew(k)]);
                    match = max(table[pbase + k], R - y) == target;
                }
                const unsigned bal = __ballot_sync(0xffffffffu, match);
                if (bal) {
                    found = k0 + __ffs(bal) - 1;
                    break;
                }
            }
            if (found < 0) {
                err = 1;
                break;
            }
            if (lane == 0) bitsw[(found - 1) >> 5] |= 1u << ((found - 1) & 31);
            __syncwarp();
            m = found;
            n -= 1;
        }
        if (lane == 0) {
            a.makespan[i] = int64_t(bv + GT[skew(L)] + shift);
            if (a.nseg) a.nseg[i] = s;
            if (a.status) a.status[i] = err ? DC_ERR_INTERNAL : DC_OK;
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// Forward direction in 32 bits for instances whose (capped) bound exceeds 2^32.
// Shift every value by n*dt + P[m] (the arrival time of the last pull):
//   E[m][n] = F[m][n] - n*dt - P[m]  lies in [0, FC[m]]
// and, with G[k] = FC[L] - FC[k], A[k] = E[k][n-1] + G[k] + P[k], Q[m] = dt + P[m],
// Eq. 8 becomes
//   E[m][n] + G[m] = min_{k} max(A[k] - Q[m], G[k]),  E[m][1] = FC[m].
// A[k] and Q[m] are large but only a non-negative difference below 2^30 matters,
// so inside a tile both are taken relative to P at the tile's lowest row: when
// the tile's rows span less than 2^30 of transfer, Q - P[bot] is signed 32-bit,
// the candidates of the far k (P[k] more than 2^30 below P[bot]) reduce to their
// G, and for the others A - P[bot] is signed 32-bit: a transition is one
// add-then-max (two candidates folding with one 3-input min); other tiles use
// the same formula in 64-bit. Candidates differ from Eq. 8's
// by the row constant n*dt + P[m] + G[m]: every argmin is unchanged, and
// F[L][n] = E[L][n] + n*dt + P[L]. Needs FC[L] < 2^29.
constexpr int32_t kSpan = 1 << 30;

__device__ __forceinline__ void fill_tiles_efwd(int L, int n, uint64_t dtv, const uint64_t *P,
                                                const int32_t *G, const uint64_t *A,
                                                int32_t *best)
{
    const int t = threadIdx.x, nt = blockDim.x;
    const int nb = (L - n + 1 + kRB - 1) / kRB;
    const int ng = (nb + 7) / 8;
    const int ntiles = 4 * ng * (ng + 1);
    for (int q = t; q < ntiles; q += nt) {
        int bot, top, k0, k1;
        if (!decode_tile(q, L, n, nb, bot, top, k0, k1)) continue;
        const int kf = k1 < bot ? k1 : bot;
        const uint64_t base = P[skew(bot)];
        int32_t acc[kRB];
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj) acc[jj] = 0x7fffffff;
        if (dtv + (P[skew(top)] - base) < uint64_t(kSpan)) {
            int32_t NQr[kRB];  // -(Q - base)
#pragma unroll
            for (int jj = 0; jj < kRB; ++jj) {
                const int m = bot + jj <= top ? bot + jj : top;
                NQr[jj] = -int32_t(dtv + (P[skew(m)] - base));
            }
            // k with P[k] < base - 2^30 have A[k] - base < -2^30 + FC[L] < -2^29 (A[k]
            // <= P[k] + FC[L]), so their candidate is exactly G[k]; G is non-increasing,
            // so together they contribute G at the last of them. The others have
            // A[k] - base in [-2^30, 2^30 + 2^29): the low 32-bit words' difference.
            int lo = k0, hi = kf;  // P is non-decreasing: the first k past the far ones
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (P[skew(mid)] + uint64_t(kSpan) < base)
                    lo = mid + 1;
                else
                    hi = mid;
            }
            if (lo > k0) {
                const int32_t gfar = G[skew(lo - 1)];
#pragma unroll
                for (int jj = 0; jj < kRB; ++jj) acc[jj] = min(acc[jj], gfar);
            }
            const uint32_t *Alo = reinterpret_cast<const uint32_t *>(A);  // low words
            const uint32_t blo = uint32_t(base);
            auto rel = [&](int k) { return int32_t(Alo[2 * skew(k)] - blo); };
            int k = lo;
            for (; k + 1 < kf; k += 2) {
                const int32_t a0 = rel(k), g0 = G[skew(k)];
                const int32_t a1 = rel(k + 1), g1 = G[skew(k + 1)];
#pragma unroll
                for (int jj = 0; jj < kRB; ++jj)
                    acc[jj] = __vimin3_s32(acc[jj], __viaddmax_s32(a0, NQr[jj], g0),
                                           __viaddmax_s32(a1, NQr[jj], g1));
            }
            if (k < kf) {
                const int32_t a0 = rel(k), g0 = G[skew(k)];
#pragma unroll
                for (int jj = 0; jj < kRB; ++jj) acc[jj] = min(acc[jj], __viaddmax_s32(a0, NQr[jj], g0));
            }
            if (k1 > bot) {
#pragma unroll
                for (int u = 0; u < kRB - 1; ++u) {
                    const int kk = bot + u;
                    if (kk >= k1) break;
                    if (kk < k0) continue;
                    const int32_t a0 = rel(kk), g0 = G[skew(kk)];
#pragma unroll
                    for (int jj = u + 1; jj < kRB; ++jj)
                        acc[jj] = min(acc[jj], __viaddmax_s32(a0, NQr[jj], g0));
                }
            }
        } else {  // wide tile: the same candidates in 64-bit
            int64_t Qw[kRB];
#pragma unroll
            for (int jj = 0; jj < kRB; ++jj) {
                const int m = bot + jj <= top ? bot + jj : top;
                Qw[jj] = int64_t(dtv + P[skew(m)]);
            }
            for (int k = k0; k < k1; ++k) {
                const int64_t ak = int64_t(A[skew(k)]);
                const int64_t gk = G[skew(k)];
#pragma unroll
                for (int jj = 0; jj < kRB; ++jj)
                    if (k < bot + jj) {
                        const int64_t x = ak - Qw[jj];
                        acc[jj] = min(acc[jj], int32_t(x > gk ? x : gk));
                    }
            }
        }
#pragma unroll
        for (int jj = 0; jj < kRB; ++jj)
            if (bot + jj <= top) atomicMin(&best[skew(bot + jj)], acc[jj]);
    }
}

__device__ void solve_efwd(const GroupArgs &a, int64_t i, int64_t dti, uint64_t shift,
                           const uint64_t *P64c, const uint64_t *P64x, unsigned char *arrays,
                           uint32_t *bitsw, int32_t *table)
{
    const int L = a.L, t = threadIdx.x, nt = blockDim.x, Ls = group_ls(L);
    // bytes [0, 8Ls): P (64-bit), [8Ls, 12Ls): G, [12Ls, 16Ls): column A,
    // [16Ls, 24Ls): A (64-bit), [24Ls, 28Ls): column B, [28Ls, 32Ls): partial minima.
    // P64c / P64x occupy bytes [16Ls, 32Ls): only P and G are written before the barrier.
    uint64_t *P = reinterpret_cast<uint64_t *>(arrays);
    int32_t *G = reinterpret_cast<int32_t *>(arrays + size_t(8) * Ls);
    int32_t *colA = G + Ls;
    uint64_t *A = reinterpret_cast<uint64_t *>(arrays + size_t(16) * Ls);
    int32_t *colB = reinterpret_cast<int32_t *>(arrays + size_t(24) * Ls);
    int32_t *best = colB + Ls;
    const uint64_t fcL = P64c[L];
    for (int m = t; m <= L; m += nt) {
        P[skew(m)] = P64x[m];
        G[skew(m)] = int32_t(fcL - P64c[m]);
    }
    __syncthreads();
    const uint64_t dtv = uint64_t(dti);
    for (int m = 1 + t; m <= L; m += nt) {  // column 1: E = FC[m]; A for column 2
        const int32_t v = int32_t(fcL) - G[skew(m)];
        colA[skew(m)] = v;
        best[skew(m)] = 0x7fffffff;
        if (DC_CHECK(tri_index(L, m, 1) < tri_cells(L))) table[tri_index(L, m, 1)] = v;
        A[skew(m)] = fcL + P[skew(m)];
    }
    __syncthreads();
    int32_t *prev = colA, *cur = colB;
    for (int n = 2; n <= L; ++n) {
        fill_tiles_efwd(L, n, dtv, P, G, A, best);
        __syncthreads();
        const int64_t cbase = tri_col(L, n) - n;
        for (int m = n + t; m <= L; m += nt) {
            const int32_t bm = best[skew(m)];
            const int32_t v = bm - G[skew(m)];
            cur[skew(m)] = v;
            best[skew(m)] = 0x7fffffff;
            if (DC_CHECK(cbase + m < tri_cells(L))) table[cbase + m] = v;
            A[skew(m)] = uint64_t(bm) + P[skew(m)];  // E + G + P for column n+1
        }
        __syncthreads();
        int32_t *tmp = prev;
        prev = cur;
        cur = tmp;
    }
    if (t < 32) {
        const int lane = t;
        uint64_t bv = ~uint64_t(0);  // E[L][n] + n*dt: F[L][n] less the constant P[L]
        int bn = 0x7fffffff;
        for (int n = 1 + lane; n <= L; n += 32) {
            const uint64_t v = uint64_t(table[tri_index(L, L, n)]) + uint64_t(n) * dtv;
            if (v < bv) {
                bv = v;
                bn = n;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const uint64_t ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int on = __shfl_xor_sync(0xffffffffu, bn, o);
            if (ov < bv || (ov == bv && on < bn)) {
                bv = ov;
                bn = on;
            }
        }
        const int s = bn;
        int err = 0, m = L, n = s;
        while (n > 1) {
            const int64_t Q = int64_t(dtv + P[skew(m)]);
            const int64_t target = int64_t(table[tri_index(L, m, n)]) + G[skew(m)];
            const int64_t pbase = tri_col(L, n - 1) - (n - 1);
            int found = -1;
            for (int k0 = n - 1; k0 < m; k0 += 32) {
                const int k = k0 + lane;
                bool match = false;
                if (k < m) {
                    const int64_t gk = G[skew(k)];
                    const int64_t x = int64_t(table[pbase + k]) + gk + int64_t(P[skew(k)]) - Q;
                    match = (x > gk ? x : gk) == target;
                }
                const unsigned bal = __ballot_sync(0xffffffffu, match);
                if (bal) {
                    found = k0 + __ffs(bal) - 1;
                    break;
                }
            }
            if (found < 0) {
                err = 1;
                break;
            }
            if (lane == 0) bitsw[(found - 1) >> 5] |= 1u << ((found - 1) & 31);
            __syncwarp();
            m = found;
            n -= 1;
        }
        if (lane == 0) {
            a.makespan[i] = int64_t(bv + P[skew(L)] + shift);
            if (a.nseg) a.nseg[i] = s;
            if (a.status) a.status[i] = err ? DC_ERR_INTERNAL : DC_OK;
        }
    }
    __syncthreads();
}

template <bool FWD>
__global__ void __launch_bounds__(256) group_kernel(GroupArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    const int L = a.L, t = threadIdx.x, nt = blockDim.x, Ls = group_ls(L);
    const int W = words_for(L);
    unsigned char *arrays = smem;
    uint32_t *bitsw = reinterpret_cast<uint32_t *>(smem + group_arrays_bytes(L));
    uint64_t *scratch =
        reinterpret_cast<uint64_t *>(smem + group_arrays_bytes(L) + group_bits_bytes(L));
    unsigned char *smem_table = smem + group_table_offset(L);
    unsigned char *slot =
        a.tables ? a.tables + size_t(blockIdx.x) * size_t(tri_cells(L)) * 8 : smem_table;
    // 64-bit prefix arrays live in the column buffers until the typed copy.
    uint64_t *P64c = reinterpret_cast<uint64_t *>(arrays) + 2 * Ls;
    uint64_t *P64x = P64c + Ls;

    const int64_t count = a.list_count ? int64_t(*a.list_count) : a.batch;
    for (int64_t j = blockIdx.x; j < count; j += gridDim.x) {
        const int64_t i = a.list ? int64_t(a.list[j]) : j;
        if (!DC_CHECK(i >= 0 && i < a.batch)) continue;
        const int64_t *crow = a.comp + i * L;
        const int64_t *xrow = a.xfer + i * L;
        const int64_t dti = a.dt[i];
        int bad_neg = dti < 0, bad_big = (dti >> 52) != 0;
        uint64_t sc = 0, sx = 0;
        for (int r = 1 + t; r <= L; r += nt) {
            const int col = FWD ? r - 1 : L - r;
            const int64_t cv = __ldg(crow + col), xv = __ldg(xrow + col);
            bad_neg |= (cv < 0) | (xv < 0);
            bad_big |= ((cv | xv) >> 52) != 0;
            P64c[r] = uint64_t(cv);
            P64x[r] = uint64_t(xv);
            sc += uint64_t(cv);
            sx += uint64_t(xv);
        }
        for (int w = t; w < W; w += nt) bitsw[w] = 0u;
        if (t == 0) {
            P64c[0] = 0;
            P64x[0] = 0;
        }
        const int any_neg = __syncthreads_or(bad_neg);
        const int any_big = __syncthreads_or(bad_big);
        int st = DC_OK;
        bool narrow = false, shifted32 = false;
        uint64_t shift = 0;
        if (any_neg) {
            st = DC_ERR_NEGATIVE;
        } else if (any_big) {
            st = DC_ERR_RANGE;
        } else {
            block_sum2_u64(sc, sx, scratch);  // raw totals (each term < 2^52, L <= 4096)
            if (exceeds_range(L, dti, sc, sx)) {
                st = DC_ERR_RANGE;
            } else {
                // cap the transfer costs at the total compute: no decision changes,
                // the makespan drops by sum(xfer) - sum(capped xfer)
                uint64_t cx = 0, unused = 0;
                for (int r = 1 + t; r <= L; r += nt) {
                    P64x[r] = P64x[r] < sc ? P64x[r] : sc;
                    cx += P64x[r];
                }
                block_sum2_u64(cx, unused, scratch);
                shift = sx - cx;
                block_prefix_u64(P64c, L, scratch);
                block_prefix_u64(P64x, L, scratch);
                const uint64_t bound = sc + cx + uint64_t(L) * uint64_t(dti);
                narrow = bound <= kNarrowLimit;
                shifted32 = bound <= kShiftedLimit;
            }
        }
        if (st != DC_OK) {
            if (t == 0) {
                a.makespan[i] = -int64_t(st);
                if (a.nseg) a.nseg[i] = 0;
                if (a.status) a.status[i] = st;
            }
            for (int w = t; w < W; w += nt) a.bits[i * W + w] = 0u;
            __syncthreads();
            continue;
        }
        if (shifted32)
            solve_s32<FWD>(a, i, dti, sx, P64c, P64x, arrays, bitsw,
                           reinterpret_cast<int32_t *>(slot));
        else if (!FWD && sc < uint64_t(kYClamp))
            solve_ebwd(a, i, dti, shift, P64c, P64x, arrays, bitsw,
                       reinterpret_cast<int32_t *>(slot));
        else if (FWD && sc < uint64_t(1) << 29)
            solve_efwd(a, i, dti, shift, P64c, P64x, arrays, bitsw,
                       reinterpret_cast<int32_t *>(slot));
        else if (narrow)
            solve<uint32_t, FWD>(a, i, dti, shift, P64c, P64x, arrays, bitsw,
                                 reinterpret_cast<uint32_t *>(slot));
        else
            solve<uint64_t, FWD>(a, i, dti, shift, P64c, P64x, arrays, bitsw,
                                 reinterpret_cast<uint64_t *>(slot));
        for (int w = t; w < W; w += nt) a.bits[i * W + w] = bitsw[w];
        __syncthreads();
    }
}

// Threads per instance: up to L = 256 a column has few (8 x 64) tiles, so one
// warp per instance and more instances per SM; deeper chains fill 8 warps.
int group_threads(int L) { return L <= 256 ? 32 : 256; }

}  // namespace

cudaError_t launch_group(bool forward, int64_t batch, int L, const int64_t *comp,
                         const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                         uint32_t *bits, int32_t *nseg, int32_t *status,
                         const uint32_t *list_count, const uint32_t *list, void *tables,
                         int64_t grid, cudaStream_t stream)
{
    if (grid <= 0) return cudaSuccess;
    GroupArgs a{batch, L, comp, xfer, dt, makespan, bits, nseg, status, list_count, list,
                static_cast<unsigned char *>(tables)};
    const size_t smem = group_smem_bytes(L, tables == nullptr);
    const int nt = forced_warps() ? 32 * forced_warps() : group_threads(L);
    cudaError_t e;
    if (forward) {
        e = cudaFuncSetAttribute(group_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(smem));
        if (e != cudaSuccess) return e;
        group_kernel<true><<<unsigned(grid), nt, smem, stream>>>(a);
    } else {
        e = cudaFuncSetAttribute(group_kernel<false>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
        group_kernel<false><<<unsigned(grid), nt, smem, stream>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace dc

DC_CHECKED_EXPORT(dp_group)
