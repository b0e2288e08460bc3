// Device building blocks of the short-L (1 <= L <= 16) DP, shared by the dense
// and list passes (dp_small.cu) and the fused generate-and-solve passes
// (dp_fused.cu). The design notes are at the top of dp_small.cu.
#pragma once

#include "gen_device.cuh"

namespace dc {

int sm_count();  // SMs of the current device (dp_small.cu)

namespace {


#ifndef DC_KEEP_COLS
#define DC_KEEP_COLS 4
#endif
#ifndef DC_SMALL_MINB
#define DC_SMALL_MINB 16  // resident single-warp CTAs per SM the registers must allow
#endif
#ifndef DC_TREE_MIN
#define DC_TREE_MIN 1
#endif
constexpr int kTbGroup = 4;  // traceback candidates loaded per round
// From this L on the dense and fused passes take their tiles from an atomic
// ticket (and the dense pass stages each tile beside its table); shorter rows
// take every grid-th tile, for which one atomic per tile costs more than the
// balance gains.
constexpr int kSplitMinL = 12;
constexpr int kKeepCols = DC_KEEP_COLS;  // the 32-bit pass stores columns 2..kKeepCols

// index of stored cell (m, n), 2 <= n <= L-1, n <= m <= L
__host__ __device__ constexpr int cell2(int L, int m, int n)
{
    return (n - 2) * L - (n - 2) * (n - 1) / 2 + (m - n);
}

// Row stride of the staging buffer in int64 units. Odd L: the odd stride L, so
// that the 16 lanes of a half-warp reading 64-bit words of their own rows hit 16
// distinct bank pairs. Even L: rows are copied and read as 16-byte pairs, so the
// stride is even (16-byte aligned rows) and 2 mod 4, so that the 8 lanes of a
// quarter-warp reading 16 bytes of their own rows hit 8 distinct 4-bank groups.
__host__ __device__ constexpr int stage_stride(int L)
{
    return (L % 2 == 1) ? L : (L % 4 == 2 ? L : L + 2);
}

// Table of the 64-bit pass: stored columns 2..C with C = min(keep, L-1) (KEEP = L
// keeps them all), then S[0..L] and R[0..L].
template <int L, typename T, int KEEP>
struct Small {
    static constexpr int kLast = KEEP < L - 1 ? KEEP : L - 1;  // last stored column
    static constexpr int kCells = kLast >= 2 ? cell2(L, L, kLast) + 1 : 0;
    static constexpr int kOffS = kCells;          // S[0..L]
    static constexpr int kOffR = kCells + L + 1;  // R[0..L]
    static constexpr int kLaneVals = kCells + 2 * (L + 1);
    static constexpr int kTableBytes = 32 * kLaneVals * int(sizeof(T));
};

// Shared memory of a warp of the 32-bit pass. Its table, per lane (32-bit words,
// lane-interleaved): word 0 unused, the kept cells of columns 2..kLast at
// 1 + cell2 (a traceback step loads one word below a column's first cell, which
// stays inside the table), then U[0..L]; column 1 is not stored, being U shifted
// by a constant. The tile's staging (comp and xfer rows at a padded stride, then
// dt) either shares the table's area (kSharedBytes) or lies beside it
// (kSplitBytes), so that the next tile can land while this one is solved.
template <int L>
struct Tab32 {
    static constexpr int kLast = kKeepCols < L - 1 ? kKeepCols : L - 1;  // last stored column
    static constexpr int kCells = kLast >= 2 ? cell2(L, L, kLast) + 1 : 0;
    static constexpr int kOffU = 1 + kCells;
    static constexpr int kWords = kOffU + L + 1;
    static constexpr int kBytes = 32 * kWords * 4;
    static constexpr int kStride = stage_stride(L);               // staging row stride (int64)
    static constexpr int kRowsBytes = 2 * 32 * kStride * 8;        // comp + xfer rows of a tile
    static constexpr int kSharedBytes = kRowsBytes > kBytes ? kRowsBytes : kBytes;
    static constexpr int kSplitBytes = kBytes + kRowsBytes + 32 * 8;  // table | rows | dt
};

template <typename T>
__device__ __forceinline__ T lds(const T *lane_base, int v) { return lane_base[32 * v]; }

// The fill. lw = this lane's values in shared memory (value v at lw[32*v]).
template <int L, bool FWD, typename T, int KEEP>
__device__ __forceinline__ void fill(const T (&S)[L + 1], const T (&Rb)[L + 1], T dtv, T c,
                                     T *lw, T &best_T, int &best_s)
{
    T col[L + 1];
#pragma unroll
    for (int m = 1; m <= L; ++m) col[m] = T((FWD ? T(dtv + Rb[m]) : Rb[m]) + S[m] + c);
    best_T = col[L];
    best_s = 1;
#pragma unroll
    for (int n = 2; n <= L; ++n) {
        // rows in descending order so column n overwrites column n-1 in place:
        // row m reads rows k < m, which still hold column n-1.
#pragma unroll
        for (int m = L; m >= n; --m) {
            const T R = FWD ? T(T(n) * dtv + Rb[m]) : Rb[m];
            constexpr int kMax = L;
            T cand[kMax];
            const int cnt = m - n + 1;  // k = n-1 .. m-1
#pragma unroll
            for (int j = 0; j < cnt; ++j) cand[j] = T(dmax(col[n - 1 + j], R) - S[n - 1 + j]);
            if (DC_TREE_MIN) {  // balanced tree: log-depth chains
#pragma unroll
                for (int w = 1; w < cnt; w *= 2) {
#pragma unroll
                    for (int j = 0; j + w < cnt; j += 2 * w) cand[j] = dmin(cand[j], cand[j + w]);
                }
            } else {
#pragma unroll
                for (int j = 1; j < cnt; ++j) cand[0] = dmin(cand[0], cand[j]);
            }
            col[m] = T(cand[0] + S[m] + c);
            if (n <= Small<L, T, KEEP>::kLast) lw[32 * cell2(L, m, n)] = col[m];
        }
        if (col[L] < best_T) {  // strict: the lowest n wins ties
            best_T = col[L];
            best_s = n;
        }
    }
}

// X[k][n-1] during the traceback: column 1 from S and R, others from the table.
template <int L, bool FWD, typename T, int KEEP>
__device__ __forceinline__ T prev_cell(const T *lw, int k, int nm1, T dtv, T c)
{
    using K = Small<L, T, KEEP>;
    if (nm1 == 1) {
        const T r = lds(lw, K::kOffR + k);
        return T((FWD ? T(dtv + r) : r) + lds(lw, K::kOffS + k) + c);
    }
    return lds(lw, cell2(L, k, nm1));
}

// Solve one instance (row data already reduced to 64-bit prefix sums in
// processing order) and write its outputs.
// Returns false (writing nothing) when the optimum's traceback needs a column the
// pass did not keep; the caller then lists the instance for the full pass.
template <int L, bool FWD, typename T, int KEEP>
__device__ __forceinline__ bool solve(const uint64_t (&Pc)[L + 1], const uint64_t (&Px)[L + 1],
                                      int64_t dti, uint64_t shift, T *lw, int64_t i,
                                      int64_t *makespan, uint32_t *bits, int32_t *nseg,
                                      int32_t *status)
{
    using K = Small<L, T, KEEP>;
    constexpr int W = (L - 1 + 31) / 32;
    T S[L + 1], Rb[L + 1];
#pragma unroll
    for (int m = 0; m <= L; ++m) {
        S[m] = T(FWD ? Pc[m] : Px[m]);
        Rb[m] = T(FWD ? Px[m] : Pc[m]);
        lw[32 * (K::kOffS + m)] = S[m];
        lw[32 * (K::kOffR + m)] = Rb[m];
    }
    const T dtv = T(dti);
    const T c = FWD ? T(0) : dtv;
    T Tbest;
    int s;
    fill<L, FWD, T, KEEP>(S, Rb, dtv, c, lw, Tbest, s);
    if (s - 1 > K::kLast && s - 1 >= 2) return false;

    // traceback: from (L, s) step to the lowest k whose candidate equals the
    // cell, set p_k / g_k, continue at (k, n-1)
    uint32_t word = 0;
    int err = 0;
    int m = L, n = s;
    T cell = Tbest;
    while (n > 1) {
        const T rm = lds(lw, K::kOffR + m);
        const T R = FWD ? T(T(n) * dtv + rm) : rm;
        const T target = T(cell - lds(lw, K::kOffS + m) - c);
        // candidates in groups of kTbGroup: the loads issue back to back, then the
        // compares run from the highest k down so that the lowest match wins
        int k = -1;
        T fk = T(0);
        for (int k0 = n - 1; k0 < m && k < 0; k0 += kTbGroup) {
            T f[kTbGroup], sk[kTbGroup];
#pragma unroll
            for (int u = 0; u < kTbGroup; ++u) {
                const int kk = k0 + u < m ? k0 + u : m - 1;  // stay inside column n-1
                f[u] = prev_cell<L, FWD, T, KEEP>(lw, kk, n - 1, dtv, c);
                sk[u] = lds(lw, K::kOffS + kk);
            }
#pragma unroll
            for (int u = kTbGroup - 1; u >= 0; --u) {
                if (k0 + u < m && T(dmax(f[u], R) - sk[u]) == target) {
                    k = k0 + u;
                    fk = f[u];
                }
            }
        }
        if (k < 0) {  // cannot happen: the fill and this check use the same arithmetic
            err = 1;
            break;
        }
        word |= 1u << ((k - 1) & 31);
        m = k;
        n -= 1;
        cell = fk;
    }
    makespan[i] = int64_t(uint64_t(Tbest) + shift);
    if (nseg) nseg[i] = s;
    if (status) status[i] = err ? DC_ERR_INTERNAL : DC_OK;
    if (W > 0) bits[i * W] = word;
    return true;
}

// ---------------------------------------------------------------------------
// The 32-bit pass in shifted form. Every value is taken relative to the time
// the last pull (forward) or push (backward) of its cell can start, which turns
// a transition into one add-then-max and the minimum into 3-input mins: on
// GB300 both are single integer-ALU instructions (the DPX forms), so a transition
// costs 1.5 ALU-pipe instructions instead of 2.
//
// forward (P = transfer prefix, FC = compute prefix, G[k] = FC[L] - FC[k],
// Q[m] = dt + P[m]): with B = X - n*dt - P[m] + G[m] (X as above) and
// A[k] = B[k][n-1] + P[k],
//   B[m][n] + Q[m] = min_k max(G[k] + Q[m], A[k]),  A[m][1] = FC[L] + P[m],
//   X[L][n] = B[L][n] + n*dt + P[L];
// the next column's A[m] is that minimum less dt;
// backward (BC = compute prefix, NGT[k] = -(transfer prefix), U = BC - dt):
// with F = X - dt - S[m],
//   F[m][n] - dt = min_k max(U[m] + NGT[k], F[k][n-1]),  F[m][1] = BC[m],
//   X[L][n] = F[L][n] + dt + S[L];
// the next column's F[m] is that minimum plus dt.
// Both are min_k max(U[m] + V[k], C[k]) with a row constant U, the same in every
// column, and the previous column C in the max operand. Each candidate differs from Eq. 8/9's by a
// constant of its row, so every argmin is the same. All values and sums lie in
// [-2^31, 2^31) when the capped bound L*dt + sum(comp) + sum(capped xfer) is
// below 2^31; other instances take the 64-bit pass. The table stores A (forward)
// or F (backward) for columns 1..kKeepCols and the row U (Q forward, BC - dt
// backward); V (G forward, NGT backward) stays in registers.

// Minimum of c[0..cnt-1] (cnt a compile-time constant after unrolling): two
// chains of 3-input mins, so that each row has two independent dependency chains
// and the rows of a column interleave.
template <int N>
__device__ __forceinline__ int32_t min_fold3(const int32_t (&c)[N], int cnt)
{
    if (cnt == 1) return c[0];
    if (cnt == 2) return min(c[0], c[1]);
    int32_t a = c[0], b = c[1];
    int j = 2;
#pragma unroll
    for (; j + 3 < cnt; j += 4) {
        a = __vimin3_s32(a, c[j], c[j + 1]);
        b = __vimin3_s32(b, c[j + 2], c[j + 3]);
    }
    if (j + 1 < cnt) return __vimin3_s32(__vimin3_s32(a, b, c[j]), c[j + 1], cnt > j + 2 ? c[j + 2] : c[j + 1]);
    if (j < cnt) return __vimin3_s32(a, b, c[j]);
    return min(a, b);
}

// The direction `fwd` is an argument: the dense passes pass a compile-time
// constant, which folds every choice below away; the fused pass solves both
// directions with one copy of this code.
template <int L>
__device__ __forceinline__ void fill_e(const bool fwd, const int32_t (&U)[L + 1],
                                       const int32_t (&V)[L + 1], int32_t dt, int32_t fcL,
                                       int32_t *lw, int32_t &bestV, int &best_s)
{
    using K = Tab32<L>;
    // forward: U = Q, V = G, col = A; backward: U = BC - dt, V = NGT, col = F
    const int32_t dt2 = 2 * dt;
    const int32_t c1 = fwd ? fcL - dt : dt;  // column 1 is U + c1
    const int32_t sdt = fwd ? -dt : dt;      // column n is its minimum + sdt
    const int32_t uL = fwd ? U[L] : 0;       // row L's minimum less uL: B[L][n] or F[L][n] - dt
    const int32_t step = fwd ? dt : 0, base = fwd ? 0 : dt2;
    int32_t col[L + 1];
#pragma unroll
    for (int m = 1; m <= L; ++m) col[m] = U[m] + c1;
    bestV = fwd ? fcL + dt : U[L] + dt2;
    best_s = 1;
#pragma unroll
    for (int n = 2; n <= L; ++n) {
        int32_t last = 0;  // B[L][n] (forward) or F[L][n] - dt (backward)
#pragma unroll
        for (int m = L; m >= n; --m) {  // descending: column n overwrites column n-1 in place
            const int cnt = m - n + 1;  // k = n-1 .. m-1
            const int32_t u = U[m];
            int32_t c[L];
#pragma unroll
            for (int j = 0; j < cnt; ++j) c[j] = __viaddmax_s32(u, V[n - 1 + j], col[n - 1 + j]);
            const int32_t b = min_fold3<L>(c, cnt);
            if (m == L) last = b - uL;
            col[m] = b + sdt;
            if (n <= K::kLast) lw[32 * (1 + cell2(L, m, n))] = col[m];
        }
        const int32_t v = last + n * step + base;  // X[L][n] - P[L] or X[L][n] - S[L]
        if (v < bestV) {  // strict: the lowest n wins ties
            bestV = v;
            best_s = n;
        }
    }
}

// The fill, the traceback and the outputs of one instance in shifted form, from
// its U and V rows (forward: U = dt + capped transfer prefix, V = FC[L] - compute
// prefix; backward: U = compute prefix - dt, V = -capped transfer prefix) and the raw
// transfer sum. Returns false (writing nothing) when the traceback needs a column
// the pass did not keep.
template <int L>
__device__ __forceinline__ bool solve_uv(const bool fwd, const int32_t (&U)[L + 1],
                                         const int32_t (&V)[L + 1], int32_t dt, uint64_t xraw,
                                         int32_t *lw, int64_t i, int64_t *makespan,
                                         uint32_t *bits, int32_t *nseg, int32_t *status)
{
    using K = Tab32<L>;
    constexpr int W = (L - 1 + 31) / 32;
    const int32_t fcL = V[0];  // forward: FC[L]
#pragma unroll
    for (int m = 0; m <= L; ++m) lw[32 * (K::kOffU + m)] = U[m];  // the traceback reads U[m]
    int32_t bestV;
    int s;
    fill_e<L>(fwd, U, V, dt, fcL, lw, bestV, s);
    if (s - 1 > K::kLast && s - 1 >= 2) return false;

    // from (L, s) step to the lowest k whose candidate equals the cell, set
    // p_k / g_k, continue at (k, n-1). A step compares every candidate at once
    // (V still in registers, compile-time k): bit k of `hit` is set when
    // candidate k equals the cell, and the lowest k inside [n-1, m-1] is the one
    // Algorithm 3/4 keeps. The loads of k outside that range read other words of
    // the lane's table and are masked off.
    uint32_t word = 0;
    int err = 0;
    int m = L, n = s;
    int32_t target = fwd ? bestV - s * dt + U[L] : bestV - 2 * dt;  // B[L][s] + Q[L] or F[L][s] - dt
    // column 1 is U shifted by off1 (A[k][1] = FC[L] + U[k] - dt forward, F[k][1] =
    // U[k] + dt backward): its step reads U and compares the candidate and the
    // cell both less off1, max(u + V, f + off1) = max(u - off1 + V, f) + off1
    const int32_t off1 = fwd ? fcL - dt : dt;
    while (n > 1) {
        const int nm1 = n - 1;
        const int32_t off = nm1 == 1 ? off1 : 0;
        const int32_t u = lds(lw, K::kOffU + m) - off;
        const int32_t tgt = target - off;
        // cell (k, n-1) of a kept column is word base + k (>= 0 for every k >= 1)
        const int base = nm1 == 1 ? K::kOffU : 1 + cell2(L, 0, nm1);
        uint32_t hit = 0u;
#pragma unroll
        for (int k = 1; k < L; ++k) {
            if (__viaddmax_s32(u, V[k], lds(lw, base + k)) == tgt) hit |= 1u << k;
        }
        hit &= ((2u << (m - 1)) - 1u) & ~((1u << nm1) - 1u);  // k in [n-1, m-1]
        if (hit == 0u) {  // cannot happen: the fill and this check use the same arithmetic
            err = 1;
            break;
        }
        const int k = __ffs(int(hit)) - 1;
        word |= 1u << ((k - 1) & 31);
        const int32_t fk = lds(lw, base + k) + off;  // the cell (k, n-1): B + Q[k] = A + dt, or F - dt
        target = fwd ? fk + dt : fk - dt;
        m = k;
        n = nm1;
    }
    makespan[i] = int64_t(uint64_t(uint32_t(bestV)) + xraw);
    if (nseg) nseg[i] = s;
    if (status) status[i] = err ? DC_ERR_INTERNAL : DC_OK;
    if (W > 0) bits[i * W] = word;
    return true;
}

// U and V from 64-bit prefix sums (the caller has checked the 32-bit range).
template <int L, bool FWD>
__device__ __forceinline__ void shifted_uv(const uint64_t (&Pc)[L + 1], const uint64_t (&Px)[L + 1],
                                           int64_t dti, int32_t (&U)[L + 1], int32_t (&V)[L + 1])
{
    const int32_t dt = int32_t(dti);
    const int32_t fcL = int32_t(Pc[L]);
#pragma unroll
    for (int m = 0; m <= L; ++m) {
        U[m] = FWD ? dt + int32_t(Px[m]) : int32_t(Pc[m]) - dt;
        V[m] = FWD ? fcL - int32_t(Pc[m]) : -int32_t(Px[m]);
    }
}

__host__ __device__ constexpr int ceil_log2(int x) { return x <= 1 ? 0 : 1 + ceil_log2((x + 1) / 2); }

// The row's U and V in 32-bit arithmetic, for the common row whose costs all lie
// in [0, 2^32) with every compute cost below 2^31 / L (then every compute sum is
// exact in 32 bits) and dt below 2^31. rc, rx: the row's costs in layer order.
// Returns false, computing nothing, for any other row: the caller takes the
// 64-bit route (which also classifies negative and out-of-range input). On true,
// `wide` says whether the capped bound L*dt + sum(comp) + sum(capped xfer) exceeds
// the shifted form's limit. Transfers are capped at the total compute as in
// row_prefix; the sums of capped transfers and raw transfers are kept in 64 bits.
template <int L, bool FWD>
__device__ __forceinline__ bool fast_uv(const int64_t *rc, const int64_t *rx, int64_t dti,
                                        int32_t (&U)[L + 1], int32_t (&V)[L + 1], uint64_t &xraw,
                                        bool &wide)
{
    constexpr int kCompBits = 31 - ceil_log2(L);
    uint32_t cl[L], xl[L];
    uint32_t hor = uint32_t(uint64_t(dti) >> 31), cor = 0u, tc = 0u;
    if constexpr (L % 2 == 0) {  // 16-byte rows: two costs per load
#pragma unroll
        for (int q = 0; q < L; q += 2) {
            const uint4 c = *reinterpret_cast<const uint4 *>(rc + q);
            const uint4 x = *reinterpret_cast<const uint4 *>(rx + q);
            const int r0 = FWD ? q : L - 1 - q, r1 = FWD ? q + 1 : L - 2 - q;
            cl[r0] = c.x;
            cl[r1] = c.z;
            xl[r0] = x.x;
            xl[r1] = x.z;
            hor |= c.y | x.y;
            hor |= c.w | x.w;
            cor |= c.x | c.z;
            tc += c.x + c.z;
        }
    } else {
#pragma unroll
        for (int r = 0; r < L; ++r) {
            const int col = FWD ? r : L - 1 - r;
            const uint2 c = *reinterpret_cast<const uint2 *>(rc + col);
            const uint2 x = *reinterpret_cast<const uint2 *>(rx + col);
            cl[r] = c.x;
            xl[r] = x.x;
            hor |= c.y | x.y;
            cor |= c.x;
            tc += c.x;
        }
    }
    if ((hor | (cor >> kCompBits)) != 0u) return false;
    uint32_t u = FWD ? uint32_t(dti) : 0u - uint32_t(dti), v = FWD ? tc : 0u;
    U[0] = int32_t(u);
    V[0] = int32_t(v);
    uint64_t px = 0, xr = 0;
#pragma unroll
    for (int r = 0; r < L; ++r) {
        const uint32_t xc = min(xl[r], tc);
        px += xc;
        xr += xl[r];
        if (FWD) {
            u += xc;
            v -= cl[r];
        } else {
            u += cl[r];
            v -= xc;
        }
        U[r + 1] = int32_t(u);
        V[r + 1] = int32_t(v);
    }
    xraw = xr;
    wide = uint64_t(L) * uint64_t(dti) + tc + px > uint64_t(kShiftedLimit);
    return true;
}

__device__ __forceinline__ void cp_async8(void *smem_dst, const void *gmem_src)
{
    const uint32_t d = uint32_t(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(d), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src)
{
    const uint32_t d = uint32_t(__cvta_generic_to_shared(smem_dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }

// Issue the copies of tile `base` (rows base..base+rows-1) into the staging area:
// 16-byte copies of cost pairs when L is even and both cost arrays are 16-byte
// aligned (`pairs`; every pair then starts on a 16-byte boundary on both sides),
// else 8-byte copies.
template <int L>
__device__ __forceinline__ void stage_tile(int64_t *stC, int64_t *stX, const int64_t *comp,
                                           const int64_t *xfer, int64_t base, int rows, int lane,
                                           bool pairs)
{
    constexpr int kStride = stage_stride(L);
    const int64_t *gC = comp + base * L;
    const int64_t *gX = xfer + base * L;
    if (L % 2 == 0 && pairs) {
        constexpr int H = L / 2 > 0 ? L / 2 : 1;  // pairs per row
        const int np = rows * H;
        for (int p = lane; p < np; p += 32) {
            const int r = p / H, cidx = 2 * (p - r * H);
            cp_async16(stC + r * kStride + cidx, gC + 2 * p);
            cp_async16(stX + r * kStride + cidx, gX + 2 * p);
        }
    } else {
        const int nel = rows * L;
        for (int e = lane; e < nel; e += 32) {
            const int r = e / L, cidx = e - r * L;
            cp_async8(stC + r * kStride + cidx, gC + e);
            cp_async8(stX + r * kStride + cidx, gX + e);
        }
    }
    cp_async_commit();
}

// Read this lane's row (processing order) into 64-bit prefix sums; flag bad
// input. Transfer costs are capped at the row's total compute: shifted by
// n*dt + (transfer prefix), every DP value lies in [0, total compute] and the
// recurrence sees transfer costs only through saturating differences, so the cap
// changes no comparison (same decision) and lowers the makespan by exactly
// sum(xfer) - sum(capped xfer), returned in `shift`.
template <int L, bool FWD, typename Src>
__device__ __forceinline__ void row_prefix(Src get, uint64_t (&Pc)[L + 1], uint64_t (&Px)[L + 1],
                                           uint64_t &xraw, bool &neg, bool &big)
{
    uint64_t tc = 0;
    xraw = 0;
#pragma unroll
    for (int r = 1; r <= L; ++r) {
        int64_t cv, xv;
        get(FWD ? r - 1 : L - r, cv, xv);
        neg |= (cv < 0) | (xv < 0);
        big |= ((cv | xv) >> 52) != 0;
        tc += uint64_t(cv);
        xraw += uint64_t(xv);
    }
    Pc[0] = 0;
    Px[0] = 0;
#pragma unroll
    for (int r = 1; r <= L; ++r) {
        int64_t cv, xv;
        get(FWD ? r - 1 : L - r, cv, xv);
        Pc[r] = Pc[r - 1] + uint64_t(cv);
        Px[r] = Px[r - 1] + (uint64_t(xv) < tc ? uint64_t(xv) : tc);
    }
}

// A staged row (rc, rx: its costs in layer order) to the 32-bit pass's U and V:
// fast_uv when the row fits, else 64-bit prefix sums with the input checks.
// st: DC_OK or the row's error; wide: the capped bound exceeds the shifted form's
// limit (the instance belongs to the 64-bit pass).
template <int L, bool FWD>
__device__ __forceinline__ void row_uv(const int64_t *rc, const int64_t *rx, int64_t dti,
                                       int32_t (&U)[L + 1], int32_t (&V)[L + 1], uint64_t &xraw,
                                       bool &wide, int &st)
{
    st = DC_OK;
    if (fast_uv<L, FWD>(rc, rx, dti, U, V, xraw, wide)) return;
    uint64_t Pc[L + 1], Px[L + 1];
    bool neg = dti < 0, big = (dti >> 52) != 0;
    row_prefix<L, FWD>(
        [&](int col, int64_t &cv, int64_t &xv) {
            cv = rc[col];
            xv = rx[col];
        },
        Pc, Px, xraw, neg, big);
    if (neg)
        st = DC_ERR_NEGATIVE;
    else if (big || uint64_t(L) * uint64_t(dti) + Pc[L] + xraw >= uint64_t(kRangeLimit))
        st = DC_ERR_RANGE;
    wide = uint64_t(L) * uint64_t(dti) + Pc[L] + Px[L] > kShiftedLimit;  // capped bound
    shifted_uv<L, FWD>(Pc, Px, dti, U, V);
}

__device__ __forceinline__ void write_failure(int st, int64_t i, int W, int64_t *makespan,
                                              uint32_t *bits, int32_t *nseg, int32_t *status)
{
    makespan[i] = -int64_t(st);
    if (nseg) nseg[i] = 0;
    if (status) status[i] = st;
    for (int w = 0; w < W; ++w) bits[i * W + w] = 0u;
}

}  // namespace
}  // namespace dc
