// Warp-per-instance DynaComm DP for deep chains (L > 256): Eq. 8 (the forward
// problem of Algorithm 3) and Eq. 9 (the backward problem of Algorithm 4).
//
// Same processing-order template as the other kernels:
//   X[m][n] = min_{k in [n-1, m-1]} max(X[k][n-1], R(m,n)) - S[k] + S[m] + c,
// solved in one of three shifted signed 32-bit forms (transfers capped at the
// total compute first, which changes no decision):
//   S32  capped bound below 2^31 (both directions): the form of the short
//        kernels, cand = max(U[m] + V[k], C[k]) with C the previous column;
//   EBWD backward, total compute below 2^31: cand = max(BC[m] + NY[k], E[k])
//        with NY[k] = -min((n-1)dt + GT[k], 2^31 - 1) (clamping is exact: the
//        candidate only matters when the first term is positive);
//   EFWD forward, total compute below 2^29: cand = max(A[k] - Q[m], G[k]) with
//        A = E + G + P, Q = dt + P, G[k] = FC[L] - FC[k]; A - Q is taken from
//        the low 32-bit words (exact while the true difference lies in
//        [-2^31, 2^31); see the plan below for the k where it does not).
// Every one is max(u[m] + x[k], y[k]): one add-then-max per transition and one
// 3-input min per two candidates (1.5 integer-ALU instructions on GB300). The
// pairs (x[k], y[k]) of the previous column sit interleaved in shared memory,
// so one 16-byte broadcast load feeds two candidates of every row of a lane.
// Other instances (the 32-bit and 64-bit literal templates), and those whose
// optimum has more than kKeep + 1 segments, go to a work list that the
// CTA-per-instance kernel (dp_group.cu) solves afterwards.
//
// Mapping (one warp per instance, persistent CTAs of one warp taking instances
// from a ticket):
//  * a column is cut, from row L down, into blocks of up to 8 strips of 32
//    rows; lane l owns row bot + l + 32 j of strip j. A block's candidates are
//    a rectangle k in [n-1, bot-1] that every row takes, walked in pairs, and a
//    triangle k in [bot, top] walked strip by strip: in strip q's 32 k, the
//    strips above take every k and strip q takes k < its row (lane-masked).
//    Block bottoms have the parity that makes every pair 16-byte aligned;
//  * entries of the previous column below n-1 (and 33 padding entries below
//    k = 0) hold y = INT_MAX, which makes their candidate INT_MAX: loops may
//    start below n-1, and blocks keep their full height near the column's
//    bottom (rows below n are computed and not written);
//  * EFWD: a block is exact in 32 bits only if its rows' transfer prefixes
//    span at most 1.5 * 2^30 (and dt + span <= 2^31). The per-instance plan
//    cuts the column into the largest blocks (256, 128, 64 or 32 rows) that
//    satisfy this, and for each records kF, the first k with
//    P[k] >= P[top] + dt - 2^31. Every k < kF has A[k] - Q[m] < 0 for every row
//    of the block, so its candidate is exactly G[k]; G is non-increasing, so
//    together they contribute G[kF - 1], which is loaded into the minima before
//    the loop starts at kF. An instance whose plan needs blocks of fewer than
//    32 rows goes to the work list;
//  * the fill keeps values only. The traceback re-derives Path[m][n] as the
//    lowest k whose candidate equals the cell (the k Algorithms 3/4 keep), with
//    one ballot per 32 candidates, from columns 1..kKeep kept in a per-CTA
//    global slot, and the last row X[L][.] kept for the final pick;
//  * the profile rows arrive by cp.async.bulk (one 1D bulk copy per row into
//    shared memory, completion on an mbarrier) when they are 16-byte aligned,
//    else by plain loads.
#include "common.cuh"

namespace dc {
namespace {

constexpr int kKeep = 64;    // traceback columns kept per instance
constexpr int kPad = 32;     // neutral pair entries below k = 0
constexpr int32_t kInf = 0x7fffffff;
constexpr int32_t kYCl = 0x7fffffff;
constexpr int kMaxStrips = 8;
constexpr int64_t kSpanLimit = (int64_t(3) << 29);  // 1.5 * 2^30
constexpr int64_t kTwo31 = int64_t(1) << 31;

enum Form { kS32 = 0, kEbwd = 1, kEfwd = 2 };

__host__ __device__ inline size_t al16(size_t b) { return (b + 15) / 16 * 16; }
__host__ __device__ inline int deep_koff(int L) { return kPad + ((L + 1) & 1); }
__host__ __device__ inline int deep_entries(int L) { return L + kPad + 2; }
__host__ __device__ inline size_t deep_pair_bytes(int L) { return al16(size_t(deep_entries(L)) * 8); }
__host__ __device__ inline int deep_plan_max(int L) { return L / 32 + 2; }
// One pair buffer with one warp per instance (the column is updated in place:
// blocks run top-down and read only rows below their own top), two otherwise.
__host__ __device__ inline int deep_buffers(int NW) { return NW == 1 ? 1 : 2; }
__host__ __device__ inline size_t deep_urow_off(int L, int NW) { return 16 + deep_buffers(NW) * deep_pair_bytes(L); }
__host__ __device__ inline size_t deep_bits_off(int L, int NW) { return deep_urow_off(L, NW) + al16(size_t(L + 1) * 4); }
__host__ __device__ inline size_t deep_plan_off(int L, int NW) { return deep_bits_off(L, NW) + al16(size_t(words_for(L) + 1) * 4); }
__host__ __device__ inline size_t deep_smem(int L, int NW) { return deep_plan_off(L, NW) + size_t(NW) * (deep_plan_max(L) + 1) * 16; }

__host__ __device__ inline int64_t kept_cols(int L) { return L < kKeep ? L : kKeep; }
__host__ __device__ inline int64_t kept_cells(int L)
{
    const int64_t K = kept_cols(L);
    return K * L - K * (K - 1) / 2;
}
// Per-CTA global slot: P or GT (64-bit prefix), the last row X[L][.], G (forward
// E form), then the kept columns 1..kKeep in the column-major triangle layout.
__host__ __device__ inline size_t slot_last_off(int L) { return size_t(L + 1) * 8; }
__host__ __device__ inline size_t slot_g_off(int L) { return size_t(L + 1) * 12; }
__host__ __device__ inline size_t slot_kept_off(int L) { return al16(size_t(L + 1) * 16); }
__host__ __device__ inline size_t slot_bytes(int L)
{
    return (slot_kept_off(L) + size_t(kept_cells(L)) * 4 + 255) / 256 * 256;
}

struct DeepArgs {
    int64_t lo, count;  // this launch solves instances lo .. lo + count - 1
    int L;
    const int64_t *comp, *xfer, *dt;
    int64_t *makespan;
    uint32_t *bits;
    int32_t *nseg, *status;
    uint32_t *ticket;                // instances taken so far (zero before the launch)
    uint32_t *list_count, *list;     // instances left to the CTA-per-instance kernel
    uint32_t *busy;                  // slot bitmap: bit set while a CTA holds the slot (zero before the first launch)
    unsigned char *slots;
    size_t slot_bytes;
    int nslots;
    int bulk;                        // profile rows may be staged with cp.async.bulk
};

// ------------------------------------------------------------- async staging
__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t *bar)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}
// Waits for the barrier's phase `parity` to complete, at most `tries` polls.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, int tries)
{
    for (int t = 0; t < tries; ++t) {
        uint32_t done = 0;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(smem_u32(bar)), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

// ------------------------------------------------------------- small helpers
__device__ __forceinline__ int32_t va(int32_t u, int32_t x, int32_t y) { return __viaddmax_s32(u, x, y); }
__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ uint64_t warp_excl_scan_u64(uint64_t v, int lane)
{
    uint64_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint64_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    return x - v;
}
__device__ __forceinline__ int32_t yclamp64(int64_t v) { return v < int64_t(kYCl) ? int32_t(v) : kYCl; }

// One block of R strips of column n: strip j holds rows b0 + S j + lane (S =
// 32 x the warps sharing the instance; top = b0 + S (R-1) + 31). Candidates:
// the rectangle k in [k_lo, b0 - 1] that every strip takes, then for each strip
// J its own 32 k (strips above take them all, strip J the k below its row) and,
// when S > 32, the gap up to the next strip (strips above J only). Then the
// finalised rows go to the next column's pairs, the kept table and the last row.
template <int R, int FORM, bool FWD, int S>
__device__ __forceinline__ void block(int L, int n, int b0, int k_lo, bool far, int32_t gfar,
                                      int64_t dt, const int2 *__restrict__ cur, int2 *__restrict__ nxt,
                                      const int32_t *__restrict__ urow, int32_t *__restrict__ kept,
                                      int32_t *__restrict__ last, int koff, int lane)
{
    // the block's pair entries (from k_lo - 1 to its top) and rows lie inside
    // the arrays
    if (!DC_CHECK(k_lo - 1 + koff >= 0 && b0 + koff >= 0 && b0 + S * (R - 1) + 31 <= L &&
                  b0 + S * (R - 1) + 31 + koff < deep_entries(L)))
        return;
    int32_t u[R], acc[R];
    const int32_t ndt1 = (FORM == kS32 && !FWD) ? int32_t(int64_t(n - 1) * dt) : 0;
#pragma unroll
    for (int j = 0; j < R; ++j) {
        int m = b0 + lane + S * j;
        m = m < 0 ? 0 : m;
        u[j] = urow[m] - ndt1;
        acc[j] = far ? gfar : kInf;
    }
    // rectangle: k in [k_lo, b0 - 1], every row
    int k = k_lo;
    if ((k + koff) & 1) {
        if (FORM == kEfwd) {  // k_lo - 1 may be a far k: take k_lo on its own
            const int2 p = cur[k + koff];
#pragma unroll
            for (int j = 0; j < R; ++j) acc[j] = min(acc[j], va(u[j], p.x, p.y));
            ++k;
        } else {
            --k;  // k_lo - 1 = n - 2 is a neutral entry
        }
    }
    {
        const int4 *pp = reinterpret_cast<const int4 *>(cur + koff + k);
        const int4 *pe = reinterpret_cast<const int4 *>(cur + koff + b0);
#pragma unroll 2
        for (; pp < pe; ++pp) {
            const int4 p = *pp;
#pragma unroll
            for (int j = 0; j < R; ++j)
                acc[j] = __vimin3_s32(acc[j], va(u[j], p.x, p.y), va(u[j], p.z, p.w));
        }
    }
#pragma unroll
    for (int q = 0; q < R; ++q) {
        // strip q's own k: strips above take every k, strip q the k below its row
        const int4 *tq = reinterpret_cast<const int4 *>(cur + koff + b0 + S * q);
#pragma unroll 2
        for (int c = 0; c < 32; c += 2) {
            const int4 p = tq[c >> 1];
#pragma unroll
            for (int j = q + 1; j < R; ++j)
                acc[j] = __vimin3_s32(acc[j], va(u[j], p.x, p.y), va(u[j], p.z, p.w));
            const int32_t c0 = c < lane ? va(u[q], p.x, p.y) : kInf;
            const int32_t c1 = c + 1 < lane ? va(u[q], p.z, p.w) : kInf;
            acc[q] = __vimin3_s32(acc[q], c0, c1);
        }
        if (S > 32 && q + 1 < R) {  // the other warps' strips between q and q + 1
            const int4 *pp = tq + 16;
            const int4 *pe = tq + S / 2;
#pragma unroll 2
            for (; pp < pe; ++pp) {
                const int4 p = *pp;
#pragma unroll
                for (int j = q + 1; j < R; ++j)
                    acc[j] = __vimin3_s32(acc[j], va(u[j], p.x, p.y), va(u[j], p.z, p.w));
            }
        }
    }
    // finalise
#pragma unroll
    for (int j = 0; j < R; ++j) {
        const int m = b0 + lane + S * j;
        if (m < n) continue;
        const int2 c = cur[m + koff];
        int32_t X, nx, ny;
        if (FORM == kS32) {
            X = FWD ? acc[j] - int32_t(dt) : acc[j];
            nx = c.x;
            ny = X;
        } else if (FORM == kEbwd) {
            X = acc[j];
            const int64_t y = int64_t(c.x) - dt;
            nx = y > -int64_t(kYCl) ? int32_t(y) : -kYCl;
            ny = X;
        } else {
            X = acc[j] - c.y;  // E = (E + G) - G
            nx = int32_t(uint32_t(acc[j]) - uint32_t(urow[m]) - uint32_t(dt));  // low word of b + P
            ny = c.y;
        }
        nxt[m + koff] = make_int2(nx, ny);
        if (n <= kKeep && DC_CHECK(tri_index(L, m, n) < kept_cells(L))) kept[tri_index(L, m, n)] = X;
        if (m == L) last[n] = X;
    }
}

template <int FORM, bool FWD, int S>
__device__ __forceinline__ void run_block(int R, int L, int n, int b0, int k_lo, bool far,
                                          int32_t gfar, int64_t dt, const int2 *cur, int2 *nxt,
                                          const int32_t *urow, int32_t *kept, int32_t *last,
                                          int koff, int lane)
{
#define DC_DEEP_BLOCK(RR)                                                                        \
    case RR:                                                                                     \
        block<RR, FORM, FWD, S>(L, n, b0, k_lo, far, gfar, dt, cur, nxt, urow, kept, last, koff, \
                                lane);                                                           \
        break;
    switch (R) {
        DC_DEEP_BLOCK(1) DC_DEEP_BLOCK(2) DC_DEEP_BLOCK(3) DC_DEEP_BLOCK(4)
        DC_DEEP_BLOCK(5) DC_DEEP_BLOCK(6) DC_DEEP_BLOCK(7) DC_DEEP_BLOCK(8)
        default: break;
    }
#undef DC_DEEP_BLOCK
}

template <int NW>
__device__ __forceinline__ void cta_sync()
{
    if (NW == 1)
        __syncwarp();
    else
        __syncthreads();
}

// The column loop of one form: columns 2..L, each warp its plan's blocks, one
// CTA barrier per column (the next column reads every warp's rows).
template <int FORM, bool FWD, int NW>
__device__ void fill(int L, int64_t dt, int2 *XY0, int2 *XY1, const int32_t *urow,
                     const int4 *plan, int nplan, int32_t *kept, int32_t *last, int koff, int tid)
{
    constexpr int S = 32 * NW;
    const int lane = tid & 31;
    for (int n = 2; n <= L; ++n) {
        const int2 *cur = (n - 1) & 1 ? XY1 : XY0;
        int2 *nxt = n & 1 ? XY1 : XY0;
        for (int e = 0; e < nplan; ++e) {
            const int4 b = plan[e];  // top, strips, kF
            const int top = b.x;
            if (top < n) break;
            const int b00 = top - 31 - S * (b.y - 1);
            const int jmin = n - b00 - 31 > 0 ? (n - b00 - 31 + S - 1) / S : 0;
            const int b0 = b00 + S * jmin;
            int k_lo = n - 1;
            bool far = false;
            int32_t gfar = 0;
            if (FORM == kEfwd && b.z > n - 1) {
                far = true;
                gfar = cur[b.z - 1 + koff].y;  // G[kF - 1]
                k_lo = b.z;
            }
            run_block<FORM, FWD, S>(b.y - jmin, L, n, b0, k_lo, far, gfar, dt, cur, nxt, urow,
                                    kept, last, koff, lane);
        }
        // entries n-2 and n-1 of the new column's pairs are stale: neutral
        if (tid < 2 && n - 2 + tid >= 0) nxt[n - 2 + tid + koff].y = kInf;
        cta_sync<NW>();
    }
}

template <bool FWD, int NW>
__global__ void __launch_bounds__(32 * NW, NW == 1 ? 16 : 24 / NW) deep_kernel(DeepArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    constexpr int S = 32 * NW;
    const int L = a.L, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int W = words_for(L), koff = deep_koff(L), PM = deep_plan_max(L);
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem);
    volatile int32_t *ctl = reinterpret_cast<volatile int32_t *>(smem + 8);  // instance, flag
    int2 *XY0 = reinterpret_cast<int2 *>(smem + 16);
    int2 *XY1 = reinterpret_cast<int2 *>(smem + 16 + (deep_buffers(NW) - 1) * deep_pair_bytes(L));
    int32_t *urow = reinterpret_cast<int32_t *>(smem + deep_urow_off(L, NW));
    uint32_t *bitsw = reinterpret_cast<uint32_t *>(smem + deep_bits_off(L, NW));
    int4 *plans = reinterpret_cast<int4 *>(smem + deep_plan_off(L, NW));
    int4 *plan = plans + warp * (PM + 1);

    // The next launch of a split batch may start filling SMs as this one's CTAs
    // exit (programmatic dependent launch); it shares no data with this one.
    pdl_trigger();
    // Claim a free slot: at most one resident wave of CTAs lives at a time, over
    // this launch and the next, and there are at least that many slots. Each
    // bitmap word is tried from a free bit until one is won or none is left.
    if (tid == 0) {
        int got = -1;
        const int nw = (a.nslots + 31) / 32;
        for (int p = 0; p < nw && got < 0; ++p) {
            const int w = int((blockIdx.x / 32u + unsigned(p)) % unsigned(nw));
            const int nbits = min(32, a.nslots - 32 * w);
            const uint32_t full = nbits == 32 ? 0xffffffffu : ((1u << nbits) - 1u);
            uint32_t v = *reinterpret_cast<volatile uint32_t *>(a.busy + w);
            for (int tries = 0; tries < 32 && (v & full) != full; ++tries) {
                const int b = __ffs(~v & full) - 1;
                const uint32_t old = atomicOr(a.busy + w, 1u << b);
                if (!(old & (1u << b))) {
                    got = 32 * w + b;
                    break;
                }
                v = old | (1u << b);
            }
        }
        reinterpret_cast<volatile int32_t *>(smem + 8)[1] = got;
    }
    __syncthreads();
    const int slot_id = reinterpret_cast<volatile int32_t *>(smem + 8)[1];
    if (!DC_CHECK(slot_id < a.nslots)) return;
    if (slot_id < 0) {  // every slot held (not expected): leave the instances to the other CTAs
        pdl_wait();
        return;
    }
    unsigned char *slot = a.slots + size_t(slot_id) * a.slot_bytes;
    uint64_t *P64 = reinterpret_cast<uint64_t *>(slot);
    int32_t *last = reinterpret_cast<int32_t *>(slot + slot_last_off(L));
    int32_t *Gk = reinterpret_cast<int32_t *>(slot + slot_g_off(L));
    int32_t *kept = reinterpret_cast<int32_t *>(slot + slot_kept_off(L));
    uint64_t *raw = reinterpret_cast<uint64_t *>(XY0);  // one profile row at a time

    if (a.bulk && tid == 0) mbar_init(bar);
    __syncthreads();
    uint32_t phase = 0;
    const int chunk = (L + 31) / 32;
    const int r_lo = 1 + lane * chunk, r_hi = min(L, r_lo + chunk - 1);
    auto col = [&](int r) { return FWD ? r - 1 : L - r; };
    enum { kListed = -1, kAbort = -2 };

    for (;;) {
        if (tid == 0) ctl[0] = int32_t(atomicAdd(a.ticket, 1u));
        __syncthreads();
        const uint32_t jt = uint32_t(ctl[0]);
        if (int64_t(jt) >= a.count) break;
        const int64_t i = a.lo + int64_t(jt);
        const int64_t dti = a.dt[i];
        uint64_t sx = 0, shift = 0;  // warp 0: raw transfer total, capped-off transfer

        // ---- warp 0: rows, checks, form, prefix sums, column 1
        if (warp == 0) {
            int flag = 0;
            // one profile row into the staging buffer: 0 landed, 1 lost (the
            // instance is marked failed), 2 lost and perhaps still in flight
            auto stage = [&](const int64_t *row) -> int {
                if (!a.bulk) {
                    for (int c = lane; c < L; c += 32) raw[c] = uint64_t(__ldg(row + c));
                    __syncwarp();
                    return 0;
                }
                // the buffer's earlier reads and writes before the copy's writes
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) {
                    mbar_expect(bar, uint32_t(8) * uint32_t(L));
                    bulk_g2s(raw, row, uint32_t(8) * uint32_t(L), bar);
                }
                const bool ok = mbar_wait(bar, phase, 1 << 22);
                phase ^= 1u;
                if (__all_sync(0xffffffffu, ok)) return 0;
                // the copy did not land in time: wait once more before the buffer
                // is given up
                const bool late = mbar_wait(bar, phase ^ 1u, 1 << 22);
                return __all_sync(0xffffffffu, late) ? 1 : 2;
            };
            // compute row: checks, total, prefix (wrapping; used only when the
            // total is below 2^31) into urow
            int lost = stage(a.comp + i * L);
            bool neg = dti < 0, big = (dti >> 52) != 0;
            uint64_t sc = 0;
            if (!lost) {
                for (int r = r_lo; r <= r_hi; ++r) {
                    const int64_t cv = int64_t(raw[col(r)]);
                    neg |= cv < 0;
                    big |= (cv >> 52) != 0;
                    sc += uint64_t(cv);
                }
                uint64_t oc = warp_excl_scan_u64(sc, lane);
                for (int r = r_lo; r <= r_hi; ++r) {
                    oc += raw[col(r)];
                    urow[r] = int32_t(oc);
                }
                sc = warp_sum_u64(sc);
                __syncwarp();  // every lane has read the row before the next one lands
                lost = stage(a.xfer + i * L);
            }
            uint64_t cx_lane = 0;
            if (!lost) {
                for (int r = r_lo; r <= r_hi; ++r) {
                    const int64_t xv = int64_t(raw[col(r)]);
                    neg |= xv < 0;
                    big |= (xv >> 52) != 0;
                    sx += uint64_t(xv);
                    cx_lane += uint64_t(xv) < sc ? uint64_t(xv) : sc;
                }
                neg = __any_sync(0xffffffffu, neg);
                big = __any_sync(0xffffffffu, big);
                sx = warp_sum_u64(sx);
            }
            if (lost) {
                if (lane == 0) {
                    a.makespan[i] = -int64_t(DC_ERR_INTERNAL);
                    if (a.nseg) a.nseg[i] = 0;
                    if (a.status) a.status[i] = DC_ERR_INTERNAL;
                }
                for (int w = lane; w < W; w += 32) a.bits[i * W + w] = 0u;
                flag = lost == 1 ? int(kListed) : int(kAbort);
            } else {
                int st = DC_OK;
                if (neg)
                    st = DC_ERR_NEGATIVE;
                else if (big || exceeds_range(L, dti, sc, sx))
                    st = DC_ERR_RANGE;
                if (st != DC_OK) {
                    if (lane == 0) {
                        a.makespan[i] = -int64_t(st);
                        if (a.nseg) a.nseg[i] = 0;
                        if (a.status) a.status[i] = st;
                    }
                    for (int w = lane; w < W; w += 32) a.bits[i * W + w] = 0u;
                    flag = kListed;  // done: nothing for the other warps
                } else {
                    // transfers capped at the total compute; the arithmetic form
                    const uint64_t cx = warp_sum_u64(cx_lane);
                    shift = sx - cx;
                    const uint64_t bound = sc + cx + uint64_t(L) * uint64_t(dti);
                    if (bound <= kShiftedLimit)
                        flag = kS32;
                    else if (!FWD && sc < uint64_t(kYCl))
                        flag = kEbwd;
                    else if (FWD && sc < (uint64_t(1) << 29))
                        flag = kEfwd;
                    else
                        flag = kListed;
                    if (flag == kListed) {  // 32/64-bit literal template: the CTA-per-instance kernel
                        if (lane == 0) {
                            const uint32_t at = atomicAdd(a.list_count, 1u);
                            if (DC_CHECK(int64_t(at) < a.lo + a.count)) a.list[at] = uint32_t(i);
                        }
                    } else {
                        // prefix of the capped transfers (64-bit) into the slot
                        uint64_t ox = warp_excl_scan_u64(cx_lane, lane);
                        for (int r = r_lo; r <= r_hi; ++r) {
                            const uint64_t xv = raw[col(r)];
                            ox += xv < sc ? xv : sc;
                            P64[r] = ox;
                        }
                        if (lane == 0) {
                            urow[0] = 0;
                            P64[0] = 0;
                        }
                        for (int w = lane; w < W + 1; w += 32) bitsw[w] = 0u;
                        __syncwarp();
                        // column 1 and the row terms
                        const int32_t fcL = urow[L];
                        __syncwarp();  // every lane has fcL before urow[L] is overwritten
                        for (int m = lane; m <= L; m += 32) {
                            const int32_t CF = urow[m];
                            const uint64_t P = P64[m];
                            int32_t u, x, y, X;
                            if (flag == kS32) {
                                if (FWD) {
                                    u = int32_t(dti) + int32_t(P);
                                    x = fcL - CF;
                                    y = fcL + int32_t(P);
                                } else {
                                    u = CF;
                                    x = -int32_t(P);
                                    y = CF;
                                }
                                X = y;
                            } else if (flag == kEbwd) {
                                u = CF;
                                x = -yclamp64(dti + int64_t(P));
                                y = CF;
                                X = CF;
                            } else {
                                u = int32_t(uint32_t(0) - uint32_t(dti) - uint32_t(P));
                                x = int32_t(uint32_t(fcL) + uint32_t(P));
                                y = fcL - CF;
                                Gk[m] = y;
                                X = CF;
                            }
                            urow[m] = u;
                            XY1[m + koff] = make_int2(x, m == 0 ? kInf : y);
                            if (m >= 1) kept[tri_index(L, m, 1)] = X;
                            if (m == L) last[1] = X;
                        }
                        for (int e = lane; e < koff; e += 32) {
                            XY0[e] = make_int2(0, kInf);
                            XY1[e] = make_int2(0, kInf);
                        }
                    }
                }
            }
            if (lane == 0) ctl[1] = flag;
        }
        __syncthreads();
        const int form = ctl[1];
        if (form == kAbort) {  // the staging buffers may still be written: keep the slot
            pdl_wait();
            return;
        }
        if (form < 0) {
            __syncthreads();  // ctl is read by every thread before the next ticket
            continue;
        }

        // ---- each warp's block plan: its strips t = warp, warp + NW, ... from
        // the top (strip t holds rows L - 32 t - 31 .. L - 32 t), up to 8 per block
        if (lane == 0) {
            const int T = (L + 31) / 32;
            int np = 0, t = warp;
            bool ok = true;
            while (t < T) {
                const int avail = (T - 1 - t) / NW + 1;
                int R = avail < kMaxStrips ? avail : kMaxStrips;
                const int top = L - 32 * t;
                int kF = 0;
                if (form == kEfwd) {
                    for (; R >= 1; --R) {
                        const int botc = max(top - 31 - S * (R - 1), 1);
                        const int64_t span = int64_t(P64[top] - P64[botc]);
                        if (span <= kSpanLimit && dti + span <= kTwo31) break;
                    }
                    if (R < 1) {
                        ok = false;
                        break;
                    }
                    // kF: first k with P[k] >= P[top] + dt - 2^31 (at most the block's bottom)
                    const int64_t thr = int64_t(P64[top]) + dti - kTwo31;
                    int lo = 0, hi = max(top - 31 - S * (R - 1), 1);
                    while (lo < hi) {
                        const int mid = (lo + hi) >> 1;
                        if (int64_t(P64[mid]) < thr)
                            lo = mid + 1;
                        else
                            hi = mid;
                    }
                    kF = lo;
                }
                plan[np++] = make_int4(top, R, kF, 0);
                t += R * NW;
            }
            plan[PM] = make_int4(ok ? np : -1, 0, 0, 0);
        }
        __syncthreads();
        bool planned = true;
        for (int w = 0; w < NW; ++w) planned &= plans[w * (PM + 1) + PM].x >= 0;
        if (!planned) {  // blocks narrower than one strip: the CTA-per-instance kernel
            if (tid == 0) {
                            const uint32_t at = atomicAdd(a.list_count, 1u);
                            if (DC_CHECK(int64_t(at) < a.lo + a.count)) a.list[at] = uint32_t(i);
                        }
            __syncthreads();
            continue;
        }
        const int nplan = plan[PM].x;

        // ---- columns 2..L
        if (form == kS32)
            fill<kS32, FWD, NW>(L, dti, XY0, XY1, urow, plan, nplan, kept, last, koff, tid);
        else if (form == kEbwd)
            fill<kEbwd, FWD, NW>(L, dti, XY0, XY1, urow, plan, nplan, kept, last, koff, tid);
        else
            fill<kEfwd, FWD, NW>(L, dti, XY0, XY1, urow, plan, nplan, kept, last, koff, tid);
        __syncthreads();

        // ---- warp 0: lowest n minimising the makespan, then the traceback
        if (warp == 0) {
            int64_t bv = INT64_MAX;
            int bn = 0x7fffffff;
            const int64_t toB = (form == kS32 && FWD) ? int64_t(dti) - int64_t(urow[L]) : 0;
            for (int n = 1 + lane; n <= L; n += 32) {
                const int64_t v = int64_t(last[n]) + toB + int64_t(n) * dti;
                if (v < bv) {
                    bv = v;
                    bn = n;
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const int64_t ov = __shfl_xor_sync(0xffffffffu, bv, o);
                const int on = __shfl_xor_sync(0xffffffffu, bn, o);
                if (ov < bv || (ov == bv && on < bn)) {
                    bv = ov;
                    bn = on;
                }
            }
            const int s = bn;
            if (s - 1 > kKeep) {  // the traceback needs columns beyond the kept ones
                if (lane == 0) {
                            const uint32_t at = atomicAdd(a.list_count, 1u);
                            if (DC_CHECK(int64_t(at) < a.lo + a.count)) a.list[at] = uint32_t(i);
                        }
            } else {
                // Path[m][n] = the lowest k whose candidate equals the cell
                int err = 0, m = L, n = s;
                const int2 *V = XY1;  // S32: x = V[k] in every entry k >= 1 of the column-1 buffer
                while (n > 1) {
                    const int32_t Xmn = (m == L && n == s) ? last[s] : kept[tri_index(L, m, n)];
                    const int64_t pbase = tri_col(L, n - 1) - (n - 1);  // + k gives (k, n-1)
                    int found = -1;
                    for (int k0 = n - 1; k0 < m; k0 += 32) {
                        const int k = k0 + lane;
                        bool match = false;
                        if (k < m) {
                            const int32_t Xk = DC_CHECK(pbase + k < kept_cells(L)) ? kept[pbase + k] : 0;
                            if (form == kS32) {
                                const int32_t u = FWD ? urow[m] : urow[m] - int32_t(int64_t(n - 1) * dti);
                                const int32_t target = FWD ? Xmn + int32_t(dti) : Xmn;
                                match = va(u, V[k + koff].x, Xk) == target;
                            } else if (form == kEbwd) {
                                const int32_t y = yclamp64(int64_t(n - 1) * dti + int64_t(P64[k]));
                                match = max(Xk, urow[m] - y) == Xmn;
                            } else {
                                const int64_t Q = dti + int64_t(P64[m]);
                                const int64_t g = Gk[k];
                                const int64_t x = int64_t(Xk) + g + int64_t(P64[k]) - Q;
                                match = (x > g ? x : g) == int64_t(Xmn) + Gk[m];
                            }
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
                __syncwarp();
                if (lane == 0) {
                    const uint64_t mk = form == kS32 ? uint64_t(bv) + sx : uint64_t(bv) + P64[L] + shift;
                    a.makespan[i] = err ? -int64_t(DC_ERR_INTERNAL) : int64_t(mk);
                    if (a.nseg) a.nseg[i] = err ? 0 : s;
                    if (a.status) a.status[i] = err ? DC_ERR_INTERNAL : DC_OK;
                }
                for (int w = lane; w < W; w += 32) a.bits[i * W + w] = err ? 0u : bitsw[w];
            }
        }
        __syncthreads();
    }
    // release the slot, then finish no earlier than the previous launch of the
    // batch, so that a kernel waiting for the last launch waits for them all
    if (tid == 0) {
        __threadfence();
        atomicAnd(a.busy + slot_id / 32, ~(1u << (slot_id % 32)));
    }
    pdl_wait();
}

}  // namespace

int sm_count();  // SMs of the current device (dp_small.cu)

size_t deep_slot_bytes(int L) { return slot_bytes(L); }

// Resident one-warp CTAs per SM for depth L: a bound from shared memory alone
// (the workspace is sized from it on the host, without a device query).
int64_t deep_slots_bound(int L)
{
    const size_t per = deep_smem(L, 1) + 1024;  // the runtime reserves 1 KB per CTA
    int64_t n = int64_t((228 * 1024) / per);
    if (n > 32) n = 32;
    if (n < 1) n = 1;
    return 152 * n;
}

namespace {

// Resident CTAs per SM of deep_kernel<FWD, NW> at depth L (raising the
// kernel's shared-memory limit once per device first).
template <bool FWD, int NW>
cudaError_t deep_occupancy(int L, int &nb)
{
    static DeviceCache attr;
    int done = 0;
    cudaError_t e = attr.get(done, [](int &v) {
        v = 1;
        return cudaFuncSetAttribute(deep_kernel<FWD, NW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    int(deep_smem(DC_L_MAX, NW)));
    });
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, deep_kernel<FWD, NW>, 32 * NW,
                                                      deep_smem(L, NW));
    if (nb < 1) nb = 1;
    return e;
}

template <bool FWD, int NW>
cudaError_t launch_deep_nw(const DeepArgs &a, int64_t grid, bool pdl, cudaStream_t stream)
{
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(unsigned(grid));
    lc.blockDim = dim3(32 * NW);
    lc.dynamicSmemBytes = deep_smem(a.L, NW);
    lc.stream = stream;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = at;
    lc.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&lc, deep_kernel<FWD, NW>, a);
}

// Warps per instance. Persistent CTAs take instances in rounds of at most one
// resident wave. An SM's throughput grows about linearly with its active warps
// up to about 10 (measured: 10 one-warp instances per SM reach 0.78 of the
// int-ALU roof, 4 about 0.23), and NW warps sharing an instance lose to their
// per-column barrier and shorter blocks (about 0.7 / 0.6 / 0.55 of the one-warp
// rate for 2 / 4 / 8 warps). Each choice's time is estimated round by round as
// (instances per SM) / (min(active warps per SM, 10) x that efficiency), the
// last round holding the remainder, and the smallest wins: one warp per
// instance once the batch fills the GPU, more for a few hundred instances.
template <bool FWD>
cudaError_t launch_deep_dir(const DeepArgs &a, int64_t nslots, bool pdl, cudaStream_t stream)
{
    const int sms = sm_count();
    const int nws[4] = {1, 2, 4, 8};
    const double eta[4] = {1.0, 0.7, 0.6, 0.55};
    int nb[4];
    cudaError_t e;
    if ((e = deep_occupancy<FWD, 1>(a.L, nb[0])) != cudaSuccess) return e;
    if ((e = deep_occupancy<FWD, 2>(a.L, nb[1])) != cudaSuccess) return e;
    if ((e = deep_occupancy<FWD, 4>(a.L, nb[2])) != cudaSuccess) return e;
    if ((e = deep_occupancy<FWD, 8>(a.L, nb[3])) != cudaSuccess) return e;
    int pick = 0;
    int64_t grid_pick = 1;
    double best = 0.0;
    for (int q = 0; q < 4; ++q) {
        int64_t G = int64_t(nb[q]) * sms;
        if (G > nslots) G = nslots;
        if (G > a.count) G = a.count;
        double t = 0.0;
        for (int64_t left = a.count; left > 0; left -= G) {
            const double per_sm = double(left < G ? left : G) / sms;
            const double active = per_sm * nws[q];
            t += per_sm / ((active < 10.0 ? active : 10.0) * eta[q]);
        }
        if (q == 0 || t < best) {
            best = t;
            pick = q;
            grid_pick = G;
        }
    }
    if (const int f = forced_warps()) {  // the test hook's warps per instance
        pick = f == 1 ? 0 : f == 2 ? 1 : f == 4 ? 2 : 3;
        grid_pick = int64_t(nb[pick]) * sms;
        if (grid_pick > nslots) grid_pick = nslots;
        if (grid_pick > a.count) grid_pick = a.count;
    }
    switch (nws[pick]) {
        case 1: return launch_deep_nw<FWD, 1>(a, grid_pick, pdl, stream);
        case 2: return launch_deep_nw<FWD, 2>(a, grid_pick, pdl, stream);
        case 4: return launch_deep_nw<FWD, 4>(a, grid_pick, pdl, stream);
        default: return launch_deep_nw<FWD, 8>(a, grid_pick, pdl, stream);
    }
}

}  // namespace

// Instances per launch: about 90 ms of work at 0.67 of the int-ALU roof
// (transitions C(L) per instance), and at least two resident waves of one-warp
// CTAs, so that a long batch runs as launches of at most ~100 ms on a shared GPU.
int64_t deep_per_launch(int64_t batch, int L)
{
    const double c = double(L) + double(L + 1) * double(L) * double(L - 1) / 6.0;
    const double rate = 152.0 * 64.0 * 2.07e9 / 1.5 * 0.67;
    int64_t per = int64_t(0.09 * rate / c);
    const int64_t wave2 = 2 * deep_slots_bound(L);
    if (per < wave2) per = wave2;
    if (per >= batch) return batch;
    const int64_t n = (batch + per - 1) / per;  // equal shares
    return (batch + n - 1) / n;
}

int64_t deep_launches(int64_t batch, int L)
{
    if (batch <= 0) return 0;
    const int64_t per = deep_per_launch(batch, L);
    return (batch + per - 1) / per;
}

cudaError_t launch_deep(bool forward, int64_t batch, int L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                        uint32_t *bits, int32_t *nseg, int32_t *status, uint32_t *tickets,
                        uint32_t *busy, uint32_t *list_count, uint32_t *list, void *slots,
                        int64_t nslots, cudaStream_t stream)
{
    if (batch <= 0) return cudaSuccess;
    const bool bulk = (L % 2 == 0) &&
                      ((reinterpret_cast<uintptr_t>(comp) | reinterpret_cast<uintptr_t>(xfer)) & 15u) == 0;
    const int64_t per = deep_per_launch(batch, L);
    // every launch's ticket and every slot's flag start at zero
    cudaError_t e = cudaMemsetAsync(busy, 0, size_t((nslots + 31) / 32) * 4, stream);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(tickets, 0, size_t(deep_launches(batch, L)) * 4, stream);
    if (e != cudaSuccess) return e;
    int64_t k = 0;
    for (int64_t lo = 0; lo < batch; lo += per, ++k) {
        const int64_t count = batch - lo < per ? batch - lo : per;
        DeepArgs a{lo, count, L, comp, xfer, dt, makespan, bits, nseg, status, tickets + k,
                   list_count, list, busy, static_cast<unsigned char *>(slots), slot_bytes(L),
                   int(nslots), bulk ? 1 : 0};
        // the first launch waits for the memsets in stream order; later ones may
        // overlap the tail of the one before
        e = forward ? launch_deep_dir<true>(a, nslots, k > 0, stream)
                    : launch_deep_dir<false>(a, nslots, k > 0, stream);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace dc

DC_CHECKED_EXPORT(dp_deep)
