// The cost measurement f_m (Sec. III-B) on the GPU: replays any decision of one
// direction under the partial orders Eq. 1-7 and returns the makespan.
//
// One thread per instance, segment by segment in processing order:
//   forward : segment j ends at layer b_j; its pull completes at
//             j*dt + sum_{l<=b_j} pt_l (pulls back to back, Eq. 4); its layers
//             compute after that and after the previous segment (Eq. 1, 5):
//             end_j = max(end_{j-1}, arrive_j) + sum of the segment's fc.
//   backward: layers compute from L down without waiting (Eq. 6); the push of
//             segment j starts after its last layer's compute and the previous
//             push (Eq. 2, 7): link_j = max(link_{j-1}, done_j) + dt + sum gt.
// Inputs are checked like the solver's (negative -> -3, bound >= 2^52 -> -4).
//
// For L <= 64 a warp first copies its 32 instances' rows into shared memory with
// coalesced asynchronous copies (16-byte copies of cost pairs for even L; a row
// stride at which every lane reads its own row without bank conflicts), then
// replays its lane's row. Warps are persistent (one resident wave) and prefetch
// their next tile into L2 while the current one is copied. For L <= 16 the
// replay is unrolled at compile time and inputs are screened on their high
// words. Longer rows are read by each thread directly.
#include "common.cuh"

namespace dc {

int sm_count();  // SMs of the current device (dp_small.cu)

namespace {

constexpr int kStagedLMax = 64;
constexpr int kEvalWarps = 4;

struct Replay {
    uint64_t clock_a = 0;  // forward: compute end; backward: link end
    uint64_t run = 0;      // forward: pull end; backward: compute end
    uint64_t seg = 0;      // forward: segment compute; backward: segment transfer
    uint64_t sc = 0, sx = 0;
    bool neg = false, big = false;

    // unsigned arithmetic: garbage from rejected inputs wraps instead of overflowing
    template <bool FWD>
    __device__ __forceinline__ void step(int64_t cv, int64_t xv, uint64_t d, bool cut)
    {
        neg |= (cv < 0) | (xv < 0);
        big |= ((cv | xv) >> 52) != 0;
        sc += uint64_t(cv);
        sx += uint64_t(xv);
        if (FWD) {
            run += uint64_t(xv);
            seg += uint64_t(cv);
            if (cut) {
                run += d;  // one more transmission set-up
                clock_a = (clock_a > run ? clock_a : run) + seg;
                seg = 0;
            }
        } else {
            run += uint64_t(cv);
            seg += uint64_t(xv);
            if (cut) {
                clock_a = (clock_a > run ? clock_a : run) + d + seg;
                seg = 0;
            }
        }
    }

    __device__ __forceinline__ int64_t result(int L, int64_t d) const
    {
        if (neg || d < 0) return -int64_t(DC_ERR_NEGATIVE);
        if (big || (d >> 52) != 0 || exceeds_range(L, d, sc, sx)) return -int64_t(DC_ERR_RANGE);
        return int64_t(clock_a);
    }
};

template <bool FWD>
__global__ void __launch_bounds__(256)
    eval_kernel(int64_t batch, int L, const int64_t *__restrict__ comp,
                const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
                const uint32_t *__restrict__ bits, int64_t *__restrict__ makespan)
{
    const int W = words_for(L);
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < batch;
         i += int64_t(gridDim.x) * blockDim.x) {
        const int64_t *crow = comp + i * L;
        const int64_t *xrow = xfer + i * L;
        const uint32_t *brow = bits + i * W;
        const int64_t d = __ldg(dt + i);
        Replay rp;
        uint32_t word = 0;
        for (int r = 1; r <= L; ++r) {
            const int col = FWD ? r - 1 : L - r;
            if (((r - 1) & 31) == 0 && r <= L - 1) word = __ldg(brow + ((r - 1) >> 5));
            const bool cut = (r == L) || ((word >> ((r - 1) & 31)) & 1u);
            rp.step<FWD>(__ldg(crow + col), __ldg(xrow + col), uint64_t(d), cut);
        }
        makespan[i] = rp.result(L, d);
    }
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

// Staging row stride (int64 units). Odd L: L (odd), so that 16 lanes reading
// 8-byte words of their own rows hit distinct bank pairs. Even L: rows are copied
// and read as 16-byte pairs; an even stride that is 2 mod 4 keeps the rows
// 16-byte aligned and lets 8 lanes reading 16 bytes hit distinct bank groups.
__host__ __device__ inline int eval_stride(int L) { return (L % 2 == 1) ? L : (L % 4 == 2 ? L : L + 2); }

template <bool FWD>
__global__ void __launch_bounds__(32 * kEvalWarps)
    eval_staged_kernel(int64_t batch, int L, const int64_t *__restrict__ comp,
                       const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
                       const uint32_t *__restrict__ bits, int64_t *__restrict__ makespan,
                       bool pairs)
{
    extern __shared__ __align__(16) int64_t stage[];
    const int stride = eval_stride(L);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int64_t *stC = stage + warp * 2 * 32 * stride;
    int64_t *stX = stC + 32 * stride;
    const int64_t tiles = (batch + 31) / 32;
    const int64_t step = int64_t(gridDim.x) * kEvalWarps;
    const bool even = (L % 2) == 0;
    const int H = L / 2;
    for (int64_t tile = int64_t(blockIdx.x) * kEvalWarps + warp; tile < tiles; tile += step) {
        const int64_t base = tile * 32;
        const int rows = int(batch - base < 32 ? batch - base : 32);
        const int64_t *gC = comp + base * L;
        const int64_t *gX = xfer + base * L;
        __syncwarp();
        // all copies in flight at once (no register round trip), then one wait
        if (even && pairs) {
            const int np = rows * H;
            for (int p = lane; p < np; p += 32) {
                const int r = p / H, cidx = 2 * (p - r * H);
                cp_async16(stC + r * stride + cidx, gC + 2 * p);
                cp_async16(stX + r * stride + cidx, gX + 2 * p);
            }
        } else {
            const int nel = rows * L;
            for (int e = lane; e < nel; e += 32) {
                const int r = e / L, cidx = e - r * L;
                cp_async8(stC + r * stride + cidx, gC + e);
                cp_async8(stX + r * stride + cidx, gX + e);
            }
        }
        asm volatile("cp.async.commit_group;\n" ::: "memory");
        if (tile + step < tiles) {  // the warp's next tile into L2 (128-byte lines)
            const int64_t nb = (tile + step) * 32;
            const int64_t nel = (batch - nb < 32 ? batch - nb : 32) * L;
            for (int64_t e = int64_t(lane) * 16; e < nel; e += 32 * 16) {
                asm volatile("prefetch.global.L2 [%0];" ::"l"(comp + nb * L + e));
                asm volatile("prefetch.global.L2 [%0];" ::"l"(xfer + nb * L + e));
            }
        }
        const bool active = lane < rows;
        const int64_t i = base + lane;
        const int64_t d = active ? __ldg(dt + i) : 0;
        const int W = words_for(L);  // 1 or 2 for L <= 64
        const uint32_t w0 = (active && W > 0) ? __ldg(bits + i * W) : 0u;
        const uint32_t w1 = (active && W > 1) ? __ldg(bits + i * W + 1) : 0u;
        // break after processing position b + 1 (0-based b)
        auto brk = [&](int b) { return ((b < 32 ? w0 >> b : w1 >> (b - 32)) & 1u) != 0u; };
        asm volatile("cp.async.wait_group 0;\n" ::: "memory");
        __syncwarp();
        if (!active) continue;
        Replay rp;
        const int64_t *rc = stC + lane * stride, *rx = stX + lane * stride;
        if (even) {  // 16-byte reads of cost pairs, in processing order
            for (int q = 0; q < L; q += 2) {
                const int col = FWD ? q : L - 2 - q;
                const longlong2 c = *reinterpret_cast<const longlong2 *>(rc + col);
                const longlong2 x = *reinterpret_cast<const longlong2 *>(rx + col);
                const int r = q + 1;
                const bool cut0 = brk(r - 1);
                const bool cut1 = (r + 1 == L) || brk(r);
                if (FWD) {
                    rp.step<FWD>(c.x, x.x, uint64_t(d), cut0);
                    rp.step<FWD>(c.y, x.y, uint64_t(d), cut1);
                } else {
                    rp.step<FWD>(c.y, x.y, uint64_t(d), cut0);
                    rp.step<FWD>(c.x, x.x, uint64_t(d), cut1);
                }
            }
        } else {
            for (int r = 1; r <= L; ++r) {
                const int col = FWD ? r - 1 : L - r;
                const bool cut = (r == L) || brk(r - 1);
                rp.step<FWD>(rc[col], rx[col], uint64_t(d), cut);
            }
        }
        makespan[i] = rp.result(L, d);
    }
}

// Replay of one staged row with L a compile-time constant (unrolled). Inputs are
// screened on their high words: a value that is negative or at least 2^52 sets a
// bit at or above bit 20 of the OR of all high words (dt included).
template <int L, bool FWD>
__device__ __forceinline__ int64_t replay_row(const int64_t *rc, const int64_t *rx, int64_t d,
                                              uint32_t word)
{
    uint64_t clock = 0, run = 0, seg = 0, sc = 0, sx = 0;
    uint32_t hor = uint32_t(uint64_t(d) >> 32);
    const uint64_t ud = uint64_t(d);
    auto step = [&](int r, uint64_t cv, uint64_t xv) {  // r: 1-based processing position
        hor |= uint32_t(cv >> 32) | uint32_t(xv >> 32);
        sc += cv;
        sx += xv;
        const bool cut = (r == L) || ((word >> (r - 1)) & 1u);
        if (FWD) {
            run += xv;
            seg += cv;
            if (cut) {
                run += ud;
                clock = (clock > run ? clock : run) + seg;
                seg = 0;
            }
        } else {
            run += cv;
            seg += xv;
            if (cut) {
                clock = (clock > run ? clock : run) + ud + seg;
                seg = 0;
            }
        }
    };
    if constexpr (L % 2 == 0) {
#pragma unroll
        for (int q = 0; q < L; q += 2) {
            const int col = FWD ? q : L - 2 - q;
            const ulonglong2 c = *reinterpret_cast<const ulonglong2 *>(rc + col);
            const ulonglong2 x = *reinterpret_cast<const ulonglong2 *>(rx + col);
            if (FWD) {
                step(q + 1, c.x, x.x);
                step(q + 2, c.y, x.y);
            } else {
                step(q + 1, c.y, x.y);
                step(q + 2, c.x, x.x);
            }
        }
    } else {
#pragma unroll
        for (int r = 1; r <= L; ++r) {
            const int col = FWD ? r - 1 : L - r;
            step(r, uint64_t(rc[col]), uint64_t(rx[col]));
        }
    }
    if ((hor >> 31) != 0u) return -int64_t(DC_ERR_NEGATIVE);
    if ((hor >> 20) != 0u || exceeds_range(L, d, sc, sx)) return -int64_t(DC_ERR_RANGE);
    return int64_t(clock);
}

template <int L, bool FWD>
__global__ void __launch_bounds__(32 * kEvalWarps)
    eval_small_kernel(int64_t batch, const int64_t *__restrict__ comp,
                      const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
                      const uint32_t *__restrict__ bits, int64_t *__restrict__ makespan,
                      bool pairs)
{
    extern __shared__ __align__(16) int64_t stage[];
    constexpr int kStride = (L % 2 == 1) ? L : (L % 4 == 2 ? L : L + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int64_t *stC = stage + warp * 2 * 32 * kStride;
    int64_t *stX = stC + 32 * kStride;
    const int64_t tiles = (batch + 31) / 32;
    const int64_t step = int64_t(gridDim.x) * kEvalWarps;
    for (int64_t tile = int64_t(blockIdx.x) * kEvalWarps + warp; tile < tiles; tile += step) {
        const int64_t base = tile * 32;
        const int rows = int(batch - base < 32 ? batch - base : 32);
        const int64_t *gC = comp + base * L;
        const int64_t *gX = xfer + base * L;
        __syncwarp();
        if (L % 2 == 0 && pairs) {
            constexpr int H = L / 2 > 0 ? L / 2 : 1;
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
        asm volatile("cp.async.commit_group;\n" ::: "memory");
        if (tile + step < tiles) {  // the warp's next tile into L2: one 128-byte line per lane and array
            const int64_t nb = (tile + step) * 32;
            if (int64_t(lane) * 16 < (batch - nb < 32 ? batch - nb : 32) * L) {
                asm volatile("prefetch.global.L2 [%0];" ::"l"(comp + nb * L + lane * 16));
                asm volatile("prefetch.global.L2 [%0];" ::"l"(xfer + nb * L + lane * 16));
            }
        }
        const bool active = lane < rows;
        const int64_t i = base + lane;
        const int64_t d = active ? __ldg(dt + i) : 0;
        const uint32_t word = (active && L > 1) ? __ldg(bits + i) : 0u;  // W = 1 for 2 <= L <= 32
        asm volatile("cp.async.wait_group 0;\n" ::: "memory");
        __syncwarp();
        if (active) makespan[i] = replay_row<L, FWD>(stC + lane * kStride, stX + lane * kStride, d, word);
    }
}

template <int L, bool FWD>
cudaError_t launch_small_eval(int64_t batch, const int64_t *comp, const int64_t *xfer,
                              const int64_t *dt, const uint32_t *bits, int64_t *makespan,
                              bool pairs, cudaStream_t stream)
{
    constexpr int kStride = (L % 2 == 1) ? L : (L % 4 == 2 ? L : L + 2);
    constexpr int smem = kEvalWarps * 2 * 32 * kStride * 8;
    static DeviceCache resident;  // CTAs of the replay kernel per SM
    int per_sm = 0;
    const cudaError_t le = resident.get(per_sm, [](int &n) {
        cudaError_t e = cudaFuncSetAttribute(eval_small_kernel<L, FWD>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, eval_small_kernel<L, FWD>,
                                                             32 * kEvalWarps, smem);
    });
    if (le != cudaSuccess) return le;
    int64_t blocks = ((batch + 31) / 32 + kEvalWarps - 1) / kEvalWarps;
    if (blocks > int64_t(sm_count()) * per_sm) blocks = int64_t(sm_count()) * per_sm;
    eval_small_kernel<L, FWD><<<unsigned(blocks), 32 * kEvalWarps, smem, stream>>>(
        batch, comp, xfer, dt, bits, makespan, pairs);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_eval(bool forward, int64_t batch, int L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                        int64_t *makespan, cudaStream_t stream)
{
    if (L <= 16) {
        const bool pairs = ((reinterpret_cast<uintptr_t>(comp) | reinterpret_cast<uintptr_t>(xfer)) & 15u) == 0;
#define DC_EVAL_CASE(LL)                                                                        \
    case LL:                                                                                    \
        return forward ? launch_small_eval<LL, true>(batch, comp, xfer, dt, bits, makespan,     \
                                                     pairs, stream)                             \
                       : launch_small_eval<LL, false>(batch, comp, xfer, dt, bits, makespan,    \
                                                      pairs, stream);
        switch (L) {
            DC_EVAL_CASE(1) DC_EVAL_CASE(2) DC_EVAL_CASE(3) DC_EVAL_CASE(4)
            DC_EVAL_CASE(5) DC_EVAL_CASE(6) DC_EVAL_CASE(7) DC_EVAL_CASE(8)
            DC_EVAL_CASE(9) DC_EVAL_CASE(10) DC_EVAL_CASE(11) DC_EVAL_CASE(12)
            DC_EVAL_CASE(13) DC_EVAL_CASE(14) DC_EVAL_CASE(15) DC_EVAL_CASE(16)
            default: break;
        }
#undef DC_EVAL_CASE
    }
    if (L <= kStagedLMax) {
        const int stride = eval_stride(L);
        const size_t smem = size_t(kEvalWarps) * 2 * 32 * stride * 8;
        const bool pairs = ((reinterpret_cast<uintptr_t>(comp) | reinterpret_cast<uintptr_t>(xfer)) & 15u) == 0;
        // up to 69.6 KB at L = 32: above the 48 KB default
        static DeviceCache attr;
        int done = 0;
        cudaError_t ae = attr.get(done, [](int &v) {
            const int most = kEvalWarps * 2 * 32 * (kStagedLMax + 2) * 8;
            v = 1;
            cudaError_t e = cudaFuncSetAttribute(
                eval_staged_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, most);
            if (e != cudaSuccess) return e;
            return cudaFuncSetAttribute(eval_staged_kernel<false>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, most);
        });
        if (ae != cudaSuccess) return ae;
        // persistent warps: one resident wave, each warp walking tiles (and
        // prefetching its next one); resident CTAs per SM by L and direction
        static DeviceCache resident[kStagedLMax + 1][2];
        int per_sm = 0;
        ae = resident[L][forward ? 1 : 0].get(per_sm, [&](int &n) {
            return forward ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                                 &n, eval_staged_kernel<true>, 32 * kEvalWarps, smem)
                           : cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                                 &n, eval_staged_kernel<false>, 32 * kEvalWarps, smem);
        });
        if (ae != cudaSuccess) return ae;
        int64_t blocks = ((batch + 31) / 32 + kEvalWarps - 1) / kEvalWarps;
        if (blocks > int64_t(sm_count()) * per_sm) blocks = int64_t(sm_count()) * per_sm;
        if (forward)
            eval_staged_kernel<true><<<unsigned(blocks), 32 * kEvalWarps, smem, stream>>>(
                batch, L, comp, xfer, dt, bits, makespan, pairs);
        else
            eval_staged_kernel<false><<<unsigned(blocks), 32 * kEvalWarps, smem, stream>>>(
                batch, L, comp, xfer, dt, bits, makespan, pairs);
        return cudaGetLastError();
    }
    int64_t blocks = (batch + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    if (forward)
        eval_kernel<true><<<unsigned(blocks), 256, 0, stream>>>(batch, L, comp, xfer, dt, bits,
                                                               makespan);
    else
        eval_kernel<false><<<unsigned(blocks), 256, 0, stream>>>(batch, L, comp, xfer, dt,
                                                                bits, makespan);
    return cudaGetLastError();
}

}  // namespace dc
