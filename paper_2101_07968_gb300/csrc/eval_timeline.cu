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
// For L <= 32 a warp first copies its 32 instances' rows into shared memory with
// coalesced asynchronous copies (odd row stride: conflict-free per-lane row
// reads); longer rows are read by each thread directly.
#include "common.cuh"

namespace dc {
namespace {

constexpr int kStagedLMax = 32;
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

template <bool FWD>
__global__ void __launch_bounds__(32 * kEvalWarps)
    eval_staged_kernel(int64_t batch, int L, const int64_t *__restrict__ comp,
                       const int64_t *__restrict__ xfer, const int64_t *__restrict__ dt,
                       const uint32_t *__restrict__ bits, int64_t *__restrict__ makespan)
{
    extern __shared__ __align__(16) int64_t stage[];
    const int stride = L | 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int64_t *stC = stage + warp * 2 * 32 * stride;
    int64_t *stX = stC + 32 * stride;
    const int64_t tiles = (batch + 31) / 32;
    for (int64_t tile = int64_t(blockIdx.x) * kEvalWarps + warp; tile < tiles;
         tile += int64_t(gridDim.x) * kEvalWarps) {
        const int64_t base = tile * 32;
        const int rows = int(batch - base < 32 ? batch - base : 32);
        const int nel = rows * L;
        const int64_t *gC = comp + base * L;
        const int64_t *gX = xfer + base * L;
        __syncwarp();
        // all copies in flight at once (no register round trip), then one wait
        for (int e = lane; e < nel; e += 32) {
            const int r = e / L, cidx = e - r * L;
            cp_async8(stC + r * stride + cidx, gC + e);
            cp_async8(stX + r * stride + cidx, gX + e);
        }
        asm volatile("cp.async.commit_group;\n" ::: "memory");
        asm volatile("cp.async.wait_group 0;\n" ::: "memory");
        __syncwarp();
        if (lane >= rows) continue;
        const int64_t i = base + lane;
        const int64_t d = __ldg(dt + i);
        const uint32_t word = L > 1 ? __ldg(bits + i) : 0u;  // W = 1 for 2 <= L <= 32
        Replay rp;
        for (int r = 1; r <= L; ++r) {
            const int col = FWD ? r - 1 : L - r;
            const bool cut = (r == L) || ((word >> ((r - 1) & 31)) & 1u);
            rp.step<FWD>(stC[lane * stride + col], stX[lane * stride + col], uint64_t(d), cut);
        }
        makespan[i] = rp.result(L, d);
    }
}

}  // namespace

cudaError_t launch_eval(bool forward, int64_t batch, int L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                        int64_t *makespan, cudaStream_t stream)
{
    if (L <= kStagedLMax) {
        const int stride = L | 1;
        const size_t smem = size_t(kEvalWarps) * 2 * 32 * stride * 8;
        int64_t blocks = ((batch + 31) / 32 + kEvalWarps - 1) / kEvalWarps;
        if (blocks > 152 * 32) blocks = 152 * 32;
        static bool attr_set = false;  // up to 67.6 KB at L = 32: above the 48 KB default
        if (!attr_set) {
            const int most = kEvalWarps * 2 * 32 * (kStagedLMax | 1) * 8;
            cudaError_t e = cudaFuncSetAttribute(
                eval_staged_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, most);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(eval_staged_kernel<false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, most);
            if (e != cudaSuccess) return e;
            attr_set = true;
        }
        if (forward)
            eval_staged_kernel<true><<<unsigned(blocks), 32 * kEvalWarps, smem, stream>>>(
                batch, L, comp, xfer, dt, bits, makespan);
        else
            eval_staged_kernel<false><<<unsigned(blocks), 32 * kEvalWarps, smem, stream>>>(
                batch, L, comp, xfer, dt, bits, makespan);
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
