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
#include "common.cuh"

namespace dc {
namespace {

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
        bool neg = d < 0, big = (d >> 52) != 0;
        uint64_t sc = 0, sx = 0;
        // unsigned so that garbage from rejected inputs wraps instead of overflowing
        uint64_t clock_a = 0;  // forward: compute end; backward: link end
        uint64_t run = 0;      // forward: pull end; backward: compute end
        uint64_t seg = 0;      // forward: segment compute; backward: segment transfer
        uint32_t word = 0;
        for (int r = 1; r <= L; ++r) {
            const int col = FWD ? r - 1 : L - r;
            const int64_t cv = __ldg(crow + col), xv = __ldg(xrow + col);
            neg |= (cv < 0) | (xv < 0);
            big |= ((cv | xv) >> 52) != 0;
            sc += uint64_t(cv);
            sx += uint64_t(xv);
            if (((r - 1) & 31) == 0 && r <= L - 1) word = __ldg(brow + ((r - 1) >> 5));
            const bool cut = (r == L) || ((word >> ((r - 1) & 31)) & 1u);
            if (FWD) {
                run += uint64_t(xv);  // pulled bytes so far
                seg += uint64_t(cv);
                if (cut) {
                    run += uint64_t(d);  // one more transmission set-up
                    clock_a = (clock_a > run ? clock_a : run) + seg;
                    seg = 0;
                }
            } else {
                run += uint64_t(cv);  // backward compute done so far
                seg += uint64_t(xv);
                if (cut) {
                    clock_a = (clock_a > run ? clock_a : run) + uint64_t(d) + seg;
                    seg = 0;
                }
            }
        }
        int64_t out = int64_t(clock_a);
        if (neg)
            out = -int64_t(DC_ERR_NEGATIVE);
        else if (big || exceeds_range(L, d, sc, sx))
            out = -int64_t(DC_ERR_RANGE);
        makespan[i] = out;
    }
}

}  // namespace

cudaError_t launch_eval(bool forward, int64_t batch, int L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                        int64_t *makespan, cudaStream_t stream)
{
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
