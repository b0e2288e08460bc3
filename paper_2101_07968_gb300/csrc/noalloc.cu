// dc_schedule_batch_static: the L <= 16 solve without a caller workspace.
//
// Some callers cannot allocate device memory at the point where they schedule:
// a scheduler embedded in a training runtime whose allocator owns all device
// memory (a framework's caching allocator or an arena reserved at start-up) and
// refuses other allocations once training runs, or one that schedules inside the
// short idle window between a gradient push and the next pull, where a
// cudaMalloc -- which can synchronise the whole device -- is not acceptable.
// This entry point needs no workspace: its scratch (the 64-bit work list and its
// counter) lives in a fixed-size array in this library's device memory.
//
// The array is a file-scope __device__ variable, so every GPU that loads this
// library holds it (4 MiB + 256 B) until the process exits, and every call on a
// device shares it: calls that overlap on one GPU race on it and must be
// serialised by the caller (one stream, or an event between them). The counter
// that must start at zero is cleared on the caller's stream by each call.
#include "common.cuh"

namespace dc {
namespace {

constexpr int64_t kStaticMaxBatch = int64_t(1) << 20;
constexpr size_t kStaticScratchBytes = 256 + size_t(kStaticMaxBatch) * 4;  // header + list

__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// In host code `g_static_scratch` names a host-side stand-in, not device memory.
// Its device address on the current device is looked up on every call: the
// lookup allocates nothing, and no address is kept that a re-created context
// (after a cudaDeviceReset, say) could have moved. On the first call on a
// device, the lookup also loads this library's device code there if that has
// not happened yet, which is why that first call belongs before any capture.
cudaError_t static_scratch(void **out)
{
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return e;
    *out = p;
    return cudaSuccess;
}

static_assert(kStaticScratchBytes >= 256 + 4 * size_t(kStaticMaxBatch),
              "the work list needs 4 bytes per instance after the 256-byte header");

}  // namespace
}  // namespace dc

extern "C" dc_status dc_schedule_batch_static(int32_t dir, int64_t batch, int32_t L,
                                              const int64_t *comp, const int64_t *xfer,
                                              const int64_t *dt, int64_t *makespan,
                                              uint32_t *bits, int32_t *nseg, int32_t *status,
                                              cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_schedule_batch_static");
    const dc::PassEvents pe = dc::take_pass_events();  // a timing request is used up here too
    if ((dir != 0 && dir != 1) || batch < 0 || L < 1 || L > dc::kSmallLMax)
        return DC_ERR_BAD_SHAPE;
    if (batch > dc::kStaticMaxBatch) return DC_ERR_WORKSPACE;  // beyond the static scratch
    if (batch == 0) return DC_OK;
    if (!comp || !xfer || !dt || !makespan || (!bits && dc::words_for(L) > 0))
        return DC_ERR_NULL;
    void *scratch = nullptr;
    if (dc::static_scratch(&scratch) != cudaSuccess) return DC_ERR_CUDA;
    const cudaError_t e = dc::launch_schedule(dir == 0, batch, L, comp, xfer, dt, makespan,
                                              bits, nseg, status, scratch, pe, stream);
    return e == cudaSuccess ? DC_OK : DC_ERR_CUDA;
}
