// Shared device/host helpers of the GB300 DynaComm library (GPU side only).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cstdlib>
#include <mutex>

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "dynacomm.h"

namespace dc {

constexpr int kSmallLMax = 16;       // unrolled thread-per-instance kernel: 1 <= L <= 16
constexpr int kMidLMax = 256;        // looped thread-per-instance kernel: 17 <= L <= 256
constexpr int kSmemTableLMax = 64;   // group kernel keeps its DP table on chip up to here
constexpr int64_t kMidSlots = 152 * 16 * 32;  // traceback slots of the looped kernel (L <= 64)
constexpr int64_t kRangeLimit = int64_t(1) << 52;
constexpr uint64_t kNarrowLimit = 0xFFFFFFFEull;  // bound that lets a DP run in 32 bits
// capped bound under which the shifted form of a DP runs in signed 32 bits
constexpr uint64_t kShiftedLimit = 0x7FFFFFFFull;

// Triangle of DP cells (m, n), 1 <= n <= m <= L, stored column by column:
// column n holds rows n..L contiguously.
__host__ __device__ inline int64_t tri_cells(int L) { return int64_t(L) * (L + 1) / 2; }
__host__ __device__ inline int64_t tri_col(int L, int n)
{
    return int64_t(n - 1) * L - int64_t(n - 1) * (n - 2) / 2;
}
__host__ __device__ inline int64_t tri_index(int L, int m, int n) { return tri_col(L, n) + (m - n); }

__host__ __device__ inline int words_for(int L) { return (L - 1 + 31) / 32; }

// Group-kernel table slots (L > kSmemTableLMax): enough CTAs to fill the GPU
// several times over, capped so one launch's tables stay within ~4 GiB.
inline int64_t table_slots(int L)
{
    const int64_t per = tri_cells(L) * 8;
    int64_t s = (int64_t(4) << 30) / per;
    if (s > 152 * 32) s = 152 * 32;  // up to 32 one-warp CTAs per SM
    if (s < 152) s = 152;
    return s;
}

size_t mid_scratch_bytes(int64_t batch, int L);  // dp_mid.cu
size_t deep_slot_bytes(int L);                   // dp_deep.cu
int64_t deep_slots_bound(int L);                 // dp_deep.cu

// CTA-per-instance tables for the instances the deep-chain kernel lists (L >
// kMidLMax): a few, within ~1 GiB.
inline int64_t list_table_slots(int L)
{
    const int64_t per = tri_cells(L) * 8;
    int64_t s = (int64_t(1) << 30) / per;
    if (s > 152 * 4) s = 152 * 4;
    if (s < 4) s = 4;
    return s;
}

struct Workspace {
    // Layout: [0, 256) header (work-list counter, tile ticket), [256, 256 +
    // 4*batch) work list, then, 256-aligned, the looped kernel's traceback slots
    // (17 <= L <= kMidLMax) or, for L > kMidLMax, the deep-chain kernel's slot
    // flags and per-launch tickets (4 bytes each) and, 256-aligned, its per-CTA
    // slots; then, 256-aligned, the per-CTA DP tables of the group kernel for
    // the listed instances (L > kSmemTableLMax).
    static size_t list_bytes(int64_t batch, int) { return size_t(batch) * 4; }
    static size_t table_offset(int64_t batch, int L)
    {
        return (256 + list_bytes(batch, L) + 255) / 256 * 256;
    }
    static size_t slots(int64_t batch, int L)
    {
        if (L <= kSmemTableLMax) return 0;
        const int64_t s = L > kMidLMax ? list_table_slots(L) : table_slots(L);
        return size_t(batch < s ? batch : s);
    }
    static int64_t deep_slots(int64_t batch, int L)
    {
        if (L <= kMidLMax) return 0;
        const int64_t s = deep_slots_bound(L);
        return batch < s ? batch : s;
    }
    static size_t deep_slots_offset(int64_t batch, int L)
    {
        return (table_offset(batch, L) + size_t(deep_slots(batch, L) + batch) * 4 + 255) / 256 * 256;
    }
    static size_t group_tables_offset(int64_t batch, int L)
    {
        if (L > kSmallLMax && L <= kMidLMax)
            return (table_offset(batch, L) + mid_scratch_bytes(batch, L) + 255) / 256 * 256;
        if (L > kMidLMax)
            return deep_slots_offset(batch, L) + size_t(deep_slots(batch, L)) * deep_slot_bytes(L);
        return table_offset(batch, L);
    }
    static size_t bytes(int64_t batch, int L)
    {
        return group_tables_offset(batch, L) + slots(batch, L) * size_t(tri_cells(L)) * 8;
    }
};

// Index checks of the checked build (compiled with -DDC_CHECKED): a check that
// fails counts itself in this translation unit's device counters (the first
// failing source line is kept) and the caller skips the access; nothing traps.
// dc_checked_<unit>() reads (and optionally clears) a unit's counters from the
// host. In the normal build DC_CHECK(cond) is `true` and costs nothing.
#ifdef DC_CHECKED
namespace {
__device__ unsigned int g_check_count;
__device__ unsigned int g_check_line;
__device__ __noinline__ bool check_failed(unsigned line)
{
    if (atomicAdd(&g_check_count, 1u) == 0u) atomicExch(&g_check_line, line);
    return false;
}
}  // namespace
#define DC_CHECK(cond) ((cond) ? true : ::dc::check_failed(__LINE__))
#define DC_CHECKED_EXPORT(unit)                                                                \
    extern "C" int dc_checked_##unit(unsigned int *count, unsigned int *line, int reset)       \
    {                                                                                          \
        if (cudaMemcpyFromSymbol(count, ::dc::g_check_count, sizeof(unsigned int)) !=          \
                cudaSuccess ||                                                                 \
            cudaMemcpyFromSymbol(line, ::dc::g_check_line, sizeof(unsigned int)) != cudaSuccess) \
            return -1;                                                                         \
        if (reset) {                                                                           \
            const unsigned int z = 0u;                                                         \
            if (cudaMemcpyToSymbol(::dc::g_check_count, &z, sizeof z) != cudaSuccess ||        \
                cudaMemcpyToSymbol(::dc::g_check_line, &z, sizeof z) != cudaSuccess)           \
                return -1;                                                                     \
        }                                                                                      \
        return 0;                                                                              \
    }
#else
#define DC_CHECK(cond) true
#define DC_CHECKED_EXPORT(unit)
#endif

// An NVTX range over one C-ABI call: named on the timelines of Nsight Systems
// and Nsight Compute when a tool is attached, a few instructions otherwise
// (header-only NVTX 3; it loads no library unless a tool asks).
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};

// Test hook for the barrier discipline: DC_BLOCK_WARPS=1|2|4|8 in the
// environment makes the looped, deep-chain and CTA-per-instance kernels run with
// that many warps per CTA where the kernel allows it (results must not change);
// unset or any other value keeps each kernel's own choice. Read on every launch.
inline int forced_warps()
{
    const char *e = std::getenv("DC_BLOCK_WARPS");
    if (!e) return 0;
    const int v = std::atoi(e);
    return (v == 1 || v == 2 || v == 4 || v == 8) ? v : 0;
}

// A per-device launch fact (resident CTAs per SM of a kernel, the SM count),
// found once per device by the first call that needs it; `lookup` may also
// raise a kernel's shared-memory limit on the way. Thread-safe: lookups run
// under the cache's mutex, so host threads that launch at once do not race,
// and each device ordinal keeps its own value. A context re-created after
// cudaDeviceReset keeps these numbers (they describe the device); a kernel
// attribute raised in the old context is gone, and a launch that needed it
// then fails with a CUDA error instead of running.
constexpr int kMaxDevices = 64;
class DeviceCache {
public:
    template <typename F>
    cudaError_t get(int &out, F &&lookup)
    {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
        std::lock_guard<std::mutex> lock(mu_);
        if (value_[dev] <= 0) {
            int v = 0;
            e = lookup(v);
            if (e != cudaSuccess) return e;
            value_[dev] = v > 0 ? v : 1;
        }
        out = value_[dev];
        return cudaSuccess;
    }

private:
    std::mutex mu_;
    int value_[kMaxDevices] = {};
};

// L*dt + sum(comp) + sum(xfer) >= 2^52, for inputs already known to be
// non-negative and below 2^52 each (so each sum of <= 4096 terms fits 64 bits).
__host__ __device__ inline bool exceeds_range(int L, int64_t dt, uint64_t sc, uint64_t sx)
{
    const uint64_t lim = uint64_t(kRangeLimit);
    if (sc >= lim || sx >= lim) return true;
    const uint64_t tl = uint64_t(L) * uint64_t(dt);
    return tl >= lim || sc + sx + tl >= lim;
}

// Programmatic dependent launch (sm_90 and later). A kernel launched with the
// programmatic stream serialization attribute may begin before the kernel ahead
// of it in the stream has finished: pdl_wait() then holds its threads (a
// hardware wait, not a spin) until that kernel has completed and its memory
// writes are visible; pdl_trigger() in the earlier kernel lets the later one
// start launching before the earlier one's CTAs exit.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename T>
__device__ __forceinline__ T dmax(T a, T b) { return a > b ? a : b; }
template <typename T>
__device__ __forceinline__ T dmin(T a, T b) { return a < b ? a : b; }

// A timing request (dc_time_next_pass) for the next schedule call made on this
// thread: events recorded on the call's stream right before and right after the
// launches of its first pass over the batch.
struct PassEvents {
    cudaEvent_t start = nullptr, stop = nullptr;
};
PassEvents take_pass_events();  // this thread's request, cleared (dynacomm_abi.cu)

// Kernel launchers implemented in the .cu files.
cudaError_t launch_schedule(bool forward, int64_t batch, int L, const int64_t *comp,
                            const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                            uint32_t *bits, int32_t *nseg, int32_t *status, void *workspace,
                            const PassEvents &pe, cudaStream_t stream);
cudaError_t launch_small(bool forward, int64_t batch, int L, const int64_t *comp,
                         const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                         uint32_t *bits, int32_t *nseg, int32_t *status,
                         uint32_t *wide_count, uint32_t *wide_list, const PassEvents &pe,
                         cudaStream_t stream);
cudaError_t launch_group(bool forward, int64_t batch, int L, const int64_t *comp,
                         const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                         uint32_t *bits, int32_t *nseg, int32_t *status,
                         const uint32_t *list_count, const uint32_t *list, void *tables,
                         int64_t grid, cudaStream_t stream);
cudaError_t launch_mid(bool forward, int64_t batch, int L, const int64_t *comp,
                       const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                       uint32_t *bits, int32_t *nseg, int32_t *status, uint32_t *ticket,
                       uint32_t *list_count, uint32_t *list, uint32_t *tb, cudaStream_t stream);
cudaError_t launch_deep(bool forward, int64_t batch, int L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                        uint32_t *bits, int32_t *nseg, int32_t *status, uint32_t *tickets,
                        uint32_t *busy, uint32_t *list_count, uint32_t *list, void *slots,
                        int64_t nslots, cudaStream_t stream);
int64_t deep_launches(int64_t batch, int L);  // launches of one deep-chain pass (dp_deep.cu)
cudaError_t launch_eval(bool forward, int64_t batch, int L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                        int64_t *makespan, cudaStream_t stream);
cudaError_t launch_roof(int variant, int blocks, int threads, int64_t iters, uint32_t *sink,
                        cudaStream_t stream);

}  // namespace dc
