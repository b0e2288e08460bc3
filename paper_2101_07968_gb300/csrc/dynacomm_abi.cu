// C ABI entry points (declared in include/dynacomm.h): host-side argument
// checks, then kernel launches on the caller's stream. No allocation, no
// synchronisation, no state kept between calls (save the timing request of
// dc_time_next_pass, which the thread's next schedule call uses up).
#include "gen_device.cuh"

namespace dc {

cudaError_t launch_gen(const dc_profile_cfg *c, int64_t *fc, int64_t *pt, int64_t *bc,
                       int64_t *gt, int64_t *dt, cudaStream_t stream);

namespace {
thread_local PassEvents t_pass_events;  // dc_time_next_pass's request for this thread
}  // namespace

PassEvents take_pass_events()
{
    const PassEvents pe = t_pass_events;
    t_pass_events = PassEvents{};
    return pe;
}

// Forward and backward solves share one path after the layers are put in
// processing order (done inside the kernels).
cudaError_t launch_schedule(bool forward, int64_t batch, int L, const int64_t *comp,
                            const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                            uint32_t *bits, int32_t *nseg, int32_t *status, void *workspace,
                            const PassEvents &pe, cudaStream_t stream)
{
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    // events around the first pass of a looped or deep-chain solve
    auto mark = [&](cudaEvent_t ev) { return ev ? cudaEventRecord(ev, stream) : cudaSuccess; };
    if (L <= kSmallLMax) {
        // header: work-list counter, then the dense pass's tile ticket
        uint32_t *count = reinterpret_cast<uint32_t *>(ws);
        uint32_t *list = reinterpret_cast<uint32_t *>(ws + 256);
        cudaError_t e = cudaMemsetAsync(count, 0, 2 * sizeof(uint32_t), stream);
        if (e != cudaSuccess) return e;
        // 32-bit pass over the batch, then a 64-bit pass over the instances it listed
        return launch_small(forward, batch, L, comp, xfer, dt, makespan, bits, nseg, status,
                            count, list, pe, stream);
    }
    if (L <= kMidLMax) {
        // looped 32-bit pass (tile ticket + work list in the header), then the
        // CTA-per-instance kernel over the listed 64-bit / deep instances
        uint32_t *count = reinterpret_cast<uint32_t *>(ws);
        uint32_t *ticket = count + 1;
        uint32_t *list = reinterpret_cast<uint32_t *>(ws + 256);
        uint32_t *tb = reinterpret_cast<uint32_t *>(ws + Workspace::table_offset(batch, L));
        cudaError_t e = cudaMemsetAsync(count, 0, 2 * sizeof(uint32_t), stream);
        if (e != cudaSuccess) return e;
        e = mark(pe.start);
        if (e != cudaSuccess) return e;
        e = launch_mid(forward, batch, L, comp, xfer, dt, makespan, bits, nseg, status, ticket,
                       count, list, tb, stream);
        if (e != cudaSuccess) return e;
        e = mark(pe.stop);
        if (e != cudaSuccess) return e;
        if (L <= kSmemTableLMax) {  // tables of the listed instances in shared memory
            const int64_t grid = batch < 152 * 8 ? batch : 152 * 8;
            return launch_group(forward, batch, L, comp, xfer, dt, makespan, bits, nseg, status,
                                count, list, nullptr, grid, stream);
        }
        return launch_group(forward, batch, L, comp, xfer, dt, makespan, bits, nseg, status,
                            count, list, ws + Workspace::group_tables_offset(batch, L),
                            int64_t(Workspace::slots(batch, L)), stream);
    }
    // warp-per-instance pass over the batch (three shifted 32-bit forms), then
    // the CTA-per-instance kernel over the instances it listed
    uint32_t *count = reinterpret_cast<uint32_t *>(ws);
    uint32_t *list = reinterpret_cast<uint32_t *>(ws + 256);
    const int64_t nslots = Workspace::deep_slots(batch, L);
    uint32_t *busy = reinterpret_cast<uint32_t *>(ws + Workspace::table_offset(batch, L));
    uint32_t *tickets = busy + nslots;
    cudaError_t e = cudaMemsetAsync(count, 0, sizeof(uint32_t), stream);
    if (e != cudaSuccess) return e;
    e = mark(pe.start);
    if (e != cudaSuccess) return e;
    e = launch_deep(forward, batch, L, comp, xfer, dt, makespan, bits, nseg, status, tickets,
                    busy, count, list, ws + Workspace::deep_slots_offset(batch, L), nslots,
                    stream);
    if (e != cudaSuccess) return e;
    e = mark(pe.stop);
    if (e != cudaSuccess) return e;
    return launch_group(forward, batch, L, comp, xfer, dt, makespan, bits, nseg, status, count,
                        list, ws + Workspace::group_tables_offset(batch, L),
                        int64_t(Workspace::slots(batch, L)), stream);
}

namespace {

dc_status schedule(bool forward, int64_t batch, int32_t L, const int64_t *comp,
                   const int64_t *xfer, const int64_t *dt, int64_t *makespan, uint32_t *bits,
                   int32_t *nseg, int32_t *status, void *workspace, size_t workspace_bytes,
                   cudaStream_t stream)
{
    const PassEvents pe = take_pass_events();  // used up by this call, whatever it returns
    if (batch < 0 || L < 1 || L > DC_L_MAX || batch > int64_t(0xffffffffll))
        return DC_ERR_BAD_SHAPE;
    if (batch == 0) return DC_OK;
    if (!comp || !xfer || !dt || !makespan || (!bits && words_for(L) > 0)) return DC_ERR_NULL;
    if (!workspace || workspace_bytes < Workspace::bytes(batch, L)) return DC_ERR_WORKSPACE;
    const cudaError_t e = launch_schedule(forward, batch, L, comp, xfer, dt, makespan, bits,
                                          nseg, status, workspace, pe, stream);
    return e == cudaSuccess ? DC_OK : DC_ERR_CUDA;
}

}  // namespace
}  // namespace dc

extern "C" {

dc_status dc_profile_gen(const dc_profile_cfg *cfg, int64_t *fc, int64_t *pt, int64_t *bc,
                         int64_t *gt, int64_t *dt, cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_profile_gen");
    if (!cfg) return DC_ERR_NULL;
    const dc_status st = dc::check_profile_cfg(cfg);
    if (st != DC_OK) return st;
    if (cfg->batch == 0) return DC_OK;
    if (!fc || !pt || !bc || !gt || !dt) return DC_ERR_NULL;
    return dc::launch_gen(cfg, fc, pt, bc, gt, dt, stream) == cudaSuccess ? DC_OK : DC_ERR_CUDA;
}

size_t dc_schedule_generated_workspace_bytes(int64_t batch, int32_t L)
{
    if (batch < 0 || L < 1 || L > dc::kSmallLMax) return 0;
    return dc::fused_workspace_bytes(batch);
}

dc_status dc_schedule_generated_batch(const dc_profile_cfg *cfg, int64_t *makespan,
                                      uint32_t *bits, int32_t *nseg, int32_t *status,
                                      void *workspace, size_t workspace_bytes,
                                      cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_schedule_generated_batch");
    if (!cfg) return DC_ERR_NULL;
    const dc_status st = dc::check_profile_cfg(cfg);
    if (st != DC_OK) return st;
    if (cfg->L > dc::kSmallLMax || cfg->batch > int64_t(0xffffffffll)) return DC_ERR_BAD_SHAPE;
    if (cfg->batch == 0) return DC_OK;
    if (!makespan || (!bits && dc::words_for(cfg->L) > 0)) return DC_ERR_NULL;
    if (!workspace || workspace_bytes < dc::fused_workspace_bytes(cfg->batch))
        return DC_ERR_WORKSPACE;
    static thread_local dc::GenParams g;  // 25 KB: kept off the caller's stack
    dc::fill_gen_params(cfg, g);
    return dc::launch_fused(g, makespan, bits, nseg, status, workspace, stream) == cudaSuccess
               ? DC_OK
               : DC_ERR_CUDA;
}

int32_t dc_schedule_kernel_launches(int64_t batch, int32_t L)
{
    if (batch <= 0 || L < 1 || L > DC_L_MAX) return 0;
    if (L <= dc::kMidLMax) return 2;
    return int32_t(dc::deep_launches(batch, L) + 1);
}

size_t dc_schedule_workspace_bytes(int64_t batch, int32_t L)
{
    if (batch < 0 || L < 1 || L > DC_L_MAX) return 0;
    return dc::Workspace::bytes(batch, L);
}

dc_status dc_schedule_forward_batch(int64_t batch, int32_t L, const int64_t *fc,
                                    const int64_t *pt, const int64_t *dt, int64_t *makespan,
                                    uint32_t *bits, int32_t *nseg, int32_t *status,
                                    void *workspace, size_t workspace_bytes, cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_schedule_forward_batch");
    return dc::schedule(true, batch, L, fc, pt, dt, makespan, bits, nseg, status, workspace,
                        workspace_bytes, stream);
}

dc_status dc_schedule_backward_batch(int64_t batch, int32_t L, const int64_t *bc,
                                     const int64_t *gt, const int64_t *dt, int64_t *makespan,
                                     uint32_t *bits, int32_t *nseg, int32_t *status,
                                     void *workspace, size_t workspace_bytes,
                                     cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_schedule_backward_batch");
    return dc::schedule(false, batch, L, bc, gt, dt, makespan, bits, nseg, status, workspace,
                        workspace_bytes, stream);
}

dc_status dc_eval_timeline_batch(int64_t batch, int32_t L, int32_t dir, const int64_t *comp,
                                 const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                                 int64_t *makespan, cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_eval_timeline_batch");
    if (batch < 0 || L < 1 || L > DC_L_MAX || (dir != 0 && dir != 1)) return DC_ERR_BAD_SHAPE;
    if (batch == 0) return DC_OK;
    if (!comp || !xfer || !dt || !makespan || (!bits && dc::words_for(L) > 0))
        return DC_ERR_NULL;
    return dc::launch_eval(dir == 0, batch, L, comp, xfer, dt, bits, makespan, stream) ==
                   cudaSuccess
               ? DC_OK
               : DC_ERR_CUDA;
}

const char *dc_status_string(dc_status s)
{
    switch (s) {
        case DC_OK: return "ok";
        case DC_ERR_NULL: return "a required pointer is NULL";
        case DC_ERR_BAD_SHAPE: return "bad batch, L or direction";
        case DC_ERR_NEGATIVE: return "negative cost or latency";
        case DC_ERR_RANGE: return "L*dt + sum(xfer) + sum(comp) >= 2^52";
        case DC_ERR_WORKSPACE: return "workspace missing or too small";
        case DC_ERR_CUDA: return "CUDA runtime error";
        case DC_ERR_BAD_CONFIG: return "profile generator config out of range";
        case DC_ERR_INTERNAL: return "solver self-check failed";
    }
    return "unknown status";
}

dc_status dc_time_next_pass(cudaEvent_t start, cudaEvent_t stop)
{
    if ((start == nullptr) != (stop == nullptr)) return DC_ERR_NULL;
    dc::t_pass_events.start = start;
    dc::t_pass_events.stop = stop;
    return DC_OK;
}

dc_status dc_roof_int_probe(int32_t variant, int32_t blocks, int32_t threads, int64_t iters,
                            uint32_t *sink, cudaStream_t stream)
{
    const dc::NvtxRange nvtx("dc_roof_int_probe");
    if (variant != 0 && variant != 1) return DC_ERR_BAD_SHAPE;
    if (blocks < 1 || threads < 32 || threads > 1024 || threads % 32 || iters < 0 || iters % 4)
        return DC_ERR_BAD_SHAPE;
    if (!sink) return DC_ERR_NULL;
    return dc::launch_roof(variant, blocks, threads, iters, sink, stream) == cudaSuccess
               ? DC_OK
               : DC_ERR_CUDA;
}

}  // extern "C"
