/*
 * dynacomm.h -- C ABI of the GB300 (sm_103a) DynaComm scheduling library.
 *
 * DynaComm (Cai et al., arXiv 2101.07968) splits the parameter pull before the
 * forward pass and the gradient push after the backward pass of one training
 * iteration into contiguous multi-layer transmissions, so that transfers
 * overlap layer computation, and picks the split that minimises the makespan
 * with two dynamic programs (Sec. IV-B, Eq. 8 / Algorithm 3 and Eq. 9 /
 * Algorithm 4). This library solves very many independent instances of that
 * problem (Sec. III-B, the 0-1 program over p and g) at once on one GPU.
 *
 * Conventions that hold for every call below:
 *  - Times are int64 microseconds (the paper uses real-valued times; integer
 *    microseconds make GPU and CPU results comparable bit for bit).
 *  - Per-layer arrays are row-major [batch][L]; element [i][l-1] belongs to layer
 *    l of instance i, layers numbered 1..L in forward order (Sec. III-A).
 *  - Unless stated otherwise, array pointers are DEVICE pointers owned by the
 *    caller, 8-byte aligned for int64 and 4-byte aligned for 32-bit arrays. The
 *    library keeps no pointer after a call returns and allocates no memory: the
 *    scratch the solver needs comes from the caller's workspace.
 *  - Calls are asynchronous on `stream` (0 = the legacy default stream). Errors
 *    the host can see (null pointers, bad sizes, short workspace, bad config)
 *    return synchronously and launch nothing. batch == 0 returns DC_OK and does
 *    nothing. DC_ERR_CUDA reports a launch error from the CUDA runtime.
 *  - Data-dependent faults are per instance and never stop the batch: an
 *    instance with a negative cost or latency gets status DC_ERR_NEGATIVE, one
 *    whose bound L*dt + sum(xfer) + sum(comp) is >= 2^52 gets DC_ERR_RANGE; its
 *    makespan is written as -(status), its nseg as 0 and its bits as 0.
 *  - Decision bits: W = ceil((L-1)/32) uint32 words per instance (W = 0 when
 *    L = 1). Bit (l-1)%32 of word (l-1)/32 is p_l for the forward direction (a
 *    new pull starts at layer l+1) and g_l for the backward direction (the last
 *    l layers are pushed apart from layer L-l), Sec. III-B.
 */
#ifndef DYNACOMM_H
#define DYNACOMM_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum dc_status {
    DC_OK = 0,
    DC_ERR_NULL = 1,       /* a required pointer is NULL */
    DC_ERR_BAD_SHAPE = 2,  /* batch < 0, L < 1, L > DC_L_MAX, or dir not 0/1 */
    DC_ERR_NEGATIVE = 3,   /* per instance: a negative cost or latency */
    DC_ERR_RANGE = 4,      /* per instance: L*dt + sum(xfer) + sum(comp) >= 2^52 */
    DC_ERR_WORKSPACE = 5,  /* workspace NULL or smaller than the query returned */
    DC_ERR_CUDA = 6,       /* the CUDA runtime reported an error for a launch */
    DC_ERR_BAD_CONFIG = 7, /* a profile-generator config field is out of range */
    DC_ERR_INTERNAL = 8    /* per instance: solver self-check failed (a bug) */
} dc_status;

#define DC_L_MAX 4096

/* ------------------------------------------------------------------------
 * dc_profile_gen -- seeded synthetic profiles (stand-in for the real-time
 * profiler of Sec. IV-A, which reads pt, fc, bc, gt and dt off a framework
 * profiler; no profiler or real training exists here).
 *
 * For instance i (global index g = cfg->inst0 + i) and layer l (0-based):
 *   draw(field, l) = SplitMix64 output number ctr+1 for state cfg->seed, with
 *                    ctr = g<<20 | field<<12 | l (field: 0 rate, 1 bandwidth,
 *                    2 latency, 3 params, 4 FLOPs)
 *   uniform-int [a,b]  = a + floor(r * (b-a+1) / 2^64)
 *   log-uniform [a,b]  = knots T(j) = llround(a * exp((j/512) * ln(b/a))),
 *                        T(0) = a, T(512) = b, evaluated in IEEE double;
 *                        j = r>>55, f = (r>>23) & 0xffffffff,
 *                        value = T(j) + floor((T(j+1)-T(j)) * f / 2^32)
 *   rate (FLOP/us), bw (kbit/s), dt (us, uniform-int) per instance;
 *   params, FLOPs per layer: fixed tables or per-instance draws;
 *   fc = ceil(FLOPs/rate), bc = ceil(bwd_flops_mult*FLOPs/rate),
 *   pt = gt = ceil(bits_per_param*1000*params/bw).
 * Outputs fc, pt, bc, gt: [batch][L] int64; dt: [batch] int64 (device).
 * fixed_params / fixed_flops are HOST pointers of L entries, read during the
 * call only. Limits (else DC_ERR_BAD_CONFIG): 1 <= L <= DC_L_MAX (<= 1024 with
 * fixed tables); inst0 >= 0, inst0 + batch <= 2^44; 1 <= rate_lo <= rate_hi <
 * 2^31 and the same for bw; 0 <= dt_lo <= dt_hi <= 2^40; params and FLOPs
 * (drawn ranges or fixed entries) in [0, 2^40], lo >= 1 for log-uniform draws;
 * 1 <= bwd_flops_mult <= 16; 1 <= bits_per_param <= 64.
 * ---------------------------------------------------------------------- */
#define DC_LAYERS_FIXED 0
#define DC_LAYERS_UNIFORM 1
#define DC_LAYERS_LOGUNIFORM 2
#define DC_DIST_UNIFORM 0
#define DC_DIST_LOGUNIFORM 1

typedef struct dc_profile_cfg {
    int32_t L;
    int32_t layer_mode; /* DC_LAYERS_* */
    int64_t batch;
    int64_t inst0;
    uint64_t seed;
    const int64_t *fixed_params; /* host, L entries, DC_LAYERS_FIXED only */
    const int64_t *fixed_flops;  /* host, L entries, DC_LAYERS_FIXED only */
    int64_t params_lo, params_hi, flops_lo, flops_hi;
    int32_t rate_dist, bw_dist; /* DC_DIST_* */
    int64_t rate_lo, rate_hi;   /* FLOP per microsecond */
    int64_t bw_lo, bw_hi;       /* kbit per second */
    int64_t dt_lo, dt_hi;       /* per-transmission overhead, microseconds */
    int32_t bwd_flops_mult;
    int32_t bits_per_param;
} dc_profile_cfg;

dc_status dc_profile_gen(const dc_profile_cfg *cfg, int64_t *fc, int64_t *pt, int64_t *bc,
                         int64_t *gt, int64_t *dt, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * dc_schedule_workspace_bytes -- device scratch a schedule call needs for
 * (batch, L): a work list for instances that the first pass leaves to a
 * second (values beyond its 32-bit forms, or an optimum with more segments
 * than it keeps traceback columns for); traceback slots of the
 * thread-per-instance kernel (17 <= L <= 256) or, for L > 256, the per-CTA
 * slots of the warp-per-instance kernel with their flags and per-launch
 * counters; for L > 64, per-CTA DP tables of the second pass. Pure host
 * function, no CUDA call.
 * ---------------------------------------------------------------------- */
size_t dc_schedule_workspace_bytes(int64_t batch, int32_t L);

/* ------------------------------------------------------------------------
 * dc_schedule_kernel_launches -- how many kernels one dc_schedule_forward_batch
 * or dc_schedule_backward_batch call with (batch, L) launches: a first pass and
 * a second pass over its work list; for L > 256 the first pass is split into
 * launches of about 90 ms of work each (at least two resident waves), chained
 * so that each may start while the one before drains. For counting only (the
 * calls need no caller action per launch). Returns 0 for batch <= 0 or L out of
 * range. Pure host function, no CUDA call.
 * ---------------------------------------------------------------------- */
int32_t dc_schedule_kernel_launches(int64_t batch, int32_t L);

/* ------------------------------------------------------------------------
 * dc_schedule_forward_batch -- Algorithm 3 / Eq. 8 for every instance:
 *   F[m][n] = min_{k} max(F[k][n-1], n*dt + sum_{l<=m} pt_l) + sum_{k<l<=m} fc_l
 * with F[0][0] = 0, then T = min_n F[L][n] (lowest n on ties), then the
 * traceback of Algorithm 3, in which every Path[m][n] is the LOWEST k that
 * attains F[m][n]. Inputs fc, pt: [batch][L]; dt: [batch]. Outputs: makespan
 * [batch] (= T), bits [batch][W] (p_1..p_{L-1}), nseg [batch] (number of
 * pulls, nullable), status [batch] (nullable). The results equal those of
 * Algorithm 3 run in exact integer arithmetic, bit for bit.
 * workspace: device, >= dc_schedule_workspace_bytes(batch, L) bytes, used
 * during the call's kernels only (reuse it after the stream passes them).
 * ---------------------------------------------------------------------- */
dc_status dc_schedule_forward_batch(int64_t batch, int32_t L, const int64_t *fc,
                                    const int64_t *pt, const int64_t *dt, int64_t *makespan,
                                    uint32_t *bits, int32_t *nseg, int32_t *status,
                                    void *workspace, size_t workspace_bytes,
                                    cudaStream_t stream);

/* ------------------------------------------------------------------------
 * dc_schedule_backward_batch -- Algorithm 4 / Eq. 9 for every instance, with m
 * counting the LAST m layers:
 *   B[m][n] = min_k max(B[k][n-1], sum_{L-m<l<=L} bc_l) + dt + sum_{L-m<l<=L-k} gt_l
 * Inputs bc, gt: [batch][L] in forward layer order; outputs as for the
 * forward call with g_1..g_{L-1} in bits. Same workspace rule.
 * ---------------------------------------------------------------------- */
dc_status dc_schedule_backward_batch(int64_t batch, int32_t L, const int64_t *bc,
                                     const int64_t *gt, const int64_t *dt, int64_t *makespan,
                                     uint32_t *bits, int32_t *nseg, int32_t *status,
                                     void *workspace, size_t workspace_bytes,
                                     cudaStream_t stream);

/* ------------------------------------------------------------------------
 * dc_schedule_generated_batch -- dc_profile_gen followed by both
 * dc_schedule_forward_batch and dc_schedule_backward_batch for 1 <= L <= 16,
 * fused: every instance's profile is drawn inside the solving kernel (the same
 * pure function of seed, instance, field and layer that dc_profile_gen writes
 * out) and never stored, so the profiles make no round trip through device
 * memory. The results are those of the unfused calls on dc_profile_gen's output,
 * bit for bit. Outputs, forward first then backward: makespan [2][batch],
 * bits [2][batch][W], nseg [2][batch] and status [2][batch] (both nullable).
 * workspace: device, >= dc_schedule_generated_workspace_bytes(batch, L) bytes
 * (the two work lists and a copy of the generator's tables). Errors: those of dc_profile_gen (config), DC_ERR_BAD_SHAPE
 * for L > 16, DC_ERR_NULL, DC_ERR_WORKSPACE, DC_ERR_CUDA. There is no counterpart
 * in the paper, whose profiler produces the profiles (Sec. IV-A).
 * ---------------------------------------------------------------------- */
size_t dc_schedule_generated_workspace_bytes(int64_t batch, int32_t L);
dc_status dc_schedule_generated_batch(const dc_profile_cfg *cfg, int64_t *makespan, uint32_t *bits,
                                      int32_t *nseg, int32_t *status, void *workspace,
                                      size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * dc_greedy_forward_batch, dc_greedy_backward_batch -- the paper's competing
 * schedulers (Sec. II-C), for comparison with the DP: greedy parameter
 * scheduling of iBatch (Algorithm 1, forward; inputs as
 * dc_schedule_forward_batch) and greedy gradient scheduling of iPart
 * (Algorithm 2, backward; inputs as dc_schedule_backward_batch). Readings of the
 * listings' open points: ties keep the first candidate of the listing's
 * enumeration; an empty Options set takes the position with the largest slack;
 * Algorithm 1's first pair is the qualifying pair with the largest first-segment
 * compute, then the smallest first transfer, then the smallest slack (with no
 * qualifying pair, the largest slack); Algorithm 2 keeps the candidate with the
 * least f_m. Outputs per instance: bits [batch][W] (the decision, same layout
 * as dc_schedule_*) and makespan [batch] (f_m of that decision, as
 * dc_eval_timeline_batch gives it), or -(status) and zero bits for an instance
 * with a negative or out-of-range input (status 3 or 4). No workspace. Errors:
 * DC_ERR_NULL, DC_ERR_BAD_SHAPE (batch < 0 or > 2^32-1, L outside [1, 4096]),
 * DC_ERR_CUDA. Asynchronous on `stream`.
 * ---------------------------------------------------------------------- */
dc_status dc_greedy_forward_batch(int64_t batch, int32_t L, const int64_t *fc, const int64_t *pt,
                                  const int64_t *dt, int64_t *makespan, uint32_t *bits,
                                  cudaStream_t stream);
dc_status dc_greedy_backward_batch(int64_t batch, int32_t L, const int64_t *bc, const int64_t *gt,
                                   const int64_t *dt, int64_t *makespan, uint32_t *bits,
                                   cudaStream_t stream);

/* ------------------------------------------------------------------------
 * dc_eval_timeline_batch -- the cost measurement f_m of Sec. III-B for one
 * direction: replays ANY decision (bits [batch][W]) under the partial orders of
 * Eq. 1-7 and writes its makespan. dir 0: comp = fc, xfer = pt, the pulls run
 * back to back on the link and layer l computes once its pull has arrived and
 * layer l-1 is done. dir 1: comp = bc, xfer = gt, the backward compute runs
 * from layer L down without waiting and a push starts once its layers are
 * computed and the previous push is done. Every transmission costs dt + the
 * sum of its layers' transfer costs. A failed instance gets -(status) as its
 * makespan (no status array here).
 * ---------------------------------------------------------------------- */
dc_status dc_eval_timeline_batch(int64_t batch, int32_t L, int32_t dir, const int64_t *comp,
                                 const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                                 int64_t *makespan, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * dc_schedule_batch_static -- the paper has no counterpart: this is a
 * deployment variant of the two schedule calls above for callers that cannot
 * allocate device memory where they schedule (a scheduler embedded in a
 * training runtime whose allocator owns all device memory and refuses other
 * allocations once training runs, or one that schedules inside the idle window
 * between a gradient push and the next pull, where a cudaMalloc that can
 * synchronise the device is not acceptable). It takes no workspace.
 *
 * dir 0 is the forward call's problem (comp = fc, xfer = pt), dir 1 the
 * backward call's (comp = bc, xfer = gt); inputs, outputs and per-instance
 * status are exactly those of dc_schedule_forward_batch /
 * dc_schedule_backward_batch, including a NULL status (a failed instance's
 * makespan then carries -status).
 * Limits: 1 <= L <= 16 (else DC_ERR_BAD_SHAPE); batch <= 1,048,576
 * (DC_STATIC_MAX_BATCH; a larger batch returns DC_ERR_WORKSPACE, launching
 * nothing).
 * Scratch: a 4 MiB + 256 B array in the library's device memory, held by every
 * GPU that loads the library until the process exits, shared by all calls on a
 * device: calls that overlap on one GPU race on it, so serialise them (one
 * stream, or an event between them). Each call clears what must start at zero.
 * Every call looks up the array's device address on the current device
 * (cudaGetSymbolAddress, which allocates nothing); on a device's first call
 * that lookup also loads the library's device code there if needed, so make
 * the first call on each device before any stream capture. No cudaMalloc,
 * cudaFree or other allocating call is made.
 * ---------------------------------------------------------------------- */
#define DC_STATIC_MAX_BATCH 1048576
dc_status dc_schedule_batch_static(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                                   const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                                   uint32_t *bits, int32_t *nseg, int32_t *status,
                                   cudaStream_t stream);

/* Static description of a status code. Never NULL. */
const char *dc_status_string(dc_status s);

/* ------------------------------------------------------------------------
 * dc_time_next_pass -- measurement support, not part of the method. The next
 * dc_schedule_forward_batch, dc_schedule_backward_batch or
 * dc_schedule_batch_static call made by the calling thread records `start` on
 * its stream right before it launches its first pass over the batch (the
 * dense, looped or deep-chain kernel, all of that pass's launches) and `stop`
 * right after them, before its work-list pass; cudaEventElapsedTime(start,
 * stop) is then that pass's time on the GPU. start, stop: events created by
 * the caller on the current device, both non-NULL (DC_ERR_NULL if only one
 * is); both NULL withdraw a pending request. The request belongs to the
 * calling thread and is used up by its next schedule call, whether that call
 * succeeds or not; no other call consumes it. This is the one state the
 * library keeps between calls.
 * ---------------------------------------------------------------------- */
dc_status dc_time_next_pass(cudaEvent_t start, cudaEvent_t stop);

/* ------------------------------------------------------------------------
 * dc_roof_int_probe -- measurement support, not part of the method: a
 * register-only loop of the DP's per-transition integer operations on
 * `blocks` x `threads` threads, `iters` iterations of 8 transitions each.
 * Variant 0: the 32-bit passes' shifted form (one 32-bit add-then-max per
 * candidate, one 3-input min per two candidates); variant 1: the 64-bit
 * passes' max, subtract, min. Time it with events on `stream`; it performs
 * blocks*threads*iters*8 transitions. sink: device, blocks*threads uint32.
 * ---------------------------------------------------------------------- */
dc_status dc_roof_int_probe(int32_t variant, int32_t blocks, int32_t threads, int64_t iters,
                            uint32_t *sink, cudaStream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* DYNACOMM_H */
