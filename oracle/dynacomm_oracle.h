/*
 * DynaComm CPU oracle: TEST INFRASTRUCTURE, not part of the product.
 *
 * A plain, slow, single-threaded C statement of what the DynaComm scheduling
 * path computes (Cai et al., "DynaComm: Accelerating Distributed CNN Training
 * between Edges and Clouds through Dynamic Communication Scheduling"):
 *   - the forward DP, Eq. 8 evaluated cell by cell (the problem Algorithm 3 solves),
 *   - the backward DP, Eq. 9 evaluated cell by cell (the problem of Algorithm 4),
 *     both returning the optimum Algorithms 3/4 return among equal ones: the
 *     lowest split index per cell, the lowest segment count overall,
 *   - the cost measurement f_m of Sec. III-B, written as an event replay of the
 *     partial orders Eq. 1-7,
 *   - brute force over all 2^(L-1) decisions (Sec. III-B, the O(L 2^L) search),
 *   - an O(L^2) one-dimensional backward DP used as an independent value check,
 *   - the seeded synthetic profile generator that stands in for the real-time
 *     profiler of Sec. IV-A,
 *   - the paper's competing greedy schedulers, Algorithm 1 (forward) and
 *     Algorithm 2 (backward), in greedy_oracle.c.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may load
 * this library. It shares no code, header or table with the CUDA library.
 *
 * Conventions (shared with the CUDA library by contract, not by code):
 *   times are int64 microseconds; arrays are per layer, layer l (1-based in the
 *   paper) at index l-1; a decision vector is p[0..L] / g[0..L] with entries
 *   1..L-1 used; packed decision bits put p_l (or g_l) at bit (l-1)%32 of word
 *   (l-1)/32, W = ceil((L-1)/32) words per instance.
 */
#ifndef DYNACOMM_ORACLE_H
#define DYNACOMM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* per-instance status codes (same numeric contract as the library) */
#define ORC_OK 0
#define ORC_NEGATIVE 3
#define ORC_RANGE 4

/* ---- one instance ---------------------------------------------------- */

/* Algorithm 3 / Eq. 8. pt, fc: L entries. Writes p[0..L] (p[l] in {0,1} for
 * 1 <= l <= L-1) and *nseg = number of enabled positions including the start.
 * Returns T_forward. */
int64_t orc_dp_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt,
                       uint8_t *p, int32_t *nseg);

/* Algorithm 4 / Eq. 9. bc, gt: L entries (layer order 1..L). Writes g[0..L]. */
int64_t orc_dp_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt,
                        uint8_t *g, int32_t *nseg);

/* f_m for one direction: replays decision p (forward) or g (backward). */
int64_t orc_replay_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt,
                           const uint8_t *p);
int64_t orc_replay_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt,
                            const uint8_t *g);

/* Brute force over all 2^(L-1) decisions (L <= 24). dir 0 = forward (comp = fc,
 * xfer = pt), 1 = backward (comp = bc, xfer = gt). Returns the optimum and the
 * fewest segments among optimal decisions in *min_nseg. If opt_table is not
 * NULL it receives opt(m, n) for 1 <= n <= m <= L at opt_table[m*(L+1)+n]: the
 * best replay value over decisions of the first m layers (forward) or last m
 * layers (backward) with exactly n segments. */
int64_t orc_brute(int32_t dir, int32_t L, const int64_t *comp, const int64_t *xfer,
                  int64_t dt, int32_t *min_nseg, int64_t *opt_table);

/* min over n of Eq. 9's B[L][n], by the one-dimensional recurrence that drops n
 * (Eq. 9's cost does not depend on n). */
int64_t orc_dp_backward_1d(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt);

/* ---- batches (instances are independent; nthreads >= 1 splits them) ---- */

/* dir 0: comp = fc, xfer = pt (Alg. 3). dir 1: comp = bc, xfer = gt (Alg. 4).
 * comp, xfer: [batch][L]; dt: [batch]. Outputs: makespan [batch] (-status on a
 * failed instance), bits [batch][W], nseg [batch], status [batch]. */
void orc_schedule_batch(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                        uint32_t *bits, int32_t *nseg, int32_t *status, int32_t nthreads);

/* f_m over a batch for the packed decisions bits [batch][W]. */
void orc_replay_batch(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                      const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                      int64_t *makespan, int32_t nthreads);

/* ---- the paper's competing greedy schedulers (greedy_oracle.c) -------- */

/* Algorithm 1 (iBatch, forward): writes p[0..L]. */
void orc_greedy_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt, uint8_t *p);
/* Algorithm 2 (iPart, backward): writes g[0..L], g[r] = break after the last r layers. */
void orc_greedy_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt, uint8_t *g);
/* Either over a batch: packed decisions bits [batch][W] and their f_m makespan
 * (-status for a failed instance, with zero bits). dir 0: comp = fc, xfer = pt;
 * dir 1: comp = bc, xfer = gt. */
void orc_greedy_batch(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                      const int64_t *xfer, const int64_t *dt, uint32_t *bits, int64_t *makespan,
                      int32_t nthreads);

/* ---- synthetic profile generator (stand-in for Sec. IV-A's profiler) ---- */

#define ORC_LAYERS_FIXED 0
#define ORC_LAYERS_UNIFORM 1
#define ORC_LAYERS_LOGUNIFORM 2
#define ORC_DIST_UNIFORM 0
#define ORC_DIST_LOGUNIFORM 1

typedef struct {
    int32_t L;
    int32_t layer_mode;
    int64_t batch;
    int64_t inst0;
    uint64_t seed;
    const int64_t *fixed_params;
    const int64_t *fixed_flops;
    int64_t params_lo, params_hi, flops_lo, flops_hi;
    int32_t rate_dist, bw_dist;
    int64_t rate_lo, rate_hi;
    int64_t bw_lo, bw_hi;
    int64_t dt_lo, dt_hi;
    int32_t bwd_flops_mult;
    int32_t bits_per_param;
} orc_profile_cfg;

/* SplitMix64 output number ctr+1 for state `seed` (Steele, Lea, Flood 2014). */
uint64_t orc_splitmix64(uint64_t seed, uint64_t ctr);

/* Per-instance draws (exposed so tests can check the ceilings). */
void orc_instance_draws(const orc_profile_cfg *cfg, int64_t i, int64_t *rate, int64_t *bw,
                        int64_t *dt);
int64_t orc_layer_draw(const orc_profile_cfg *cfg, int64_t i, int32_t field, int32_t l);
int64_t orc_loguniform(int64_t lo, int64_t hi, uint64_t r);
int64_t orc_uniform_int(int64_t lo, int64_t hi, uint64_t r);

/* fc, pt, bc, gt: [batch][L]; dt: [batch]. Returns 0, or -1 on a bad config. */
int32_t orc_profile_gen(const orc_profile_cfg *cfg, int64_t *fc, int64_t *pt, int64_t *bc,
                        int64_t *gt, int64_t *dt);

#ifdef __cplusplus
}
#endif
#endif
