/*
 * DynaComm CPU oracle: TEST INFRASTRUCTURE, not part of the product.
 * See dynacomm_oracle.h for what each function follows in the paper.
 *
 * Written to be checked by eye against the paper, not to be fast: each DP is
 * its recurrence (Eq. 8, Eq. 9) evaluated cell by cell over every candidate
 * split, with the choice among equal optima stated as a property, and every
 * sum is a prefix-sum difference (Sec. IV-B4, "partial accumulations").
 */
#include "dynacomm_oracle.h"

#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

#define INF INT64_MAX /* brute force: no decision seen yet */

static int64_t max64(int64_t a, int64_t b) { return a > b ? a : b; }

/* P[m] = sum of v over layers 1..m (v holds layer l at index l-1). */
static void prefix_first(int32_t L, const int64_t *v, int64_t *P)
{
    P[0] = 0;
    for (int32_t m = 1; m <= L; m++) P[m] = P[m - 1] + v[m - 1];
}

/* S[m] = sum of v over the last m layers, L-m+1..L (backward processing order). */
static void prefix_last(int32_t L, const int64_t *v, int64_t *S)
{
    S[0] = 0;
    for (int32_t m = 1; m <= L; m++) S[m] = S[m - 1] + v[L - m];
}

/* ------------------------------------------------------------------------
 * The two dynamic programs of Sec. IV-B, written from their recurrences.
 *
 * Take the layers in the order a direction handles them ("processing order":
 * the forward pull starts with layer 1; the backward push starts with layer L,
 * which is why Eq. 9 speaks of the LAST m layers). Processed layer j is layer j
 * forward and layer L+1-j backward. C(m) and T(m) are the compute and transfer
 * costs summed over the first m processed layers (prefix sums, Sec. IV-B4).
 * X(m, n) is the least finishing time of the first m processed layers when
 * their transfer is cut into exactly n segments, the last one holding
 * processed layers k+1..m:
 *
 *   forward,  Eq. 8:  X(m, n) = min_k max(X(k, n-1), n*dt + T(m)) + C(m) - C(k)
 *     (the n-th pull has arrived at n*dt + T(m); layers k+1..m then compute
 *      after the first k layers are done);
 *   backward, Eq. 9:  X(m, n) = min_k max(X(k, n-1), C(m)) + dt + T(m) - T(k)
 *     (the n-th push waits for the backward compute of its layers and for the
 *      previous push, then carries dt plus the gradients of layers k+1..m).
 *
 * X(0, 0) = 0 and X(k, n-1) exists only when 0 layers are cut into 0 segments
 * or 1 <= n-1 <= k; that is reading R1 (the paper's +infinity entries never
 * win, so they are simply not candidates).
 *
 * Which of several optima is returned is fixed by the paper's algorithms
 * (reading R3), and stated here as properties:
 *   - Path(m, n) is the SMALLEST k attaining the minimum (their strict
 *     improvement test keeps the first minimiser as k grows);
 *   - the segment count s is the SMALLEST n attaining min_n X(L, n);
 *   - the decision is read from state (L, s) by stepping (m, n) ->
 *     (Path(m, n), n-1) down to (0, 0); every k reached with 1 <= k <= L-1
 *     enables the position after processed layer k: p_k forward (a new pull
 *     from layer k+1), g_k backward (a new push after the last k layers,
 *     between layers L-k and L-k+1; reading R4, which Algorithm 4's index
 *     conversion expresses).
 * Storage: X and Path are (L+1) x (L+1), column n contiguous (n*(L+1) + m).
 * ---------------------------------------------------------------------- */

/* can the first k processed layers be cut into exactly n segments? */
static int split_exists(int32_t k, int32_t n) { return n == 0 ? k == 0 : (n >= 1 && n <= k); }

static int64_t segment_end(int32_t dir, int64_t before, int32_t m, int32_t n, int32_t k,
                           const int64_t *C, const int64_t *T, int64_t dt)
{
    if (dir == 0) /* Eq. 8 */
        return max64(before, (int64_t)n * dt + T[m]) + (C[m] - C[k]);
    return max64(before, C[m]) + dt + (T[m] - T[k]); /* Eq. 9 */
}

/* comp/xfer hold layer l at index l-1 (l = 1..L), in layer order. Writes the
 * decision d[0..L] (entries 1..L-1 used) and *nseg; returns min_n X(L, n). */
static int64_t solve_dp(int32_t dir, int32_t L, const int64_t *comp, const int64_t *xfer,
                        int64_t dt, uint8_t *d, int32_t *nseg)
{
    const size_t W = (size_t)L + 1;
    int64_t *X = (int64_t *)malloc(W * W * sizeof(int64_t));
    int32_t *Path = (int32_t *)malloc(W * W * sizeof(int32_t));
    int64_t *C = (int64_t *)malloc(W * sizeof(int64_t));
    int64_t *T = (int64_t *)malloc(W * sizeof(int64_t));
    if (dir == 0) {
        prefix_first(L, comp, C);
        prefix_first(L, xfer, T);
    } else {
        prefix_last(L, comp, C);
        prefix_last(L, xfer, T);
    }
    X[0] = 0; /* X(0, 0) */
    for (int32_t n = 1; n <= L; n++)      /* column by column: X(., n) needs X(., n-1) */
        for (int32_t m = n; m <= L; m++) { /* cells that exist: n <= m */
            int64_t best = 0;
            int32_t arg = -1;
            for (int32_t k = n - 1; k <= m - 1; k++) {
                if (!split_exists(k, n - 1)) continue;
                int64_t c = segment_end(dir, X[(size_t)(n - 1) * W + (size_t)k], m, n, k, C, T, dt);
                if (arg < 0 || c < best) { /* ties keep the smaller k */
                    best = c;
                    arg = k;
                }
            }
            X[(size_t)n * W + (size_t)m] = best;
            Path[(size_t)n * W + (size_t)m] = arg;
        }
    int32_t s = 1;
    for (int32_t n = 2; n <= L; n++) /* ties keep the smaller n */
        if (X[(size_t)n * W + (size_t)L] < X[(size_t)s * W + (size_t)L]) s = n;
    const int64_t opt = X[(size_t)s * W + (size_t)L];
    memset(d, 0, W);
    for (int32_t m = L, n = s; n > 0; n--) {
        const int32_t k = Path[(size_t)n * W + (size_t)m];
        if (k >= 1 && k <= L - 1) d[k] = 1;
        m = k;
    }
    *nseg = s;
    free(X);
    free(Path);
    free(C);
    free(T);
    return opt;
}

/* Forward (Eq. 8, the problem of Algorithm 3): comp = fc, xfer = pt. */
int64_t orc_dp_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt,
                       uint8_t *p, int32_t *nseg)
{
    return solve_dp(0, L, fc, pt, dt, p, nseg);
}

/* Backward (Eq. 9, the problem of Algorithm 4): comp = bc, xfer = gt. */
int64_t orc_dp_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt,
                        uint8_t *g, int32_t *nseg)
{
    return solve_dp(1, L, bc, gt, dt, g, nseg);
}

/* ------------------------------------------------------------------------
 * f_m (Sec. III-B), one direction, as an event replay of Eq. 1-7.
 *
 * Forward: the transmissions are serialised on the link in layer order (Eq. 4);
 * the transmission that starts at layer l carries layers l..e and costs
 * dt + sum pt over them; layer l computes after its parameters have arrived
 * (Eq. 1) and after layer l-1 has computed (Eq. 5). Returns ed(fc_L).
 * ---------------------------------------------------------------------- */
int64_t orc_replay_forward(int32_t L, const int64_t *pt, const int64_t *fc, int64_t dt,
                           const uint8_t *p)
{
    int64_t link_free = 0, comp_free = 0, arrive = 0;
    for (int32_t l = 1; l <= L; l++) {
        if (l == 1 || p[l - 1]) { /* a new pull starts with layer l */
            int32_t e = l;
            while (e < L && !p[e]) e++;
            int64_t xfer = dt;
            for (int32_t i = l; i <= e; i++) xfer += pt[i - 1];
            link_free += xfer;
            arrive = link_free;
        }
        int64_t start = max64(comp_free, arrive);
        comp_free = start + fc[l - 1];
    }
    return comp_free;
}

/* Backward: layers compute from L down to 1 back to back from time 0 (Eq. 6);
 * the push of a segment starts after the backward compute of all its layers
 * (Eq. 2) and after the previous push (Eq. 7). g_r = 1 ends a segment after the
 * last r layers. Returns ed(gt_1). */
int64_t orc_replay_backward(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt,
                            const uint8_t *g)
{
    int64_t comp = 0, link = 0, seg_xfer = 0;
    for (int32_t r = 1; r <= L; r++) {
        int32_t l = L + 1 - r; /* r-th layer in backward order */
        comp += bc[l - 1];
        seg_xfer += gt[l - 1];
        if (r == L || g[r]) {
            link = max64(link, comp) + dt + seg_xfer;
            seg_xfer = 0;
        }
    }
    return link;
}

/* ------------------------------------------------------------------------
 * Brute force over the 0-1 program of Sec. III-B.
 * ---------------------------------------------------------------------- */
static int64_t replay_dir(int32_t dir, int32_t L, const int64_t *comp, const int64_t *xfer,
                          int64_t dt, const uint8_t *d)
{
    return dir == 0 ? orc_replay_forward(L, xfer, comp, dt, d)
                    : orc_replay_backward(L, comp, xfer, dt, d);
}

static void mask_to_decision(int32_t L, uint64_t mask, uint8_t *d, int32_t *nseg)
{
    int32_t s = 1;
    d[0] = 0;
    d[L] = 0;
    for (int32_t l = 1; l <= L - 1; l++) {
        d[l] = (uint8_t)((mask >> (l - 1)) & 1u);
        s += d[l];
    }
    *nseg = s;
}

int64_t orc_brute(int32_t dir, int32_t L, const int64_t *comp, const int64_t *xfer,
                  int64_t dt, int32_t *min_nseg, int64_t *opt_table)
{
    uint8_t d[32];
    if (L < 1 || L > 24) return -1;
    int64_t best = INF;
    int32_t best_s = 0;
    for (uint64_t mask = 0; mask < (1ull << (L - 1)); mask++) {
        int32_t s;
        mask_to_decision(L, mask, d, &s);
        int64_t v = replay_dir(dir, L, comp, xfer, dt, d);
        if (v < best || (v == best && s < best_s)) {
            best = v;
            best_s = s;
        }
    }
    *min_nseg = best_s;
    if (opt_table) {
        for (int32_t i = 0; i < (L + 1) * (L + 1); i++) opt_table[i] = INF;
        for (int32_t m = 1; m <= L; m++) {
            /* sub-problem: first m layers (forward) / last m layers (backward) */
            const int64_t *c = dir == 0 ? comp : comp + (L - m);
            const int64_t *x = dir == 0 ? xfer : xfer + (L - m);
            for (uint64_t mask = 0; mask < (1ull << (m - 1)); mask++) {
                int32_t s;
                mask_to_decision(m, mask, d, &s);
                int64_t v = replay_dir(dir, m, c, x, dt, d);
                int64_t *slot = &opt_table[m * (L + 1) + s];
                if (v < *slot) *slot = v;
            }
        }
    }
    return best;
}

/* One-dimensional backward recurrence: Eq. 9 with the segment count dropped. */
int64_t orc_dp_backward_1d(int32_t L, const int64_t *bc, const int64_t *gt, int64_t dt)
{
    const size_t W = (size_t)L + 1;
    int64_t *X = (int64_t *)malloc(W * sizeof(int64_t));
    int64_t *SBC = (int64_t *)malloc(W * sizeof(int64_t));
    int64_t *SGT = (int64_t *)malloc(W * sizeof(int64_t));
    prefix_last(L, bc, SBC);
    prefix_last(L, gt, SGT);
    X[0] = 0;
    for (int32_t m = 1; m <= L; m++) {
        X[m] = INF;
        for (int32_t k = 0; k < m; k++) {
            int64_t c = max64(X[k], SBC[m]) + dt + (SGT[m] - SGT[k]);
            if (c < X[m]) X[m] = c;
        }
    }
    int64_t r = X[L];
    free(X);
    free(SBC);
    free(SGT);
    return r;
}

/* ------------------------------------------------------------------------
 * Batches: per-instance input checks, then Algorithm 3 / 4.
 * ---------------------------------------------------------------------- */
static int32_t instance_status(int32_t L, const int64_t *comp, const int64_t *xfer, int64_t dt)
{
    if (dt < 0) return ORC_NEGATIVE;
    for (int32_t l = 0; l < L; l++)
        if (comp[l] < 0 || xfer[l] < 0) return ORC_NEGATIVE;
    unsigned __int128 total = (unsigned __int128)(uint64_t)L * (uint64_t)dt;
    for (int32_t l = 0; l < L; l++) total += (uint64_t)comp[l] + (unsigned __int128)(uint64_t)xfer[l];
    if (total >= ((unsigned __int128)1 << 52)) return ORC_RANGE;
    return ORC_OK;
}

typedef struct {
    int32_t dir, L, W;
    int64_t lo, hi;
    const int64_t *comp, *xfer, *dt;
    int64_t *makespan;
    uint32_t *bits;
    int32_t *nseg, *status;
    const uint32_t *in_bits;
} batch_job;

static void *schedule_range(void *arg)
{
    batch_job *j = (batch_job *)arg;
    uint8_t *d = (uint8_t *)malloc((size_t)j->L + 1);
    for (int64_t i = j->lo; i < j->hi; i++) {
        const int64_t *c = j->comp + i * j->L, *x = j->xfer + i * j->L;
        uint32_t *w = j->bits + i * j->W;
        for (int32_t q = 0; q < j->W; q++) w[q] = 0;
        int32_t st = instance_status(j->L, c, x, j->dt[i]);
        j->status[i] = st;
        if (st != ORC_OK) {
            j->makespan[i] = -(int64_t)st;
            j->nseg[i] = 0;
            continue;
        }
        int32_t s;
        int64_t v = j->dir == 0 ? orc_dp_forward(j->L, x, c, j->dt[i], d, &s)
                                : orc_dp_backward(j->L, c, x, j->dt[i], d, &s);
        j->makespan[i] = v;
        j->nseg[i] = s;
        for (int32_t l = 1; l <= j->L - 1; l++)
            if (d[l]) w[(l - 1) / 32] |= 1u << ((l - 1) % 32);
    }
    free(d);
    return NULL;
}

static void *replay_range(void *arg)
{
    batch_job *j = (batch_job *)arg;
    uint8_t *d = (uint8_t *)malloc((size_t)j->L + 1);
    for (int64_t i = j->lo; i < j->hi; i++) {
        const int64_t *c = j->comp + i * j->L, *x = j->xfer + i * j->L;
        const uint32_t *w = j->in_bits + i * j->W;
        int32_t st = instance_status(j->L, c, x, j->dt[i]);
        if (st != ORC_OK) {
            j->makespan[i] = -(int64_t)st;
            continue;
        }
        d[0] = 0;
        d[j->L] = 0;
        for (int32_t l = 1; l <= j->L - 1; l++) d[l] = (uint8_t)((w[(l - 1) / 32] >> ((l - 1) % 32)) & 1u);
        j->makespan[i] = replay_dir(j->dir, j->L, c, x, j->dt[i], d);
    }
    free(d);
    return NULL;
}

static void run_split(batch_job base, int64_t batch, int32_t nthreads, void *(*fn)(void *))
{
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    if ((int64_t)nthreads > batch) nthreads = batch > 0 ? (int32_t)batch : 1;
    pthread_t th[256];
    batch_job jobs[256];
    for (int32_t t = 0; t < nthreads; t++) {
        jobs[t] = base;
        jobs[t].lo = batch * t / nthreads;
        jobs[t].hi = batch * (t + 1) / nthreads;
    }
    if (nthreads == 1) {
        fn(&jobs[0]);
        return;
    }
    for (int32_t t = 0; t < nthreads; t++) pthread_create(&th[t], NULL, fn, &jobs[t]);
    for (int32_t t = 0; t < nthreads; t++) pthread_join(th[t], NULL);
}

static void *greedy_range(void *arg)
{
    batch_job *j = (batch_job *)arg;
    uint8_t *d = (uint8_t *)malloc((size_t)j->L + 1);
    for (int64_t i = j->lo; i < j->hi; i++) {
        const int64_t *c = j->comp + i * j->L, *x = j->xfer + i * j->L;
        uint32_t *w = j->bits + i * j->W;
        for (int32_t q = 0; q < j->W; q++) w[q] = 0;
        int32_t st = instance_status(j->L, c, x, j->dt[i]);
        if (st != ORC_OK) {
            j->makespan[i] = -(int64_t)st;
            continue;
        }
        if (j->dir == 0)
            orc_greedy_forward(j->L, x, c, j->dt[i], d);
        else
            orc_greedy_backward(j->L, c, x, j->dt[i], d);
        d[0] = 0;
        d[j->L] = 0;
        for (int32_t l = 1; l <= j->L - 1; l++)
            if (d[l]) w[(l - 1) / 32] |= 1u << ((l - 1) % 32);
        j->makespan[i] = replay_dir(j->dir, j->L, c, x, j->dt[i], d);
    }
    free(d);
    return NULL;
}

void orc_schedule_batch(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                        const int64_t *xfer, const int64_t *dt, int64_t *makespan,
                        uint32_t *bits, int32_t *nseg, int32_t *status, int32_t nthreads)
{
    batch_job b;
    memset(&b, 0, sizeof b);
    b.dir = dir;
    b.L = L;
    b.W = (L - 1 + 31) / 32;
    b.comp = comp;
    b.xfer = xfer;
    b.dt = dt;
    b.makespan = makespan;
    b.bits = bits;
    b.nseg = nseg;
    b.status = status;
    run_split(b, batch, nthreads, schedule_range);
}

void orc_replay_batch(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                      const int64_t *xfer, const int64_t *dt, const uint32_t *bits,
                      int64_t *makespan, int32_t nthreads)
{
    batch_job b;
    memset(&b, 0, sizeof b);
    b.dir = dir;
    b.L = L;
    b.W = (L - 1 + 31) / 32;
    b.comp = comp;
    b.xfer = xfer;
    b.dt = dt;
    b.makespan = makespan;
    b.in_bits = bits;
    run_split(b, batch, nthreads, replay_range);
}

/* ------------------------------------------------------------------------
 * Synthetic profile generator (stands in for the real-time profiler, Sec. IV-A).
 *
 * Randomness: draw(field, layer) of instance gi is SplitMix64 output number
 * ctr+1 for state `seed`, ctr = gi<<20 | field<<12 | layer, i.e.
 * mix(seed + (ctr+1) * 0x9e3779b97f4a7c15) with the SplitMix64 finaliser.
 * uniform-int [a,b] = a + floor(r * (b-a+1) / 2^64).
 * log-uniform [lo,hi]: knots T(j) = round(lo * exp((j/512) * ln(hi/lo))),
 * T(0) = lo, T(512) = hi; with j = r's top 9 bits and f = its next 32 bits,
 * value = T(j) + floor((T(j+1) - T(j)) * f / 2^32).
 * Costs (integer microseconds): fc = ceil(FLOPs / rate), bc = ceil(mult * FLOPs
 * / rate), pt = gt = ceil(bits_per_param * 1000 * params / bw) with rate in
 * FLOP/us and bw in kbit/s.
 * ---------------------------------------------------------------------- */
enum { FIELD_RATE = 0, FIELD_BW = 1, FIELD_DT = 2, FIELD_PARAMS = 3, FIELD_FLOPS = 4 };

uint64_t orc_splitmix64(uint64_t seed, uint64_t ctr)
{
    uint64_t z = seed + (ctr + 1) * 0x9e3779b97f4a7c15ull;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

static uint64_t draw(uint64_t seed, int64_t gi, int32_t field, int32_t layer)
{
    uint64_t ctr = ((uint64_t)gi << 20) | ((uint64_t)field << 12) | (uint64_t)layer;
    return orc_splitmix64(seed, ctr);
}

int64_t orc_uniform_int(int64_t lo, int64_t hi, uint64_t r)
{
    uint64_t span = (uint64_t)(hi - lo) + 1u;
    return lo + (int64_t)(((unsigned __int128)r * span) >> 64);
}

static int64_t log_knot(int64_t lo, int64_t hi, int32_t j)
{
    if (j <= 0) return lo;
    if (j >= 512) return hi;
    double x = (double)j / 512.0;
    double y = log((double)hi / (double)lo);
    return (int64_t)llround((double)lo * exp(x * y));
}

int64_t orc_loguniform(int64_t lo, int64_t hi, uint64_t r)
{
    int32_t j = (int32_t)(r >> 55);
    uint64_t f = (r >> 23) & 0xffffffffull;
    int64_t t0 = log_knot(lo, hi, j), t1 = log_knot(lo, hi, j + 1);
    return t0 + (int64_t)(((uint64_t)(t1 - t0) * f) >> 32);
}

static int64_t dist_draw(int32_t dist, int64_t lo, int64_t hi, uint64_t r)
{
    return dist == ORC_DIST_LOGUNIFORM ? orc_loguniform(lo, hi, r) : orc_uniform_int(lo, hi, r);
}

void orc_instance_draws(const orc_profile_cfg *cfg, int64_t i, int64_t *rate, int64_t *bw,
                        int64_t *dt)
{
    int64_t gi = cfg->inst0 + i;
    *rate = dist_draw(cfg->rate_dist, cfg->rate_lo, cfg->rate_hi, draw(cfg->seed, gi, FIELD_RATE, 0));
    *bw = dist_draw(cfg->bw_dist, cfg->bw_lo, cfg->bw_hi, draw(cfg->seed, gi, FIELD_BW, 0));
    *dt = orc_uniform_int(cfg->dt_lo, cfg->dt_hi, draw(cfg->seed, gi, FIELD_DT, 0));
}

int64_t orc_layer_draw(const orc_profile_cfg *cfg, int64_t i, int32_t field, int32_t l)
{
    int64_t gi = cfg->inst0 + i;
    int64_t lo = field == FIELD_PARAMS ? cfg->params_lo : cfg->flops_lo;
    int64_t hi = field == FIELD_PARAMS ? cfg->params_hi : cfg->flops_hi;
    if (cfg->layer_mode == ORC_LAYERS_FIXED)
        return field == FIELD_PARAMS ? cfg->fixed_params[l] : cfg->fixed_flops[l];
    int32_t dist = cfg->layer_mode == ORC_LAYERS_LOGUNIFORM ? ORC_DIST_LOGUNIFORM : ORC_DIST_UNIFORM;
    return dist_draw(dist, lo, hi, draw(cfg->seed, gi, field, l));
}

static int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

static int range_ok(int64_t lo, int64_t hi, int64_t min_lo, int64_t max_hi)
{
    return lo >= min_lo && lo <= hi && hi <= max_hi;
}

int32_t orc_profile_gen(const orc_profile_cfg *cfg, int64_t *fc, int64_t *pt, int64_t *bc,
                        int64_t *gt, int64_t *dt)
{
    const int64_t CAP = (int64_t)1 << 40, RCAP = ((int64_t)1 << 31) - 1;
    const int32_t L = cfg->L;
    if (L < 1 || L > 4096 || cfg->batch < 0 || cfg->inst0 < 0) return -1;
    if ((cfg->inst0 + cfg->batch) > ((int64_t)1 << 44)) return -1;
    if (cfg->bwd_flops_mult < 1 || cfg->bwd_flops_mult > 16) return -1;
    if (cfg->bits_per_param < 1 || cfg->bits_per_param > 64) return -1;
    if (!range_ok(cfg->rate_lo, cfg->rate_hi, 1, RCAP) || !range_ok(cfg->bw_lo, cfg->bw_hi, 1, RCAP))
        return -1;
    if (!range_ok(cfg->dt_lo, cfg->dt_hi, 0, CAP)) return -1;
    if (cfg->rate_dist < 0 || cfg->rate_dist > 1 || cfg->bw_dist < 0 || cfg->bw_dist > 1) return -1;
    if (cfg->layer_mode == ORC_LAYERS_FIXED) {
        if (L > 1024 || !cfg->fixed_params || !cfg->fixed_flops) return -1;
        for (int32_t l = 0; l < L; l++)
            if (!range_ok(cfg->fixed_params[l], cfg->fixed_params[l], 0, CAP) ||
                !range_ok(cfg->fixed_flops[l], cfg->fixed_flops[l], 0, CAP))
                return -1;
    } else if (cfg->layer_mode == ORC_LAYERS_UNIFORM || cfg->layer_mode == ORC_LAYERS_LOGUNIFORM) {
        int64_t min_lo = cfg->layer_mode == ORC_LAYERS_LOGUNIFORM ? 1 : 0;
        if (!range_ok(cfg->params_lo, cfg->params_hi, min_lo, CAP) ||
            !range_ok(cfg->flops_lo, cfg->flops_hi, min_lo, CAP))
            return -1;
    } else {
        return -1;
    }
    for (int64_t i = 0; i < cfg->batch; i++) {
        int64_t rate, bw, d;
        orc_instance_draws(cfg, i, &rate, &bw, &d);
        dt[i] = d;
        for (int32_t l = 0; l < L; l++) {
            int64_t params = orc_layer_draw(cfg, i, FIELD_PARAMS, l);
            int64_t flops = orc_layer_draw(cfg, i, FIELD_FLOPS, l);
            fc[i * L + l] = ceil_div(flops, rate);
            bc[i * L + l] = ceil_div((int64_t)cfg->bwd_flops_mult * flops, rate);
            pt[i * L + l] = ceil_div((int64_t)cfg->bits_per_param * 1000 * params, bw);
            gt[i * L + l] = pt[i * L + l];
        }
    }
    return 0;
}

void orc_greedy_batch(int32_t dir, int64_t batch, int32_t L, const int64_t *comp,
                      const int64_t *xfer, const int64_t *dt, uint32_t *bits, int64_t *makespan,
                      int32_t nthreads)
{
    batch_job b;
    memset(&b, 0, sizeof b);
    b.dir = dir;
    b.L = L;
    b.W = (L - 1 + 31) / 32;
    b.comp = comp;
    b.xfer = xfer;
    b.dt = dt;
    b.makespan = makespan;
    b.bits = bits;
    run_split(b, batch, nthreads, greedy_range);
}
