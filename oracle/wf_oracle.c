/*
 * CPU ORACLE for batched plan evaluation -- TEST INFRASTRUCTURE ONLY.
 *
 * Only the tests, the smoke check and the benchmark's CPU-baseline leg may
 * load this file's library.  It shares no code, header, table or helper with
 * the GPU library; the two meet only at the generated input arrays.
 *
 * What it computes (paper Sections 3.3-3.5).  A plan for one window of the
 * activation DAG fixes a device per activation (the x variables of Eq. 9), a
 * dispatch sequence that orients every resource conflict (z of Eq. 10), and
 * per-activation fusion / prefetch / retain bits (the lifecycle choices h of
 * Eq. 5).  The oracle plays the plan forward as a plain discrete-event list
 * schedule, one dispatch position at a time:
 *
 *   - fused chains (Eq. 3) run as one unit under one grant, with admission
 *     memory = weights + the largest KV need on the chain and run time = the
 *     sum of the members' run times (Eq. 4);
 *   - release r = max(session arrival, finish of every graph predecessor)
 *     (Eq. 2, Eq. 7);
 *   - a unit starts after its release and after the previous unit on its
 *     device (Eq. 7, Eq. 10), and after its model is loaded when it is not
 *     resident (Eq. 5, Eq. 9: the load sits on the consumer's device);
 *   - resident weights plus the unit's KV admission never exceed the device
 *     capacity (Eq. 8, Eq. 11); least-recently-used models are reclaimed
 *     until they fit (the LRU fallback of Section 3.5);
 *   - a prefetched load may start as soon as the device is free and the
 *     session has arrived, before the unit's release (Eq. 5, Section 3.5);
 *   - makespan = last finish - first arrival, p95 = nearest-rank 95th
 *     percentile of per-session completion latency (Section 4.2), GPU time =
 *     time each device holds at least one model: loading, generating or idle
 *     resident (Section 4.3);
 *   - beside them, the window terms of the ranking key of Eq. 12: timely
 *     prefetches and the lifecycle overhead (ready-work loading delay plus
 *     reloads after reclamation), see orc_eval_phi_batch;
 *   - with a replica batch limit B_q (Section 3.5, batch >= 1), units of a
 *     device's current replica run up to B_q at once and Eq. 11 sums the KV
 *     needs of every running unit, see simulate_batched.
 *
 * Every time is an int64 microsecond count and every memory an int32 MiB
 * count, so results are exact.  Points the paper leaves open are read as
 * follows and restated where they apply: devices start empty and run one
 * unit at a time in dispatch order; reclamation happens when a unit is
 * admitted and costs no time; a fused chain runs at its head's position;
 * an ineligible fuse bit is ignored; an invalid plan scores INT64_MAX.
 *
 * Parity pins: every function here is pinned by the CPU test suite
 * (hand-worked windows, closed forms, textbook-routine reductions,
 * invariants replayed from the trace, brute force).  The stochastic
 * multiplier draw is pinned by the published SplitMix64 vector, by three
 * multipliers worked by hand from that vector and the table formulas (each
 * nested hash input chosen to be a published generator state), and by the
 * sample statistics of the multipliers.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_NONE INT64_MIN
#define ORC_INF INT64_MAX

typedef struct {
    int32_t N, D, M, W;
    const int32_t *pred_off;   /* [N+1] */
    const int32_t *pred_idx;   /* [E]   */
    const uint8_t *model;      /* [N]   */
    const int32_t *session;    /* [N]   */
    const int64_t *arrival;    /* [W]   */
    const int32_t *lat;        /* [N][D] run time, us */
    const int32_t *peak;       /* [N][D] peak memory, MiB */
    const int32_t *weight;     /* [M] model weights, MiB */
    const int32_t *load;       /* [M][D] load time, us */
    const int32_t *cap;        /* [D] capacity, MiB */
    int32_t grant;             /* admission overhead per unit, us */
    int32_t S;                 /* latency samples (0 = deterministic) */
    uint64_t seed;
    const int32_t *bm_r, *bm_c, *bm_e;
    int32_t bm_rn, bm_cn, bm_en;
    int32_t reclaim;           /* 0: least recently used first; 1: by next use (see next_use_victim) */
    int32_t batch;             /* replica batch limit B_q (simulate_batched); 0: one unit at a time per device */
} orc_problem;

/* Optional record of one deterministic run, for the invariant checker. */
typedef struct {
    int32_t *unit_head;   /* [N] heads in dispatch order */
    int32_t *n_units;     /* [1] */
    int32_t *head_of;     /* [N] the head of each node's unit */
    int64_t *start;       /* [N] start of each node's execution */
    int64_t *finish;      /* [N] finish c[n] */
    int64_t *rel;         /* [N] release of each head (-1 for chain members) */
    int64_t *load_start;  /* [N] per head, -1 when the model was resident */
    int64_t *load_end;    /* [N] per head, -1 when the model was resident */
    int32_t *kv_adm;      /* [N] per head: KV admission of the unit */
    int32_t *used_after;  /* [N] per head: resident weights after admission */
    uint32_t *evicted;    /* [N] per head: bit m set when model m was reclaimed at admission */
    uint8_t *reclaimed;   /* [N] per head: model unloaded after the unit (retain bit 0) */
    int64_t *occ_start;   /* [N+D] occupancy intervals */
    int64_t *occ_end;
    int32_t *occ_dev;
    int32_t *n_occ;       /* [1] */
    int64_t *adm;         /* [N] per head: admission time (the load start on a miss); NULL: not kept */
} orc_trace;

static int64_t imax64(int64_t a, int64_t b) { return a > b ? a : b; }
static int64_t imin64(int64_t a, int64_t b) { return a < b ? a : b; }

static int bit_of(const uint32_t *row, int32_t n)
{
    return (int)((row[n >> 5] >> (n & 31)) & 1u);
}

static int cmp_i64(const void *a, const void *b)
{
    int64_t x = *(const int64_t *)a, y = *(const int64_t *)b;
    return (x > y) - (x < y);
}

/* Nearest-rank percentile: the ceil(q*n/100)-th smallest value (1-based). */
static int64_t nearest_rank(int64_t *v, int64_t n, int32_t q)
{
    qsort(v, (size_t)n, sizeof(int64_t), cmp_i64);
    int64_t rank = (q * n + 99) / 100;
    if (rank < 1) rank = 1;
    return v[rank - 1];
}

/*
 * Eq. 3: edge (u, v) is fusible when succ(u) = {v}, pred(v) = {u} and both
 * use the same deployment (configuration compatibility collapses into model
 * equality).  fnext[u] = v for such an edge, else -1.
 */
int orc_fusible_next(const orc_problem *pb, int32_t *fnext)
{
    const int32_t N = pb->N;
    int32_t *nsucc = (int32_t *)calloc((size_t)N, sizeof(int32_t));
    int32_t *only = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    if (!nsucc || !only) { free(nsucc); free(only); return -1; }
    for (int32_t v = 0; v < N; ++v)
        for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) {
            int32_t u = pb->pred_idx[e];
            nsucc[u] += 1;
            only[u] = v;
        }
    for (int32_t u = 0; u < N; ++u) {
        fnext[u] = -1;
        if (nsucc[u] != 1) continue;
        int32_t v = only[u];
        int32_t npred_v = pb->pred_off[v + 1] - pb->pred_off[v];
        if (npred_v == 1 && pb->model[u] == pb->model[v]) fnext[u] = v;
    }
    free(nsucc);
    free(only);
    return 0;
}

/*
 * Release forecast, Eq. 2, over the whole window with no contention and no
 * loading: rel[n] = max(arrival of n's session, max over preds v of comp[v]),
 * comp[n] = rel[n] + Lmin[n], where Lmin[n] is the shortest run time of n over
 * the devices whose capacity admits its peak memory (Eq. 8).
 * Returns 0, -1 on allocation failure, -2 if the DAG has a cycle, -3 if a
 * node fits on no device.
 */
int orc_forecast(const orc_problem *pb, int64_t *rel, int64_t *comp)
{
    const int32_t N = pb->N, D = pb->D;
    int32_t *indeg = (int32_t *)calloc((size_t)N, sizeof(int32_t));
    int32_t *queue = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int32_t *soff = (int32_t *)calloc((size_t)N + 1, sizeof(int32_t));
    int32_t *sidx = (int32_t *)malloc(sizeof(int32_t) * (size_t)(pb->pred_off[N] + 1));
    int32_t *fill = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int rc = 0;
    if (!indeg || !queue || !soff || !sidx || !fill) { rc = -1; goto out; }
    for (int32_t v = 0; v < N; ++v) {
        indeg[v] = pb->pred_off[v + 1] - pb->pred_off[v];
        for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) soff[pb->pred_idx[e] + 1] += 1;
    }
    for (int32_t u = 0; u < N; ++u) soff[u + 1] += soff[u];
    for (int32_t u = 0; u < N; ++u) fill[u] = soff[u];
    for (int32_t v = 0; v < N; ++v)
        for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) sidx[fill[pb->pred_idx[e]]++] = v;

    int32_t head = 0, tail = 0;
    for (int32_t v = 0; v < N; ++v) if (indeg[v] == 0) queue[tail++] = v;
    while (head < tail) {
        int32_t n = queue[head++];
        int64_t r = pb->arrival[pb->session[n]];
        for (int32_t e = pb->pred_off[n]; e < pb->pred_off[n + 1]; ++e) r = imax64(r, comp[pb->pred_idx[e]]);
        int64_t lmin = ORC_INF;
        for (int32_t d = 0; d < D; ++d)
            if (pb->peak[(int64_t)n * D + d] <= pb->cap[d]) lmin = imin64(lmin, pb->lat[(int64_t)n * D + d]);
        if (lmin == ORC_INF) { rc = -3; goto out; }
        rel[n] = r;
        comp[n] = r + lmin;
        for (int32_t e = soff[n]; e < soff[n + 1]; ++e)
            if (--indeg[sidx[e]] == 0) queue[tail++] = sidx[e];
    }
    if (tail != N) rc = -2;
out:
    free(indeg); free(queue); free(soff); free(sidx); free(fill);
    return rc;
}

/*
 * Plan validity.  Bit 1: a device index outside [0, D).  Bit 2: a node placed
 * on a device whose capacity is below its peak memory (Eq. 8).  Bit 4: the
 * dispatch sequence is not a permutation of the nodes.  Bit 8 (only examined
 * when bit 4 is clear): some edge u -> v has v dispatched before u, i.e. the
 * resource order would contradict the logical order (Eq. 9, Eq. 10).
 */
int orc_status(const orc_problem *pb, const uint8_t *place, const uint16_t *order, uint32_t *status)
{
    const int32_t N = pb->N, D = pb->D;
    uint32_t st = 0;
    for (int32_t n = 0; n < N; ++n) {
        if (place[n] >= D) st |= 1u;
        else if (pb->peak[(int64_t)n * D + place[n]] > pb->cap[place[n]]) st |= 2u;
    }
    int32_t *pos = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    if (!pos) return -1;
    for (int32_t n = 0; n < N; ++n) pos[n] = -1;
    for (int32_t i = 0; i < N; ++i) {
        int32_t h = order[i];
        if (h >= N || pos[h] >= 0) { st |= 4u; continue; }
        pos[h] = i;
    }
    if (!(st & 4u)) {
        for (int32_t v = 0; v < N; ++v)
            for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e)
                if (pos[pb->pred_idx[e]] > pos[v]) st |= 8u;
    }
    free(pos);
    *status = st;
    return 0;
}

/*
 * One deterministic play of a valid plan with run times L (int64 [N][D]).
 * Writes c[n], per-session completion comp_w[w] = max_{n in w} c[n] - arrival[w],
 * *makespan and *gpu.  Returns 0, -1 on allocation failure, -2 if a unit
 * cannot be admitted even on an empty device (never for a valid plan).
 */
/*
 * Reclamation by next use (the paper's preference order when it reclaims,
 * Section 3.5: redundant copies first, then the model whose next use is
 * farthest relative to its reload cost, least recently used for the rest).
 * Among the models resident on device d other than m, the victim is the
 * first by:
 *   1. resident on another device too (a redundant copy);
 *   2. larger (next use - i) / load[k][d], where next use is the dispatch
 *      position of the next unit on d with model k after position i (none:
 *      infinitely far) and a zero load cost makes the ratio infinite; two
 *      infinite ratios tie;
 *   3. smaller last-use stamp (least recently used).
 * is_head[j] marks the dispatch positions that start a unit.
 */
static int32_t next_use_victim(const orc_problem *pb, const uint8_t *place, const uint16_t *order,
                               const uint8_t *is_head, int32_t i, int32_t d, int32_t m, const int64_t *stamp)
{
    const int32_t N = pb->N, D = pb->D, M = pb->M;
    int32_t best = -1, best_red = 0, best_inf = 0;
    int64_t best_dist = 0, best_cost = 0;
    for (int32_t k = 0; k < M; ++k) {
        if (k == m || stamp[(int64_t)d * M + k] == 0) continue;
        int32_t red = 0;
        for (int32_t e = 0; e < D; ++e)
            if (e != d && stamp[(int64_t)e * M + k] != 0) red = 1;
        int64_t dist = -1;
        for (int32_t j = i + 1; j < N && dist < 0; ++j)
            if (is_head[j] && place[order[j]] == d && pb->model[order[j]] == k) dist = j - i;
        const int64_t cost = pb->load[(int64_t)k * D + d];
        const int inf = dist < 0 || cost == 0;
        int better;
        if (best < 0) better = 1;
        else if (red != best_red) better = red > best_red;
        else if (inf != best_inf) better = inf > best_inf;
        else if (!inf && dist * best_cost != best_dist * cost) better = dist * best_cost > best_dist * cost;
        else better = stamp[(int64_t)d * M + k] < stamp[(int64_t)d * M + best];
        if (better) { best = k; best_red = red; best_inf = inf; best_dist = dist; best_cost = cost; }
    }
    return best;
}

static int simulate(const orc_problem *pb, const int32_t *fnext,
                    const uint8_t *place, const uint16_t *order,
                    const uint32_t *fuse, const uint32_t *prefetch, const uint32_t *retain,
                    const int64_t *L, int64_t *c, int64_t *comp_w,
                    int64_t *makespan, int64_t *gpu_total, orc_trace *tr, int64_t *phi)
{
    const int32_t N = pb->N, D = pb->D, M = pb->M, W = pb->W;
    int64_t *t_free = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int64_t *occ_since = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int64_t *gpu = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int64_t *used = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int32_t *nres = (int32_t *)malloc(sizeof(int32_t) * (size_t)D);
    int64_t *stamp = (int64_t *)malloc(sizeof(int64_t) * (size_t)D * (size_t)M);
    uint8_t *done = (uint8_t *)malloc((size_t)N);
    uint8_t *loaded = (uint8_t *)calloc((size_t)D * (size_t)M, 1);  /* model m was ever resident on d */
    int64_t timely = 0, life = 0;
    int32_t *chain = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    uint8_t *is_head = (uint8_t *)malloc((size_t)N);
    int32_t *fprev = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int rc = 0;
    if (!t_free || !occ_since || !gpu || !used || !nres || !stamp || !done || !chain || !is_head || !fprev ||
        !loaded) {
        rc = -1;
        goto out;
    }
    /* Dispatch positions that start a unit: every node but those that run
     * inside their fusible predecessor's unit (fuse bit set, same device). */
    for (int32_t v = 0; v < N; ++v) fprev[v] = -1;
    for (int32_t u = 0; u < N; ++u)
        if (fnext[u] >= 0) fprev[fnext[u]] = u;
    for (int32_t j = 0; j < N; ++j) {
        const int32_t x = order[j];
        is_head[j] = !(fprev[x] >= 0 && bit_of(fuse, x) && place[x] == place[fprev[x]]);
    }

    /* Initial snapshot: every device idle and empty at t = 0. */
    for (int32_t d = 0; d < D; ++d) {
        t_free[d] = 0; occ_since[d] = ORC_NONE; gpu[d] = 0; used[d] = 0; nres[d] = 0;
        for (int32_t m = 0; m < M; ++m) stamp[(int64_t)d * M + m] = 0;  /* 0 = not resident */
    }
    memset(done, 0, (size_t)N);
    int64_t seq = 0;
    if (tr) { *tr->n_units = 0; *tr->n_occ = 0; }

    for (int32_t i = 0; i < N; ++i) {
        const int32_t h = order[i];
        if (done[h]) continue;  /* already ran inside an earlier chain */

        /* Fused chain (Eq. 3 with the plan's fuse bit and a shared device). */
        int32_t len = 0;
        chain[len++] = h;
        for (;;) {
            int32_t s = fnext[chain[len - 1]];
            if (s < 0 || !bit_of(fuse, s) || place[s] != place[h]) break;
            chain[len++] = s;
        }
        const int32_t last = chain[len - 1];
        const int32_t d = place[h];
        const int32_t m = pb->model[h];
        const int32_t w = pb->session[h];
        int64_t *st = &stamp[(int64_t)d * M];

        /* Release (Eq. 2, Eq. 7): session arrival and every graph predecessor. */
        int64_t rel = pb->arrival[w];
        for (int32_t e = pb->pred_off[h]; e < pb->pred_off[h + 1]; ++e)
            rel = imax64(rel, c[pb->pred_idx[e]]);

        /* Admission memory of the unit (Eq. 4): weights + largest KV on the chain. */
        int64_t kv_adm = 0;
        for (int32_t j = 0; j < len; ++j)
            kv_adm = imax64(kv_adm, (int64_t)pb->peak[(int64_t)chain[j] * D + d] - pb->weight[m]);

        const int hit = st[m] != 0;
        int64_t start, ls = -1, le = -1;
        uint32_t evicted = 0;
        const int64_t need = hit ? kv_adm : pb->weight[m] + kv_adm;
        /* Eq. 11: reclaim least-recently-used models (never the unit's own)
         * until resident weights plus the incoming demand fit the device. */
        while (used[d] + need > pb->cap[d]) {
            int32_t victim = -1;
            if (pb->reclaim) {
                victim = next_use_victim(pb, place, order, is_head, i, d, m, stamp);
            } else {
                for (int32_t k = 0; k < M; ++k)
                    if (k != m && st[k] != 0 && (victim < 0 || st[k] < st[victim])) victim = k;
            }
            if (victim < 0) { rc = -2; goto out; }
            used[d] -= pb->weight[victim];
            st[victim] = 0;
            nres[d] -= 1;
            evicted |= 1u << victim;
        }
        if (hit) {
            start = imax64(t_free[d], rel);
        } else {
            /* Load on the consumer's device (Eq. 5, Eq. 9).  A prefetched load
             * waits only for the device and the session's arrival. */
            ls = bit_of(prefetch, h) ? imax64(t_free[d], pb->arrival[w]) : imax64(t_free[d], rel);
            if (occ_since[d] == ORC_NONE) occ_since[d] = ls;
            le = ls + pb->load[(int64_t)m * D + d];
            used[d] += pb->weight[m];
            nres[d] += 1;
            start = imax64(le, rel);
            /* Eq. 12's lifecycle terms: a prefetched load that started before
             * the release and ended by it is timely; a load of a model this
             * device held before is a reload caused by reclamation. */
            if (bit_of(prefetch, h) && ls < rel && le <= rel) ++timely;
            if (loaded[(int64_t)d * M + m]) life += pb->load[(int64_t)m * D + d];
            loaded[(int64_t)d * M + m] = 1;
        }
        /* The ready-work loading delay: how far the load pushes the start
         * beyond the later of the release and the device's free time. */
        life += start - imax64(t_free[d], rel);
        start += pb->grant;  /* one grant per unit, however long the chain */

        /* Execute the chain back to back (Eq. 4 run time = sum of members). */
        int64_t t = start;
        for (int32_t j = 0; j < len; ++j) {
            int32_t n = chain[j];
            if (tr) { tr->start[n] = t; tr->head_of[n] = h; tr->rel[n] = (j == 0) ? rel : -1; }
            t += L[(int64_t)n * D + d];
            c[n] = t;
            done[n] = 1;
        }
        t_free[d] = c[last];
        st[m] = ++seq;

        if (tr) {
            tr->unit_head[(*tr->n_units)++] = h;
            tr->load_start[h] = ls;
            tr->load_end[h] = le;
            tr->kv_adm[h] = (int32_t)kv_adm;
            tr->used_after[h] = (int32_t)used[d];
            tr->evicted[h] = evicted;
            tr->reclaimed[h] = 0;
        }

        /* Retain bit 0: reclaim the model when the unit ends (zero-cost
         * reclaim); an emptied device stops accruing GPU time. */
        if (retain && !bit_of(retain, last)) {
            used[d] -= pb->weight[m];
            st[m] = 0;
            nres[d] -= 1;
            if (tr) tr->reclaimed[h] = 1;
            if (nres[d] == 0) {
                gpu[d] += c[last] - occ_since[d];
                if (tr) {
                    int32_t k = (*tr->n_occ)++;
                    tr->occ_start[k] = occ_since[d]; tr->occ_end[k] = c[last]; tr->occ_dev[k] = d;
                }
                occ_since[d] = ORC_NONE;
            }
        }
    }

    /* Metrics (Section 4.2-4.3). */
    int64_t end = 0, first = ORC_INF;
    for (int32_t n = 0; n < N; ++n) end = imax64(end, c[n]);
    for (int32_t w = 0; w < W; ++w) first = imin64(first, pb->arrival[w]);
    *makespan = end - first;
    int64_t g = 0;
    for (int32_t d = 0; d < D; ++d) {
        if (occ_since[d] != ORC_NONE) {
            gpu[d] += end - occ_since[d];
            if (tr) {
                int32_t k = (*tr->n_occ)++;
                tr->occ_start[k] = occ_since[d]; tr->occ_end[k] = end; tr->occ_dev[k] = d;
            }
        }
        g += gpu[d];
    }
    *gpu_total = g;
    for (int32_t w = 0; w < W; ++w) comp_w[w] = ORC_NONE;
    for (int32_t n = 0; n < N; ++n) {
        int32_t w = pb->session[n];
        comp_w[w] = imax64(comp_w[w], c[n] - pb->arrival[w]);
    }
    if (tr) for (int32_t n = 0; n < N; ++n) tr->finish[n] = c[n];
    if (phi) { phi[0] = timely; phi[1] = life; }
out:
    free(t_free); free(occ_since); free(gpu); free(used); free(nres); free(stamp); free(done); free(chain);
    free(is_head); free(fprev); free(loaded);
    return rc;
}

/*
 * The same play with the replica batch limit B_q of Section 3.5 (B = batch
 * >= 1).  Eq. 11 sums the request memory of every unit active at a
 * transition boundary, and concurrent units of one replica respect its batch
 * limit.  A replica is a model resident on a device; a device runs units of
 * one replica at a time, up to B of them at once:
 *   - units are admitted in the plan's dispatch order;
 *   - a unit of the device's current replica joins it: it takes the slot
 *     (of B) that frees earliest, no earlier than its release and than the
 *     previous admission on the device, and is admitted once resident
 *     weights + the KV needs of the units still running + its own KV fit the
 *     capacity (least-recently-used idle models are reclaimed first; if that
 *     is not enough, it waits for the next running unit to end);
 *   - a unit of another model waits until the device has drained (every
 *     running unit ended) and then hits or loads exactly as in simulate,
 *     with the device free at the drain time; it becomes the current
 *     replica, and its other slots free when the model is ready;
 *   - a unit's KV is held from its admission (the load start on a miss) to
 *     its end.
 * With admissions in dispatch order, memory use over a unit's interval peaks
 * at its admission, so one check there covers Eq. 11 for it.  With B = 1 the
 * play equals simulate's.  Retain rows are modelled for B = 1 only; the
 * window terms of Eq. 12 and reclamation by next use are not modelled here.
 */
static int simulate_batched(const orc_problem *pb, const int32_t *fnext,
                            const uint8_t *place, const uint16_t *order,
                            const uint32_t *fuse, const uint32_t *prefetch, const uint32_t *retain,
                            const int64_t *L, int64_t *c, int64_t *comp_w,
                            int64_t *makespan, int64_t *gpu_total, orc_trace *tr)
{
    const int32_t N = pb->N, D = pb->D, M = pb->M, W = pb->W, B = pb->batch;
    if (B < 1 || (B > 1 && retain) || pb->reclaim) return -3;
    int64_t *slot_end = (int64_t *)malloc(sizeof(int64_t) * (size_t)D * (size_t)B);
    int64_t *slot_kv = (int64_t *)malloc(sizeof(int64_t) * (size_t)D * (size_t)B);
    int64_t *last_adm = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int32_t *cur = (int32_t *)malloc(sizeof(int32_t) * (size_t)D);
    int64_t *occ_since = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int64_t *gpu = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int64_t *used = (int64_t *)malloc(sizeof(int64_t) * (size_t)D);
    int32_t *nres = (int32_t *)malloc(sizeof(int32_t) * (size_t)D);
    int64_t *stamp = (int64_t *)malloc(sizeof(int64_t) * (size_t)D * (size_t)M);
    uint8_t *done = (uint8_t *)malloc((size_t)N);
    int32_t *chain = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int rc = 0;
    if (!slot_end || !slot_kv || !last_adm || !cur || !occ_since || !gpu || !used || !nres || !stamp || !done ||
        !chain) {
        rc = -1;
        goto out;
    }
    for (int32_t d = 0; d < D; ++d) {
        for (int32_t j = 0; j < B; ++j) { slot_end[(int64_t)d * B + j] = 0; slot_kv[(int64_t)d * B + j] = 0; }
        last_adm[d] = 0; cur[d] = -1; occ_since[d] = ORC_NONE; gpu[d] = 0; used[d] = 0; nres[d] = 0;
        for (int32_t m = 0; m < M; ++m) stamp[(int64_t)d * M + m] = 0;  /* 0 = not resident */
    }
    memset(done, 0, (size_t)N);
    int64_t seq = 0;
    if (tr) { *tr->n_units = 0; *tr->n_occ = 0; }

    for (int32_t i = 0; i < N; ++i) {
        const int32_t h = order[i];
        if (done[h]) continue;  /* already ran inside an earlier chain */
        int32_t len = 0;
        chain[len++] = h;
        for (;;) {
            int32_t s = fnext[chain[len - 1]];
            if (s < 0 || !bit_of(fuse, s) || place[s] != place[h]) break;
            chain[len++] = s;
        }
        const int32_t last = chain[len - 1];
        const int32_t d = place[h];
        const int32_t m = pb->model[h];
        const int32_t w = pb->session[h];
        int64_t *st = &stamp[(int64_t)d * M];
        int64_t *se = &slot_end[(int64_t)d * B];
        int64_t *sk = &slot_kv[(int64_t)d * B];
        int64_t rel = pb->arrival[w];
        for (int32_t e = pb->pred_off[h]; e < pb->pred_off[h + 1]; ++e)
            rel = imax64(rel, c[pb->pred_idx[e]]);
        int64_t kv_adm = 0;
        for (int32_t j = 0; j < len; ++j)
            kv_adm = imax64(kv_adm, (int64_t)pb->peak[(int64_t)chain[j] * D + d] - pb->weight[m]);

        int64_t adm, start, ls = -1, le = -1;
        int32_t slot = 0;
        uint32_t evicted = 0;
        if (m == cur[d]) {
            /* Join the current replica: the earliest-free slot (lowest index
             * on ties), in dispatch order, once memory allows (Eq. 11). */
            for (int32_t j = 1; j < B; ++j)
                if (se[j] < se[slot]) slot = j;
            adm = imax64(imax64(rel, se[slot]), last_adm[d]);
            for (;;) {
                int64_t running = 0;
                for (int32_t j = 0; j < B; ++j)
                    if (se[j] > adm) running += sk[j];
                while (used[d] + running + kv_adm > pb->cap[d]) {
                    int32_t victim = -1;
                    for (int32_t k = 0; k < M; ++k)
                        if (k != m && st[k] != 0 && (victim < 0 || st[k] < st[victim])) victim = k;
                    if (victim < 0) break;
                    used[d] -= pb->weight[victim];
                    st[victim] = 0;
                    nres[d] -= 1;
                    evicted |= 1u << victim;
                }
                if (used[d] + running + kv_adm <= pb->cap[d]) break;
                /* not even without idle models: wait for the next running unit to end */
                int64_t next = ORC_INF;
                for (int32_t j = 0; j < B; ++j)
                    if (se[j] > adm) next = imin64(next, se[j]);
                if (next == ORC_INF) { rc = -2; goto out; }  /* unreachable for a valid plan */
                adm = next;
            }
            start = adm;
        } else {
            /* Another model: the device drains, then the unit hits or loads as
             * in simulate with the device free at the drain time. */
            int64_t drain = 0;
            for (int32_t j = 0; j < B; ++j) drain = imax64(drain, se[j]);
            const int hit = st[m] != 0;
            const int64_t need = hit ? kv_adm : pb->weight[m] + kv_adm;
            while (used[d] + need > pb->cap[d]) {
                int32_t victim = -1;
                for (int32_t k = 0; k < M; ++k)
                    if (k != m && st[k] != 0 && (victim < 0 || st[k] < st[victim])) victim = k;
                if (victim < 0) { rc = -2; goto out; }
                used[d] -= pb->weight[victim];
                st[victim] = 0;
                nres[d] -= 1;
                evicted |= 1u << victim;
            }
            int64_t ready;
            if (hit) {
                adm = start = imax64(drain, rel);
                ready = drain;
            } else {
                ls = bit_of(prefetch, h) ? imax64(drain, pb->arrival[w]) : imax64(drain, rel);
                if (occ_since[d] == ORC_NONE) occ_since[d] = ls;
                le = ls + pb->load[(int64_t)m * D + d];
                used[d] += pb->weight[m];
                nres[d] += 1;
                adm = ls;
                start = imax64(le, rel);
                ready = le;
            }
            for (int32_t j = 0; j < B; ++j) { se[j] = ready; sk[j] = 0; }
            cur[d] = m;
        }
        start += pb->grant;
        int64_t t = start;
        for (int32_t j = 0; j < len; ++j) {
            int32_t n = chain[j];
            if (tr) { tr->start[n] = t; tr->head_of[n] = h; tr->rel[n] = (j == 0) ? rel : -1; }
            t += L[(int64_t)n * D + d];
            c[n] = t;
            done[n] = 1;
        }
        se[slot] = c[last];
        sk[slot] = kv_adm;
        last_adm[d] = adm;
        st[m] = ++seq;
        if (tr) {
            tr->unit_head[(*tr->n_units)++] = h;
            tr->load_start[h] = ls;
            tr->load_end[h] = le;
            tr->kv_adm[h] = (int32_t)kv_adm;
            tr->used_after[h] = (int32_t)used[d];
            tr->evicted[h] = evicted;
            tr->reclaimed[h] = 0;
            if (tr->adm) tr->adm[h] = adm;
        }
        /* Retain bit 0 (B = 1 only): the model leaves when the unit ends, and
         * the device has no current replica. */
        if (retain && !bit_of(retain, last)) {
            used[d] -= pb->weight[m];
            st[m] = 0;
            nres[d] -= 1;
            cur[d] = -1;
            if (tr) tr->reclaimed[h] = 1;
            if (nres[d] == 0) {
                gpu[d] += c[last] - occ_since[d];
                if (tr) {
                    int32_t k = (*tr->n_occ)++;
                    tr->occ_start[k] = occ_since[d]; tr->occ_end[k] = c[last]; tr->occ_dev[k] = d;
                }
                occ_since[d] = ORC_NONE;
            }
        }
    }

    int64_t end = 0, first = ORC_INF;
    for (int32_t n = 0; n < N; ++n) end = imax64(end, c[n]);
    for (int32_t w = 0; w < W; ++w) first = imin64(first, pb->arrival[w]);
    *makespan = end - first;
    int64_t g = 0;
    for (int32_t d = 0; d < D; ++d) {
        if (occ_since[d] != ORC_NONE) {
            gpu[d] += end - occ_since[d];
            if (tr) {
                int32_t k = (*tr->n_occ)++;
                tr->occ_start[k] = occ_since[d]; tr->occ_end[k] = end; tr->occ_dev[k] = d;
            }
        }
        g += gpu[d];
    }
    *gpu_total = g;
    for (int32_t w = 0; w < W; ++w) comp_w[w] = ORC_NONE;
    for (int32_t n = 0; n < N; ++n) {
        int32_t w = pb->session[n];
        comp_w[w] = imax64(comp_w[w], c[n] - pb->arrival[w]);
    }
    if (tr) for (int32_t n = 0; n < N; ++n) tr->finish[n] = c[n];
out:
    free(slot_end); free(slot_kv); free(last_adm); free(cur); free(occ_since); free(gpu); free(used); free(nres);
    free(stamp); free(done); free(chain);
    return rc;
}

/* SplitMix64 (Steele, Lea and Flood, OOPSLA 2014): advance by the golden
 * gamma, then the variant-13 finaliser.  mix(x) is one output for state x. */
uint64_t orc_splitmix64(uint64_t x)
{
    uint64_t z = x + 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/*
 * Latency multiplier of (plan, sample, node), 16 fractional bits:
 * h = mix(mix(mix(seed ^ plan) ^ sample) ^ node); a radius index from the low
 * bits and an angle index from bits 32 and up; zq = floor(R * Cc / 2^18) (an
 * integer Box-Muller normal in units of 1/256); the multiplier is E[zq + ZOFF]
 * with ZOFF = (len(E) - 1) / 2.
 */
int64_t orc_multiplier(const orc_problem *pb, uint64_t plan, uint64_t sample, uint64_t node)
{
    uint64_t h = orc_splitmix64(orc_splitmix64(orc_splitmix64(pb->seed ^ plan) ^ sample) ^ node);
    int64_t i1 = (int64_t)(h & (uint64_t)(pb->bm_rn - 1));
    int64_t i2 = (int64_t)((h >> 32) & (uint64_t)(pb->bm_cn - 1));
    int64_t prod = (int64_t)pb->bm_r[i1] * (int64_t)pb->bm_c[i2];
    int64_t zq = prod / 262144;                    /* C division truncates toward 0 ... */
    if (prod % 262144 != 0 && prod < 0) zq -= 1;   /* ... so step down to the floor */
    return pb->bm_e[zq + (pb->bm_en - 1) / 2];
}

/*
 * Evaluate one plan: status bits, then the deterministic play (S = 0) or S
 * stochastic plays with L' = (L * mult + 2^15) >> 16.  Outputs: makespan,
 * p95 and gpu (INT64_MAX each for an invalid plan); stochastic makespan and
 * gpu are floor means over samples, p95 is over the pooled S*W completions.
 * tr (deterministic only) may be NULL.
 */
int orc_eval_plan(const orc_problem *pb, const int32_t *fnext,
                  const uint8_t *place, const uint16_t *order,
                  const uint32_t *fuse, const uint32_t *prefetch, const uint32_t *retain,
                  int64_t plan_index, int64_t *out3, uint32_t *status, orc_trace *tr)
{
    const int32_t N = pb->N, D = pb->D, W = pb->W;
    int rc = orc_status(pb, place, order, status);
    if (rc) return rc;
    if (*status != 0) { out3[0] = out3[1] = out3[2] = ORC_INF; return 0; }

    const int32_t S = pb->S > 0 ? pb->S : 1;
    int64_t *L = (int64_t *)malloc(sizeof(int64_t) * (size_t)N * (size_t)D);
    int64_t *c = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
    int64_t *pool = (int64_t *)malloc(sizeof(int64_t) * (size_t)S * (size_t)W);
    if (!L || !c || !pool) { rc = -1; goto out; }
    int64_t sum_mk = 0, sum_gpu = 0;
    for (int32_t s = 0; s < S; ++s) {
        for (int32_t n = 0; n < N; ++n)
            for (int32_t d = 0; d < D; ++d) {
                int64_t base = pb->lat[(int64_t)n * D + d];
                if (pb->S > 0) {
                    int64_t mult = orc_multiplier(pb, (uint64_t)plan_index, (uint64_t)s, (uint64_t)n);
                    L[(int64_t)n * D + d] = (base * mult + 32768) >> 16;
                } else {
                    L[(int64_t)n * D + d] = base;
                }
            }
        int64_t mk, g;
        rc = pb->batch > 0
                 ? simulate_batched(pb, fnext, place, order, fuse, prefetch, retain, L, c, &pool[(int64_t)s * W],
                                    &mk, &g, pb->S > 0 ? NULL : tr)
                 : simulate(pb, fnext, place, order, fuse, prefetch, retain, L, c,
                            &pool[(int64_t)s * W], &mk, &g, pb->S > 0 ? NULL : tr, NULL);
        if (rc) goto out;
        sum_mk += mk;
        sum_gpu += g;
    }
    out3[0] = sum_mk / S;
    out3[1] = nearest_rank(pool, (int64_t)S * W, 95);
    out3[2] = sum_gpu / S;
out:
    free(L); free(c); free(pool);
    return rc;
}

/*
 * Evaluate plans [lo, hi) of a batch (row strides in bytes; retain may be
 * NULL = all retained).  Plan p's global index is plan_base + p.
 */
int orc_eval_batch(const orc_problem *pb, const int32_t *fnext,
                   const uint8_t *place, int64_t place_stride,
                   const uint16_t *order, int64_t order_stride,
                   const uint32_t *fuse, const uint32_t *prefetch, const uint32_t *retain,
                   int64_t bits_stride, int64_t plan_base, int64_t lo, int64_t hi,
                   int64_t *makespan, int64_t *p95, int64_t *gpu, uint32_t *status)
{
    for (int64_t p = lo; p < hi; ++p) {
        int64_t o[3];
        const uint8_t *pl = place + p * place_stride;
        const uint16_t *od = (const uint16_t *)((const uint8_t *)order + p * order_stride);
        const uint32_t *fu = (const uint32_t *)((const uint8_t *)fuse + p * bits_stride);
        const uint32_t *pf = (const uint32_t *)((const uint8_t *)prefetch + p * bits_stride);
        const uint32_t *rt = retain ? (const uint32_t *)((const uint8_t *)retain + p * bits_stride) : NULL;
        int rc = orc_eval_plan(pb, fnext, pl, od, fu, pf, rt, plan_base + p, o, &status[p], NULL);
        if (rc) return rc;
        makespan[p] = o[0]; p95[p] = o[1]; gpu[p] = o[2];
    }
    return 0;
}

/*
 * The window terms of the ranking key of Eq. 12 for plans [lo, hi) of a
 * deterministic batch (S = 0).  Over a whole window every unit is admitted,
 * so the coverage counts A_k are equal for all valid plans and the key
 * reduces to (latest completion, -P_N, H_life):
 *   timely[p]  P_N, the units whose model load ran under their prefetch bit,
 *              started before the unit's release and ended by it;
 *   life[p]    H_life, the sum over units of the delay the load adds to the
 *              start, max(load end, release) - max(device free, release)
 *              (zero on a hit), plus the load time of every load of a model
 *              its device had held before (a reload after reclamation).
 * Invalid plans get INT64_MAX for both.  Returns -3 when S > 0.
 */
int orc_eval_phi_batch(const orc_problem *pb, const int32_t *fnext,
                       const uint8_t *place, int64_t place_stride,
                       const uint16_t *order, int64_t order_stride,
                       const uint32_t *fuse, const uint32_t *prefetch, const uint32_t *retain,
                       int64_t bits_stride, int64_t lo, int64_t hi, int64_t *timely, int64_t *life)
{
    if (pb->S > 0 || pb->batch > 0) return -3;  /* deterministic, one unit at a time per device */
    const int32_t N = pb->N, D = pb->D, W = pb->W;
    int64_t *L = (int64_t *)malloc(sizeof(int64_t) * (size_t)N * (size_t)D);
    int64_t *c = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
    int64_t *comp = (int64_t *)malloc(sizeof(int64_t) * (size_t)W);
    int rc = 0;
    if (!L || !c || !comp) { rc = -1; goto out; }
    for (int64_t k = 0; k < (int64_t)N * D; ++k) L[k] = pb->lat[k];
    for (int64_t p = lo; p < hi; ++p) {
        const uint8_t *pl = place + p * place_stride;
        const uint16_t *od = (const uint16_t *)((const uint8_t *)order + p * order_stride);
        const uint32_t *fu = (const uint32_t *)((const uint8_t *)fuse + p * bits_stride);
        const uint32_t *pf = (const uint32_t *)((const uint8_t *)prefetch + p * bits_stride);
        const uint32_t *rt = retain ? (const uint32_t *)((const uint8_t *)retain + p * bits_stride) : NULL;
        uint32_t st;
        rc = orc_status(pb, pl, od, &st);
        if (rc) goto out;
        if (st != 0) { timely[p] = life[p] = ORC_INF; continue; }
        int64_t mk, g, phi[2];
        rc = simulate(pb, fnext, pl, od, fu, pf, rt, L, c, comp, &mk, &g, NULL, phi);
        if (rc) goto out;
        timely[p] = phi[0];
        life[p] = phi[1];
    }
out:
    free(L); free(c); free(comp);
    return rc;
}

/*
 * Local search around the best plans (the scheduler's re-ranking of its
 * uncommitted decisions after new information, Section 3.5): each child is a
 * copy of a parent with n_ops point changes.  Child c (0-based within the
 * call) copies parent c mod n_parents; change s of child c is decoded from
 *   h = mix(mix(mix(seed ^ round) ^ c) ^ s),  x = bits 8..39 of h,  y = bits 40..63:
 *   h mod 4 = 0  move:     n = x mod N; the device becomes the (y mod f)-th
 *                          (0-based, ascending) of the f devices whose
 *                          capacity holds peak[n][d] (Eq. 8);
 *             1  fuse:     n = x mod N; flip the fuse bit of n (Eq. 3);
 *             2  prefetch: n = x mod N; flip the prefetch bit of n (Eq. 5);
 *             3  swap:     i = x mod (N - 1); exchange dispatch positions i
 *                          and i + 1 unless the node at i is a graph
 *                          predecessor of the node at i + 1 (Eq. 10 keeps
 *                          the sequence topological); no change when N = 1
 *                          or the node at i + 1 is not an activation.
 * Retain bits are copied unchanged.  Rows are addressed with byte strides.
 */
static int is_pred(const orc_problem *pb, int32_t u, int32_t v)
{
    for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e)
        if (pb->pred_idx[e] == u) return 1;
    return 0;
}

int orc_mutate(const orc_problem *pb,
               const uint8_t *place, int64_t place_stride,
               const uint16_t *order, int64_t order_stride,
               const uint32_t *fuse, const uint32_t *prefetch, const uint32_t *retain, int64_t bits_stride,
               int64_t n_parents,
               uint8_t *c_place, int64_t c_place_stride,
               uint16_t *c_order, int64_t c_order_stride,
               uint32_t *c_fuse, uint32_t *c_prefetch, uint32_t *c_retain, int64_t c_bits_stride,
               int64_t n_children, uint64_t seed, int64_t round, int32_t n_ops)
{
    const int32_t N = pb->N, D = pb->D, words = (N + 31) / 32;
    for (int64_t c = 0; c < n_children; ++c) {
        const int64_t p = c % n_parents;
        const uint8_t *pp = place + p * place_stride;
        const uint16_t *po = (const uint16_t *)((const uint8_t *)order + p * order_stride);
        const uint32_t *pf = (const uint32_t *)((const uint8_t *)fuse + p * bits_stride);
        const uint32_t *pr = (const uint32_t *)((const uint8_t *)prefetch + p * bits_stride);
        uint8_t *cp = c_place + c * c_place_stride;
        uint16_t *co = (uint16_t *)((uint8_t *)c_order + c * c_order_stride);
        uint32_t *cf = (uint32_t *)((uint8_t *)c_fuse + c * c_bits_stride);
        uint32_t *cr = (uint32_t *)((uint8_t *)c_prefetch + c * c_bits_stride);
        memcpy(cp, pp, (size_t)N);
        memcpy(co, po, 2 * (size_t)N);
        memcpy(cf, pf, 4 * (size_t)words);
        memcpy(cr, pr, 4 * (size_t)words);
        if (retain)
            memcpy((uint8_t *)c_retain + c * c_bits_stride, (const uint8_t *)retain + p * bits_stride,
                   4 * (size_t)words);
        for (int32_t s = 0; s < n_ops; ++s) {
            const uint64_t h = orc_splitmix64(orc_splitmix64(orc_splitmix64(seed ^ (uint64_t)round) ^ (uint64_t)c) ^
                                              (uint64_t)s);
            const uint32_t x = (uint32_t)(h >> 8);
            const uint32_t y = (uint32_t)(h >> 40);
            const int op = (int)(h & 3u);
            if (op == 3) {
                if (N < 2) continue;
                const int32_t i = (int32_t)(x % (uint32_t)(N - 1));
                const int32_t u = co[i], v = co[i + 1];
                if (v < N && !(u < N && is_pred(pb, u, v))) { co[i] = (uint16_t)v; co[i + 1] = (uint16_t)u; }
                continue;
            }
            const int32_t n = (int32_t)(x % (uint32_t)N);
            if (op == 0) {
                int32_t f = 0;
                for (int32_t d = 0; d < D; ++d) f += pb->peak[(int64_t)n * D + d] <= pb->cap[d];
                if (f == 0) continue;
                int32_t r = (int32_t)(y % (uint32_t)f);
                for (int32_t d = 0; d < D; ++d)
                    if (pb->peak[(int64_t)n * D + d] <= pb->cap[d] && r-- == 0) { cp[n] = (uint8_t)d; break; }
            } else if (op == 1) {
                cf[n >> 5] ^= 1u << (n & 31);
            } else {
                cr[n >> 5] ^= 1u << (n & 31);
            }
        }
    }
    return 0;
}

/*
 * Plan construction (Algorithm 1 read for a whole window, one plan per
 * call).  The constructor is a list scheduler that plays each decision
 * forward with the evaluation rules above, so the finish times it sees are
 * the ones the evaluator will report for its plan:
 *
 *   RankReady: a unit is ready once every graph predecessor is dispatched;
 *     its rank is its release (Eq. 2: session arrival and predecessor
 *     finishes) plus a jitter drawn per (plan, node); the ready unit with
 *     the smallest (rank, node id) goes next -- the one that has waited
 *     longest (aging).
 *   BestFeasibleBinding: among the devices whose capacity holds the node
 *     (Eq. 8), the one with the smallest predicted finish of the node
 *     (a resident model costs no load; a missing one is loaded on the
 *     device, prefetched when the device would otherwise idle before the
 *     release) plus a jitter drawn per (plan, node, device); ties go to
 *     the lower device.
 *   Units: the node's fusible chain (Eq. 3) follows it on the same device
 *     while each next member fits there (fuse bit 1), dispatched at once.
 *   PlanPrefetch: the head's prefetch bit is set when its model is not
 *     resident on the device and the device is free before the release.
 *   Retain: every model stays resident (no retain row).
 *
 * Jitter: h = mix(mix(seed ^ plan) ^ node); rank jitter h mod (J + 1),
 * device jitter mix(h ^ (d + 1)) mod (J + 1); J = 0 gives the plain greedy.
 * Outputs the plan rows (fuse / prefetch rows of ceil(N/32) words) and the
 * largest finish.  Returns 0, or -1 when memory runs out.
 */
int orc_construct(const orc_problem *pb, const int32_t *fnext, uint64_t seed, uint64_t plan, int64_t jitter,
                  uint8_t *place, uint16_t *order, uint32_t *fuse, uint32_t *prefetch, int64_t *end_out)
{
    const int32_t N = pb->N, D = pb->D, M = pb->M;
    const int32_t E = pb->pred_off[N];
    const int32_t words = (N + 31) / 32;
    int64_t *c = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
    int64_t *rel = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
    int64_t *rank = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
    int32_t *pending = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int32_t *ready = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int32_t *succ_off = (int32_t *)calloc((size_t)N + 1, sizeof(int32_t));
    int32_t *succ = (int32_t *)malloc(sizeof(int32_t) * (size_t)(E > 0 ? E : 1));
    int32_t *chain = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int64_t *t_free = (int64_t *)calloc((size_t)D, sizeof(int64_t));
    int64_t *used = (int64_t *)calloc((size_t)D, sizeof(int64_t));
    int64_t *stamp = (int64_t *)calloc((size_t)D * (size_t)M, sizeof(int64_t));
    int rc = 0;
    if (!c || !rel || !rank || !pending || !ready || !succ_off || !succ || !chain || !t_free || !used || !stamp) {
        rc = -1;
        goto out;
    }
    /* Successor lists (the transpose of the predecessor CSR). */
    for (int32_t e = 0; e < E; ++e) succ_off[pb->pred_idx[e] + 1] += 1;
    for (int32_t v = 0; v < N; ++v) succ_off[v + 1] += succ_off[v];
    {
        int32_t *fill = pending;  /* scratch, reset below */
        for (int32_t v = 0; v < N; ++v) fill[v] = succ_off[v];
        for (int32_t v = 0; v < N; ++v)
            for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) succ[fill[pb->pred_idx[e]]++] = v;
    }
    memset(fuse, 0, sizeof(uint32_t) * (size_t)words);
    memset(prefetch, 0, sizeof(uint32_t) * (size_t)words);

    int32_t nready = 0, pos = 0;
    int64_t end = 0, seq = 0;
    for (int32_t v = 0; v < N; ++v) {
        pending[v] = pb->pred_off[v + 1] - pb->pred_off[v];
        if (pending[v] == 0) {
            const uint64_t h = orc_splitmix64(orc_splitmix64(seed ^ plan) ^ (uint64_t)v);
            rel[v] = pb->arrival[pb->session[v]];
            rank[v] = rel[v] + (jitter > 0 ? (int64_t)(h % (uint64_t)(jitter + 1)) : 0);
            ready[nready++] = v;
        }
    }
    while (nready > 0) {
        /* RankReady: smallest (rank, node id). */
        int32_t j = 0;
        for (int32_t k = 1; k < nready; ++k) {
            const int32_t a = ready[k], b = ready[j];
            if (rank[a] < rank[b] || (rank[a] == rank[b] && a < b)) j = k;
        }
        const int32_t u = ready[j];
        ready[j] = ready[--nready];
        const int32_t m = pb->model[u];
        const int64_t arr = pb->arrival[pb->session[u]];
        const uint64_t hu = orc_splitmix64(orc_splitmix64(seed ^ plan) ^ (uint64_t)u);

        /* BestFeasibleBinding: smallest predicted finish (+ jitter). */
        int32_t d = -1;
        int64_t best = 0;
        for (int32_t dd = 0; dd < D; ++dd) {
            if (pb->peak[(int64_t)u * D + dd] > pb->cap[dd]) continue;
            int64_t start;
            if (stamp[(int64_t)dd * M + m] != 0) {
                start = imax64(t_free[dd], rel[u]);
            } else {
                const int64_t ls = t_free[dd] < rel[u] ? imax64(t_free[dd], arr) : imax64(t_free[dd], rel[u]);
                start = imax64(ls + pb->load[(int64_t)m * D + dd], rel[u]);
            }
            const int64_t fin = start + pb->grant + pb->lat[(int64_t)u * D + dd];
            const int64_t score =
                fin + (jitter > 0 ? (int64_t)(orc_splitmix64(hu ^ (uint64_t)(dd + 1)) % (uint64_t)(jitter + 1)) : 0);
            if (d < 0 || score < best) { d = dd; best = score; }
        }
        if (d < 0) { rc = -2; goto out; }  /* no device holds u: the problem is invalid */

        /* The unit: u and the members of its fusible chain that fit on d. */
        int32_t len = 0;
        chain[len++] = u;
        for (int32_t s = fnext[u]; s >= 0 && pb->peak[(int64_t)s * D + d] <= pb->cap[d]; s = fnext[s])
            chain[len++] = s;
        const int hit = stamp[(int64_t)d * M + m] != 0;
        const int pf = !hit && t_free[d] < rel[u];
        for (int32_t k = 0; k < len; ++k) {
            const int32_t x = chain[k];
            place[x] = (uint8_t)d;
            order[pos++] = (uint16_t)x;
            if (k > 0) fuse[x >> 5] |= 1u << (x & 31);
        }
        if (pf) prefetch[u >> 5] |= 1u << (u & 31);

        /* Play the unit forward exactly as the evaluation does. */
        int64_t kv_adm = 0;
        for (int32_t k = 0; k < len; ++k)
            kv_adm = imax64(kv_adm, (int64_t)pb->peak[(int64_t)chain[k] * D + d] - pb->weight[m]);
        const int64_t admit = hit ? kv_adm : pb->weight[m] + kv_adm;
        int64_t *lru = &stamp[(int64_t)d * M];
        while (used[d] + admit > pb->cap[d]) {  /* Eq. 11, least recently used first */
            int32_t victim = -1;
            for (int32_t k = 0; k < M; ++k)
                if (k != m && lru[k] != 0 && (victim < 0 || lru[k] < lru[victim])) victim = k;
            if (victim < 0) { rc = -3; goto out; }
            used[d] -= pb->weight[victim];
            lru[victim] = 0;
        }
        int64_t start;
        if (hit) {
            start = imax64(t_free[d], rel[u]);
        } else {
            const int64_t ls = pf ? imax64(t_free[d], arr) : imax64(t_free[d], rel[u]);
            start = imax64(ls + pb->load[(int64_t)m * D + d], rel[u]);
            used[d] += pb->weight[m];
        }
        int64_t t = start + pb->grant;
        for (int32_t k = 0; k < len; ++k) {
            t += pb->lat[(int64_t)chain[k] * D + d];
            c[chain[k]] = t;
        }
        t_free[d] = t;
        lru[m] = ++seq;
        end = imax64(end, t);

        /* Successors of the unit's last member become ready when their
         * last predecessor is dispatched (the other members' only
         * successors are inside the unit). */
        const int32_t tail = chain[len - 1];
        for (int32_t e = succ_off[tail]; e < succ_off[tail + 1]; ++e) {
            const int32_t y = succ[e];
            if (--pending[y] > 0) continue;
            int64_t r = pb->arrival[pb->session[y]];
            for (int32_t f = pb->pred_off[y]; f < pb->pred_off[y + 1]; ++f) r = imax64(r, c[pb->pred_idx[f]]);
            const uint64_t h = orc_splitmix64(orc_splitmix64(seed ^ plan) ^ (uint64_t)y);
            rel[y] = r;
            rank[y] = r + (jitter > 0 ? (int64_t)(h % (uint64_t)(jitter + 1)) : 0);
            ready[nready++] = y;
        }
    }
    if (pos != N) rc = -4;  /* unreachable for an acyclic window */
    *end_out = end;
out:
    free(c); free(rel); free(rank); free(pending); free(ready); free(succ_off); free(succ); free(chain);
    free(t_free); free(used); free(stamp);
    return rc;
}
