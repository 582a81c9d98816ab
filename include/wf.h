/*
 * wf.h -- C ABI of the GB300 batched plan evaluator (libwf.so).
 *
 * A *problem* is one window of the activation DAG of concurrent multi-agent
 * workflows (paper Section 3.2) together with Predictor-style cost tables
 * (Eq. 1).  A *plan* fixes a device per activation, a dispatch sequence that
 * orients every resource conflict, and per-activation fusion / prefetch /
 * retain bits (Eq. 3-10).  The library evaluates batches of plans on one GPU
 * and ranks them:
 *
 *   wf_problem_check        validate a problem on the host (no GPU needed)
 *   wf_ctx_create           validate, derive and upload a problem (once)
 *   wf_forecast_readiness   release forecast of every activation (Eq. 2)
 *   wf_eval_plans           play every plan forward (Eq. 2-11) -> metrics
 *   wf_topk                 the k best plans by the ranking key
 *   wf_eval_topk_host       forecast + evaluation + top-k from and to host memory
 *   wf_ctx_reserve_host     allocate wf_eval_topk_host's staging up front
 *   wf_eval_plans_static    wf_eval_plans without a context or any allocation
 *   wf_static_status        device-side outcome of the last wf_eval_plans_static
 *   wf_mutate_plans         children of plans with a few point changes each
 *   wf_merge_elite          keep the k best of an elite and its children
 *   wf_local_search         rounds of mutate -> evaluate -> merge
 *   wf_construct_plans      plans built by a list scheduler (Algorithm 1)
 *   wf_ctx_set_reclaim      reclamation order: LRU or by next use
 *   wf_eval_plans_phi       wf_eval_plans plus the window terms of Eq. 12
 *   wf_topk_phi             the k best plans by Eq. 12's window key
 *   wf_ctx_status           device-side failures of earlier calls
 *   wf_ctx_check_wait_expiry  the bounded device wait's expiry path (tests)
 *   wf_ctx_set_eval_path    every plan on the exact int64 path (tests, cross-checks)
 *   wf_ctx_set_batch        replica batch limit B_q (Eq. 11, Section 3.5)
 *   wf_ctx_destroy, wf_strerror, wf_last_error
 *
 * Conventions.
 *   - Times are int64 microseconds, memory int32 MiB; every output is an
 *     exact integer.
 *   - Tables are row-major: lat_us and peak_mib are [N][D] (index n*D + d),
 *     load_us is [M][D].
 *   - Problem pointers are HOST pointers, read during wf_ctx_create only; the
 *     caller keeps ownership.  Plan and output pointers are DEVICE pointers
 *     owned by the caller (HOST pointers for wf_eval_topk_host); the library
 *     never frees them.
 *   - Calls taking a stream (a cudaStream_t passed as void*, NULL = the
 *     legacy default stream) are asynchronous on it and allocate nothing:
 *     the context owns every scratch buffer, sized at creation for up to
 *     max_P plans per call (wf_eval_topk_host's staging, and the plan
 *     constructor's state, at their first use).  One context serves one
 *     stream at a time.
 *   - Return codes: WF_OK (0) or a WF_E* code below.  Problems with single
 *     plans are data (status bits), never return codes.
 */
#ifndef WF_H
#define WF_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    WF_OK = 0,
    WF_EINVAL = 1,    /* a null pointer, a size or stride out of range, a malformed problem */
    WF_ENOMEM = 2,    /* device or host allocation failed */
    WF_ECUDA = 3,     /* a CUDA launch or runtime error (see wf_strerror) */
    WF_ETIMEOUT = 4   /* a bounded device-side wait expired; results are invalid */
};

/* Evaluation path (wf_ctx_set_eval_path). */
enum {
    WF_PATH_AUTO = 0,     /* the shared-memory sweeps, the exact int64 path for what they hand on (the default) */
    WF_PATH_INT64 = 1,    /* every plan on the exact int64 path (a thread per plan, state in global memory) */
    WF_PATH_WIDE = 2,     /* every plan starts in the 64-bit sweep */
    WF_PATH_RELATIVE = 3  /* every plan starts in the sweep with 32-bit times relative to a per-plan base */
};

/* Reclamation order (wf_ctx_set_reclaim). */
enum {
    WF_RECLAIM_LRU = 0,      /* least recently used first (the default) */
    WF_RECLAIM_NEXT_USE = 1  /* redundant copies, then farthest next use per reload cost, then LRU */
};

/* Plan status bits (wf_eval_out.status). */
enum {
    WF_ST_DEVICE = 1u,      /* some place[n] >= D */
    WF_ST_CAPACITY = 2u,    /* some peak[n][place[n]] > cap[place[n]] (Eq. 8) */
    WF_ST_PERMUTATION = 4u, /* order is not a permutation of 0..N-1 */
    WF_ST_TOPOLOGY = 8u,    /* an edge u -> v with v dispatched before u (Eq. 9-10);
                               examined only when WF_ST_PERMUTATION is clear */
    WF_ST_TABLES = 16u      /* wf_eval_plans_static only: the problem tables failed its
                               device check, so no plan of the batch was evaluated */
};

typedef struct wf_ctx wf_ctx;

/*
 * One planning window (Section 3.2) and its cost tables (Eq. 1).
 *
 *   N activations (1..65535), D devices (1..32), M models (1..16),
 *   W sessions (>= 1, every session owns >= 1 activation).
 *   pred_off[N+1], pred_idx[E=pred_off[N]]: CSR lists of graph predecessors
 *     (acyclic, no self-loops, no duplicates, never across sessions).
 *   model[N] < M: deployment identity of each activation (Section 3.2).
 *   session[N] < W; arrival_us[W] >= 0: session arrival times.
 *   lat_us[N*D] >= 0: predicted run time of activation n on device d.
 *   peak_mib[N*D] >= weight_mib[model[n]]: predicted peak memory; the
 *     activation's KV / request memory is peak - weight.  Every activation
 *     must fit (peak <= cap) on at least one device.
 *   weight_mib[M] >= 1, load_us[M*D] >= 0, cap_mib[D] >= 1.
 *   grant_us >= 0: admission overhead charged once per scheduling unit.
 *   S >= 0: latency samples per plan (0 = deterministic).  For S > 0 the run
 *     time of activation n in sample s of plan p is
 *       (lat * bm_e[zq + (bm_en-1)/2] + 2^15) >> 16,
 *     h  = mix(mix(mix(seed ^ p) ^ s) ^ n)   (mix = SplitMix64 output),
 *     zq = floor(bm_r[h & (bm_rn-1)] * bm_c[(h >> 32) & (bm_cn-1)] / 2^18);
 *     bm_rn and bm_cn must be powers of two, bm_en odd and large enough
 *     for every zq, bm_e >= 0.  Ignored when S == 0.
 *   margin_mib >= 0: the admission margin epsilon_M of Section 3.3 (memory
 *     reserved for admission = predicted peak + margin).  Every capacity
 *     check -- a node fitting a device (Eq. 8) and the admission of a unit
 *     (Eq. 11) -- uses peak + margin_mib in place of peak.
 */
typedef struct {
    int32_t N, D, M, W;
    const int32_t *pred_off;
    const int32_t *pred_idx;
    const uint8_t *model;
    const int32_t *session;
    const int64_t *arrival_us;
    const int32_t *lat_us;
    const int32_t *peak_mib;
    const int32_t *weight_mib;
    const int32_t *load_us;
    const int32_t *cap_mib;
    int32_t grant_us;
    int32_t S;
    uint64_t seed;
    const int32_t *bm_r, *bm_c, *bm_e;
    int32_t bm_rn, bm_cn, bm_en;
    int32_t margin_mib;
} wf_problem;

/*
 * A batch of P candidate plans (Eq. 6-10), DEVICE pointers, caller-owned.
 *   place[p*place_stride + n]: device of activation n (uint8).
 *   order[p*order_stride/2 + i]: activation dispatched at position i (uint16).
 *   fuse / prefetch / retain[p*bits_stride/4 + (n>>5)] bit (n&31): the
 *     plan's fusion (Eq. 3-4), prefetch (Eq. 5) and retain bits of n.
 *     retain may be NULL (every model retained after its units).
 *   Strides are in bytes and multiples of 16; place_stride >= N,
 *   order_stride >= 2N, bits_stride >= 4*ceil(N/32).  Base pointers must be
 *   16-byte aligned, and each array spans P whole rows of its stride (the
 *   kernels read rows in 16-byte pieces, up to the row's padding).  plan_base is the global index of row 0 (it seeds the
 *   latency samples, so shards of one batch reproduce the whole batch).
 */
typedef struct {
    int64_t P;
    int64_t plan_base;
    const uint8_t *place;
    int64_t place_stride;
    const uint16_t *order;
    int64_t order_stride;
    const uint32_t *fuse;
    const uint32_t *prefetch;
    const uint32_t *retain;
    int64_t bits_stride;
} wf_plans;

/* Per-plan results, DEVICE pointers [P], caller-owned. */
typedef struct {
    int64_t *makespan_us;  /* last finish - first arrival (Section 4.2) */
    int64_t *p95_us;       /* nearest-rank 95th percentile of session completion latency */
    int64_t *gpu_us;       /* summed device occupancy: loading + generating + idle resident (Section 4.3) */
    uint32_t *status;      /* WF_ST_* bits; a nonzero status sets the three metrics to INT64_MAX */
} wf_eval_out;

/*
 * Validate a problem on the host without touching a GPU.  Returns WF_OK or
 * WF_EINVAL (with a reason retrievable through wf_last_error()).
 */
int wf_problem_check(const wf_problem *prob);

/*
 * Validate *prob, derive the fusible edges of Eq. 3 (succ(u) = {v},
 * pred(v) = {u}, same model) and the topological levels, and copy every
 * table to device `device`.  Scratch for up to max_P plans per call is
 * allocated here (and only here).  On success *out owns all device memory it
 * allocated.  Returns WF_OK, WF_EINVAL, WF_ENOMEM or WF_ECUDA.
 */
int wf_ctx_create(const wf_problem *prob, int device, int64_t max_P, wf_ctx **out);

/*
 * Release forecast of Eq. 2 over the window, free of contention and loads:
 *   rel[n]  = max(arrival[session[n]], max over preds v of comp[v])
 *   comp[n] = rel[n] + min over devices d with peak[n][d] <= cap[d] of lat[n][d]
 * rel_dev and comp_dev are DEVICE int64 [N].  Asynchronous on `stream`.
 */
int wf_forecast_readiness(wf_ctx *ctx, int64_t *rel_dev, int64_t *comp_dev, void *stream);

/*
 * Evaluate plans->P plans (0 < P <= max_P).  Per plan: the status bits;
 * then fused chains (Eq. 3-4), releases (Eq. 2, Eq. 7), per-device order
 * (Eq. 10), least-recently-used reclamation so that resident weights plus
 * the unit's KV fit at every admission (Eq. 11, Section 3.5), loads and
 * prefetches on the consumer's device (Eq. 5, Eq. 9), retain / reclaim, and
 * the three metrics; for S > 0 the floor means over samples and the pooled
 * p95.  Asynchronous on `stream`.  Returns WF_EINVAL for bad sizes, strides
 * or alignment, WF_ECUDA for a launch error.
 */
int wf_eval_plans(wf_ctx *ctx, const wf_plans *plans, const wf_eval_out *out, void *stream);

/*
 * The k best of P evaluated plans (1 <= k <= min(P, 1024), P <= max_P) by the
 * key (status != 0, makespan, p95, gpu, plan index), ascending -- the
 * single-objective analog of the ranking key of Eq. 12.  ids_dev: DEVICE
 * int32 [k] plan indices (0-based within the batch); keys_dev: DEVICE int64
 * [k][3] (makespan, p95, gpu) or NULL.  Asynchronous on `stream`.
 */
int wf_topk(wf_ctx *ctx, const wf_eval_out *res, int64_t P, int32_t k,
            int32_t *ids_dev, int64_t *keys_dev, void *stream);

/*
 * One step of the hot path from and to HOST memory: copy a batch of plans
 * in, optionally forecast readiness (as wf_forecast_readiness), evaluate the
 * batch (as wf_eval_plans) and select its k best (as wf_topk), then copy the
 * results out.  host_plans has the layout of wf_plans, but its five arrays
 * are HOST pointers (retain may be NULL); its strides need only be >= the
 * row sizes and multiples of 16 bytes.  ids_host: int32 [k]; keys_host: int64
 * [k][3] or NULL; out_host: every plan's metrics and status ([P] each, HOST
 * pointers) or NULL; rel_host / comp_host: int64 [N] each, both or neither
 * (neither: no forecast).  1 <= k <= min(P, 1024), P <= max_P.
 *
 * The context copies the plans into one of two device staging slots on a
 * copy stream of its own, and calls alternate between the slots, so a call's
 * copy overlaps the previous call's evaluation on `stream`; each copy first
 * waits for the call that last used its slot.  The forecast, which depends on
 * the window only, runs on the copy stream too.  The results are in host
 * memory once `stream` has passed the call (synchronize or record an event
 * after it).  The host plan arrays must stay unchanged until the call's copy
 * has run (at the latest, when `stream` has passed the call).  Host memory
 * should be page-locked (cudaHostAlloc, or a pinned torch tensor); pageable
 * memory works, but then its copies do not overlap the GPU's work.  Under
 * stream capture the copies go on `stream` itself (page-locked memory
 * only).  The device results, top-k and forecast buffers are single, so the
 * calls on one context must all use one stream.  The staging (two slots of
 * max_P plan rows, the results, the forecast) is allocated by the first call
 * or by wf_ctx_reserve_host, and freed with the context.  Returns WF_OK,
 * WF_EINVAL, WF_ENOMEM or WF_ECUDA.
 */
int wf_eval_topk_host(wf_ctx *ctx, const wf_plans *host_plans, int32_t k, int32_t *ids_host,
                      int64_t *keys_host, const wf_eval_out *out_host, int64_t *rel_host,
                      int64_t *comp_host, void *stream);

/*
 * Allocate wf_eval_topk_host's staging now (see above), so that no call of
 * it allocates.  Returns WF_OK, WF_ENOMEM or WF_ECUDA; a second call does
 * nothing.
 */
int wf_ctx_reserve_host(wf_ctx *ctx);

/*
 * The paper has no counterpart to this entry point; it serves callers that
 * cannot allocate device memory when they score plans -- for example a
 * scheduler inside a serving engine that reserved nearly all GPU memory up
 * front for weights and KV cache, where another cudaMalloc fails or eats into
 * the cache -- or whose device memory belongs to an allocator that must not
 * be bypassed.
 *
 * Same results as wf_eval_plans with least-recently-used reclamation (the
 * default of a context) for a deterministic problem (S must be 0), without a
 * context and without allocating anything: every table of *prob is a DEVICE
 * pointer here (same layouts as above), plans and outputs are DEVICE
 * pointers as for wf_eval_plans.  Before anything is indexed by them, a
 * device check confirms model < M, 0 <= session < W, pred_off starting at 0
 * and non-decreasing, 0 <= pred_idx < N without self-loops, non-negative run
 * times, loads and arrivals, weights and capacities >= 1 and peak >= weight;
 * when it fails, every plan of the batch gets status WF_ST_TABLES and
 * INT64_MAX metrics, and wf_static_status reports it.  (Acyclicity,
 * duplicate or cross-session edges and "every activation fits somewhere" are
 * not checked: the caller guarantees them, as wf_problem_check does for a
 * context; pred_off[N] must be the length of pred_idx.)
 * Scratch is a 32 MiB file-scope device array that every GPU loading this
 * library holds until the process exits.  A call needs 256 B, plus three
 * tables of 4*N bytes each rounded up to 256 B, plus one state row per plan
 * of 8*(N + W + 3*D) + 4*D*(M + 3) bytes rounded up to 128 B; a batch that
 * does not fit returns WF_EINVAL naming the largest batch that does (about
 * 1,900 plans of a 2,000-activation window) -- split larger batches by
 * plan_base.  Each call made outside stream capture looks the array's
 * address up (cudaGetSymbolAddress) with the current device; a call under
 * capture reuses the address of the last call outside capture on that
 * device, so make one call before capturing, and again after a device
 * reset.  All calls share the array and each call re-initialises what it
 * relies on; calls that overlap on the GPU (other streams, other threads)
 * race on it and must be serialised by the caller.  Asynchronous on
 * `stream`; returns WF_OK, WF_EINVAL or WF_ECUDA.
 */
int wf_eval_plans_static(const wf_problem *prob, const wf_plans *plans, const wf_eval_out *out,
                         void *stream);

/*
 * The paper has no counterpart to this call either: the device-side outcome
 * of the last wf_eval_plans_static call on the current device.  Synchronizes
 * `stream`, reads the static array's error word (no allocation) and clears
 * it: WF_OK, WF_EINVAL when the problem tables failed the device check, or
 * WF_ECUDA when an evaluation hit a state no valid plan reaches.
 */
int wf_static_status(void *stream);

/*
 * Local search around the best plans.  The paper's scheduler re-ranks its
 * uncommitted decisions whenever arrivals, completions or model transitions
 * change the picture (Section 3.5); these calls search the neighbourhood of
 * the k best evaluated plans (the elite) for better ones.  All plan and
 * result pointers are DEVICE pointers owned by the caller; parents and
 * children are separate buffers that must not overlap, and either both or
 * neither carry retain rows.  Asynchronous on `stream`; no allocation.
 *
 * wf_mutate_plans: children->P children.  Child c copies parent
 * c mod parents->P and then takes n_ops (0..4096) changes in turn; change s
 * is decoded from h = mix(mix(mix(seed ^ round) ^ c) ^ s) (mix = SplitMix64
 * output), x = bits 8..39 of h, y = bits 40..63:
 *   h mod 4 = 0  place[n] for n = x mod N becomes the (y mod f)-th, in
 *               ascending order, of the f devices whose capacity holds
 *               peak[n][d] (Eq. 8);
 *             1  flip fuse bit n = x mod N (Eq. 3);
 *             2  flip prefetch bit n = x mod N (Eq. 5);
 *             3  swap dispatch positions i = x mod (N - 1) and i + 1 unless
 *               the node at i is a graph predecessor of the node at i + 1
 *               (Eq. 10); no change when N = 1 or order[i + 1] >= N.
 * Retain rows are copied.  Children of valid plans are valid.  Returns
 * WF_EINVAL for bad sizes, strides, alignment or n_ops.
 *
 * wf_merge_elite: elite->P = k (1..1024) evaluated plans and
 * children->P evaluated children, k + children->P <= max_P.  The union is
 * ranked by the wf_topk key with the elite at indices 0..k-1 and child c at
 * k + c (so ties keep elite plans); the k best stay.  An elite slot whose
 * plan stays is untouched; the slots whose plans left, in ascending order,
 * receive the entering children in key order (rows and results).
 *
 * wf_local_search: `rounds` times: wf_mutate_plans(elite -> children, round
 * = round0 + r), wf_eval_plans(children), wf_merge_elite.  The elite's
 * results must be those of its plans on entry.
 */
int wf_mutate_plans(wf_ctx *ctx, const wf_plans *parents, const wf_plans *children, uint64_t seed,
                    int64_t round, int32_t n_ops, void *stream);
int wf_merge_elite(wf_ctx *ctx, const wf_plans *elite, const wf_eval_out *elite_res,
                   const wf_plans *children, const wf_eval_out *child_res, void *stream);
int wf_local_search(wf_ctx *ctx, const wf_plans *elite, const wf_eval_out *elite_res,
                    const wf_plans *children, const wf_eval_out *child_res, uint64_t seed,
                    int64_t round0, int32_t rounds, int32_t n_ops, void *stream);

/*
 * Plan construction: Algorithm 1 (rank the ready units, bind each to one
 * feasible device, load / prefetch, Section 3.5) read as a list scheduler
 * over the whole window, one plan per row of *out (DEVICE pointers, the
 * layout of wf_plans; out->P plans).  Repeatedly:
 *   - the ready node (every graph predecessor dispatched) with the smallest
 *     (release + jitter, node id) goes next; release = max(session arrival,
 *     predecessor finishes) (Eq. 2);
 *   - its device is the one, among those whose capacity holds it (Eq. 8),
 *     with the smallest predicted finish + jitter (ties: lower device): a
 *     resident model starts at max(device free, release); a missing one is
 *     loaded first, from max(device free, arrival) when the device is free
 *     before the release (the prefetch bit is then set), else from
 *     max(device free, release);
 *   - its fusible chain (Eq. 3) follows it on that device while each next
 *     member fits there (fuse bits 1), and the unit is played forward with
 *     the rules of wf_eval_plans (reclamation, Eq. 11), so evaluating the
 *     plan reproduces the constructor's timeline.
 * Jitter of plan index g = out->plan_base + p: h = mix(mix(seed ^ g) ^ node),
 * rank jitter h mod (jitter_us + 1), device jitter mix(h ^ (d + 1)) mod
 * (jitter_us + 1); jitter_us = 0 makes every plan the plain greedy one.
 * Retain rows, if given, are set to all ones.  WF_EINVAL when the window's
 * horizon (latest arrival + every node's worst load + run + grant) plus
 * jitter_us reaches 2^47 us.  The first call on a context allocates the
 * constructor's state (about 20 N bytes per plan built at once, at most
 * 128 plans per SM); later calls allocate nothing.  Asynchronous on stream.
 */
int wf_construct_plans(wf_ctx *ctx, const wf_plans *out, uint64_t seed, int64_t jitter_us, void *stream);

/*
 * Reclamation order of the context's evaluations (Eq. 11 admission).  The
 * paper reclaims idle replicas preferring redundant copies, then distant next
 * use relative to reload cost, with least-recently-used order as the fallback
 * (Section 3.5).  WF_RECLAIM_LRU (the default) evicts least recently used
 * first.  WF_RECLAIM_NEXT_USE evicts, one at a time until the unit fits:
 * first a model also resident on another device; among equals the one whose
 * next use on this device (the next dispatch position whose unit runs that
 * model there; none = infinitely far) lies farthest from the current position
 * per microsecond of its reload cost (a zero cost counts as infinitely far);
 * among equals the least recently used.  The next-use policy needs S = 0, a
 * window the shared-memory sweep holds, and fusible chains whose run time
 * stays below 2^32 us; otherwise WF_EINVAL.  The first switch to it allocates
 * a [max_P][N] u16 table.  Not thread-safe with calls in flight on the
 * context.  wf_eval_plans_static always uses WF_RECLAIM_LRU.
 */
int wf_ctx_set_reclaim(wf_ctx *ctx, int32_t policy);

/*
 * wf_eval_plans, plus the window terms of the ranking key of Eq. 12.  That
 * key ranks a tick's partial plan by (-A_1, ..., -A_K, C_F, -P_N, H_life);
 * over a whole window every unit is admitted, so the coverage counts A_k are
 * equal for all valid plans and it reduces to (C_F, -P_N, H_life), C_F the
 * latest completion (the makespan's order).  Per plan:
 *   timely_dev[p]  P_N: the units whose model load ran under their prefetch
 *                  bit (Eq. 5), started before the unit's release and ended
 *                  by it;
 *   life_dev[p]    H_life (us): over the units, the delay the load adds to
 *                  the start, max(load end, release) - max(device free,
 *                  release) (0 on a hit), plus the load time of every load of
 *                  a model its device held before (a reload after reclamation,
 *                  Eq. 11 or a retain bit of 0).
 * Both are INT64_MAX for an invalid plan.  DEVICE int64 [P] each.  Needs
 * S = 0 (WF_EINVAL otherwise); either reclamation order.  The context carries
 * the two pointers during the call, so calls on one context are not
 * thread-safe.  Otherwise as wf_eval_plans.
 */
int wf_eval_plans_phi(wf_ctx *ctx, const wf_plans *plans, const wf_eval_out *out, int64_t *timely_dev,
                      int64_t *life_dev, void *stream);

/*
 * The k best plans by Eq. 12's window key (status != 0, makespan, -timely,
 * life, plan index), ascending, from wf_eval_plans_phi's outputs.  keys_dev:
 * DEVICE int64 [k][3] (makespan, timely, life) or NULL.  Otherwise as
 * wf_topk.
 */
int wf_topk_phi(wf_ctx *ctx, const wf_eval_out *out, const int64_t *timely_dev, const int64_t *life_dev, int64_t P,
                int32_t k, int32_t *ids_dev, int64_t *keys_dev, void *stream);

/*
 * Synchronize `stream` and report device-side failures of earlier calls on
 * this context (WF_ETIMEOUT when a bounded wait expired), clearing them.
 */
int wf_ctx_status(wf_ctx *ctx, void *stream);

/*
 * Diagnostic: launches, on `stream`, one device-side bounded wait that
 * nothing completes (an mbarrier armed for bytes that no copy delivers, the
 * wait the bulk-copy kernels use).  It gives up after 2^20 polls of about
 * 4 us each (about 4 s on a GB300) and
 * records the expiry, so the next wf_ctx_status returns WF_ETIMEOUT; the
 * context stays usable.  Returns WF_EINVAL for a NULL context, WF_ECUDA when
 * the launch fails.
 */
int wf_ctx_check_wait_expiry(wf_ctx *ctx, void *stream);

/*
 * Which kernels later evaluation calls on this context use.  All give the
 * same results.
 *   WF_PATH_AUTO (default): the 32-bit sweep, which hands a plan whose times
 *     reach 2^32 us to the 64-bit sweep; once more than half of a batch has
 *     left 32 bits, later calls start every plan in the relative sweep
 *     (below), or in the 64-bit sweep where that does not apply.
 *   WF_PATH_INT64: every plan on the exact int64 path (slower; for tests and
 *     cross-checks of the sweeps).
 *   WF_PATH_WIDE: every plan starts in the 64-bit sweep.
 *   WF_PATH_RELATIVE: every plan starts in the relative sweep: 32-bit times
 *     counted from a per-plan base that rises with the plan's devices' free
 *     times, so a window whose times run far past 2^32 us still plays on
 *     32-bit arithmetic; a plan whose times leave 32 bits even so goes on to
 *     the 64-bit sweep.  Calls under next-use reclamation or for Eq. 12's
 *     terms, and contexts too small for its scratch rows, start as
 *     WF_PATH_WIDE.
 * A unit whose summed run time saturates 32 bits always goes on to the int64
 * path.  Not thread-safe with calls in flight on the context.  Returns
 * WF_EINVAL for a NULL context or another value, and for WF_PATH_RELATIVE or
 * WF_PATH_WIDE when the window does not fit those sweeps' shared memory.
 */
int wf_ctx_set_eval_path(wf_ctx *ctx, int32_t path);

/*
 * Replica batch limit B_q (Eq. 11 and the batch limit stated with it,
 * Section 3.5) for later evaluation calls on this context; 0 (the default)
 * keeps one unit at a time per device.  With B_q >= 1 a device runs units of
 * one replica (a model resident on it) at a time, up to B_q of them at once:
 * units are admitted in dispatch order; a unit of the device's current
 * replica takes the slot that frees earliest, no earlier than its release
 * and the device's latest admission, once resident weights + the KV needs
 * of the units still running + its own KV fit the capacity (idle models are
 * reclaimed least recently used first; if that is not enough the unit waits
 * for the next running unit to end); a unit of another model waits for the
 * device to drain, then hits or loads as without the limit.  B_q = 1 gives
 * the same results as 0.  Deterministic problems with least-recently-used
 * reclamation only.  Evaluation calls then play the plans in a shared-memory
 * sweep of their own (the exact int64 path for a unit whose summed run time
 * saturates 32 bits, or for every plan when the window's state does not fit
 * a CTA), and reject retain rows when B_q > 1 and the window terms of Eq. 12
 * (WF_EINVAL).  The first increase may reallocate the evaluation
 * scratch; not thread-safe with calls in flight on the context.  Returns
 * WF_EINVAL for a value outside 0..64 or such a problem.
 */
int wf_ctx_set_batch(wf_ctx *ctx, int32_t batch);

/* Release every device and host allocation of the context (NULL is a no-op). */
void wf_ctx_destroy(wf_ctx *ctx);

/* Static description of a return code. */
const char *wf_strerror(int code);

/* Thread-local detail of the last WF_EINVAL / WF_ECUDA on this thread. */
const char *wf_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* WF_H */
