// Internal definitions shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <cstdint>
#include <vector>

#include "../../include/wf.h"

#define WF_INF64 INT64_MAX

// Device-resident copy of a problem plus derived tables.  Owned by wf_ctx.
struct wf_dev_problem {
    int32_t N, D, M, W, E;
    int32_t grant;
    int32_t S;
    uint64_t seed;
    int32_t bm_rn, bm_cn, bm_en;
    int64_t first_arrival;      // min over sessions of arrival_us
    const int32_t *pred_off;    // [N+1]
    const int32_t *pred_idx;    // [E]
    const int32_t *fnext;       // [N] fusible successor (Eq. 3) or -1
    const int32_t *fprev;       // [N] fusible predecessor (Eq. 3) or -1
    const uint8_t *model;       // [N]
    const int32_t *session;     // [N]
    const int64_t *arrival;     // [W]
    const int32_t *lat;         // [N][D]
    const int32_t *peak;        // [N][D]
    const int32_t *weight;      // [M]
    const int32_t *load;        // [M][D]
    const int32_t *cap;         // [D]
    const int32_t *lev_off;     // [nlev+1] topological levels
    const int32_t *lev_nodes;   // [N]
    int32_t nlev;
    const int32_t *bm_r, *bm_c, *bm_e;
    const int16_t *bm_r16, *bm_c16;  // bm_r, bm_c as int16 when every value fits (else null)
    int *err;                   // device error word (0 = ok)

    // Finish-time slots of the per-plan sweep (see wf_slots.cpp).  Slots
    // [0, W) hold the sessions' latest finish; the others carry release
    // times from producers to consumers.
    int32_t nslots;             // 0 when the slot sweep is not usable
    const int4 *noderec;        // [2N]: {fprev, fnext, rslot code, model | session << 8},
                                //       {write-list start, length, first two codes, 0}
    const int32_t *wl_off;      // [N+1] write list of each node when it ends a unit
    const uint16_t *wl;         // [wl_off[N]] slot | (max-accumulate << 15)
    const int2 *lk;             // [N][D] {run time, KV need = peak - weight}
    const uint32_t *links;      // [N] fusible predecessor | fusible successor << 16 (0xFFFF = none)
    const uint4 *hrec;          // [N] {links, release slot | model << 16 | writes << 20, arrival, codes 0 | 1 << 16}
    const uint32_t *wc23;       // [N] third | fourth << 16 write code of each node's write list (the sink slot when shorter)
    const uint32_t *fitmask;    // [N rounded up to 16] bit d: peak[n][d] <= cap[d]
    const uint8_t *fit8;        // [N rounded up to 16] the low byte of fitmask (all of it when D <= 8)
    const uint32_t *edges;      // [E rounded up to 4] predecessor | successor << 16
    const int32_t *succ_off;    // [N+1] successor lists (CSR)
    const int32_t *succ_idx;    // [E]
    int64_t horizon;            // no finish of any plan exceeds this (latest arrival + every node's worst load + run + grant)
    // Reclamation order (0: least recently used; 1: by next use) and, for 1,
    // the next use of each unit's model on its device: [max_P][N] dispatch
    // positions (0xFFFF = none), filled per call.
    int32_t reclaim;
    uint16_t *nextuse;
    // Replica batch limit B_q (wf_ctx_set_batch): 0 = one unit at a time per
    // device (the sweeps); >= 1 = up to B_q units of a device's current
    // replica at once, played by the int64 path.
    int32_t batch;
    int64_t max_chain_run;      // the longest fusible chain's run time on its slowest devices, plus the grant
    // Outputs of the window terms of Eq. 12 ([P] each, wf_eval_plans_phi);
    // null outside such a call.
    int64_t *phi_timely;
    int64_t *phi_life;
    // The relative-time sweep's exact session finishes that fell below a
    // plan's base, [W][CTAs x plans per CTA]: the context's evaluation
    // scratch, set for that launch only.
    uint64_t *rel_ret;
    int64_t max_arrival;
};

// rslot code of noderec.z: -1 = no predecessor (release = arrival), else the
// slot index, with bit 30 set when the slot is an accumulator that the
// reader resets to 0 after reading.
#define WF_RSLOT_ACC (1 << 30)

struct wf_ctx {
    int device;
    int64_t max_P;
    wf_dev_problem dp;
    void *tables;               // one device allocation holding every table
    size_t tables_bytes;
    void *eval_scratch;         // per-simulation state (and sample pools)
    size_t eval_scratch_bytes;
    int64_t eval_threads;       // launch units (plans, or sample CTAs) the scratch holds
    size_t eval_row_bytes;
    void *topk_scratch;
    size_t topk_scratch_bytes;
    int *err;
    int sms;                    // streaming multiprocessors of the device
    bool force_int64;           // wf_ctx_set_eval_path(WF_PATH_INT64): every plan on the int64 path
    int32_t start_path;         // wf_ctx_set_eval_path's value (WF_PATH_WIDE / RELATIVE: the first sweep)
    int32_t *ovf_count;         // [2]: plans the u32 sweep hands on, plans left for the int64 path (the sweep
                                // calls use words 0-1 and 2-3 in turn)
    int32_t *ovf_list;          // [max_P] the u32 sweep's hand-offs (and the stochastic sweep's)
    int32_t *ovf_list2;         // [max_P] plans for the int64 path
    // Path choice from an earlier call: when more than half of a batch left
    // 32 bits, later calls start past the u32 sweep (the relative sweep, or
    // the u64 one).  The count is read back through pinned memory and an
    // event, never waited for.
    bool prefer_wide;
    bool wide_pending;
    int64_t wide_P;
    int ovf_pair;               // the pair of ovf_count words the last sweep call used (0 or 1)
    int rb_pair;                // the pair whose count the pending read-back copies
    void *search_scratch;       // local search: the union's results [max_P], top-k ids, slot pairs
    void *construct_scratch;    // plan constructor: per-plan state of the plans built at once, allocated by its first call
    int64_t construct_threads;  // plans built at once (a warp each)
    int32_t *h_ovf;             // pinned host copy of ovf_count[0]
    cudaEvent_t sweep_done;     // recorded on the caller's stream after the sweeps
    cudaEvent_t ovf_event;      // recorded on side after the read-back
    cudaStream_t side;          // the read-back's own stream, off the caller's critical path
    struct wf_host_stage *host; // wf_eval_topk_host's staging (wf_host.cu), made by its first use
};

// Frees wf_eval_topk_host's staging once its copies have finished (wf_host.cu).
void wf_host_release(wf_ctx *c);

// Static slot assignment (wf_slots.cpp).  Fills rslot code per node, write
// lists (CSR) and returns the slot count, or -1 when it exceeds 32767.
int32_t wf_assign_slots(int32_t N, int32_t W, const int32_t *pred_off, const int32_t *pred_idx,
                        const int32_t *session, const int32_t *fprev, const int32_t *fnext,
                        int32_t *rslot, std::vector<int32_t> &wl_off, std::vector<uint16_t> &wl);

// Error plumbing and argument checks (wf_ctx.cu).
int wf_set_error(int code, const char *fmt, ...);
int wf_cuda_check(cudaError_t e, const char *what);
int wf_check_plans(const wf_ctx *c, const wf_plans *pl, const char *what);
int wf_check_out(const wf_eval_out *out, const char *what);
int wf_select_device(const wf_ctx *c);

// Launchers (one per translation unit).
int wf_launch_forecast(wf_ctx *ctx, int64_t *rel, int64_t *comp, cudaStream_t st);
int wf_launch_eval(wf_ctx *ctx, const wf_plans *plans, const wf_eval_out *out, cudaStream_t st);
// The k best plans by (invalid, makespan, term2, term3, index); term2 and
// term3 default to p95 and GPU time, and sign2 = -1 ranks term2 largest
// first (the timely prefetches of Eq. 12).
int wf_launch_topk(wf_ctx *ctx, const wf_eval_out *res, int64_t P, int32_t k, int32_t *ids,
                   int64_t *keys, cudaStream_t st, const int64_t *term2 = nullptr, const int64_t *term3 = nullptr,
                   int64_t sign2 = 1);
size_t wf_eval_row_bytes(const wf_dev_problem &dp);
size_t wf_eval_scratch_bytes(const wf_dev_problem &dp, int64_t max_P, int64_t *units);
size_t wf_topk_scratch_bytes(int64_t max_P);
size_t wf_search_scratch_bytes(int64_t max_P);
// The shared-memory sweeps that apply to a problem: u32 times with 16 plans
// per CTA, u64 times with plans64 plans per CTA, and relative u32 times with
// plansRel plans per CTA (0 bytes = not usable); res32 / res64 / resRel are
// the CTAs of each resident on one SM.
struct wf_sweep_cfg {
    size_t smem32;
    size_t smem64;
    size_t smemRel;
    int plans64;
    int plansRel;
    int res32;
    int res64;
    int resRel;
};
wf_sweep_cfg wf_sweep_config(const wf_dev_problem &dp);
int wf_launch_nextuse(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, cudaStream_t st);
size_t wf_stoch_smem(const wf_dev_problem &dp);
size_t wf_batch_smem(const wf_dev_problem &dp);
int wf_launch_batch(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, size_t smem, int32_t *ovf_list,
                    int32_t *ovf_count, cudaStream_t st);
int wf_launch_stoch(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, size_t smem,
                    int32_t *ovf_list, int32_t *ovf_count, cudaStream_t st);
// Status pass, then the sweeps (u32 first unless wide_first; then the
// relative sweep where it applies and the context's path is not
// WF_PATH_WIDE, else u64); on return *rest_list / *rest_count name the plans
// left for the int64 path.
int wf_launch_sweep(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, const wf_sweep_cfg &cfg,
                    bool wide_first, int32_t *counts, int32_t *list1, int32_t *list2, cudaStream_t st,
                    const int32_t **rest_list, const int32_t **rest_count);
