// Plan evaluation (rows a3-a11): status bits, then a list-schedule play of
// each plan over the window with fused chains (Eq. 3-4), releases (Eq. 2,
// Eq. 7), per-device order (Eq. 10), LRU residency under capacity (Eq. 11),
// loads / prefetches on the consumer's device (Eq. 5, Eq. 9), retain /
// reclaim and the metrics of Section 4.2-4.3.
//
// Mapping: one thread plays one (plan, sample).  Its mutable state (chain-tail
// finish times, per-device and per-session state) lives in a scratch row of
// the context; plans beyond the number of rows are taken in rounds.  For
// wf_eval_plans_phi a deterministic play also returns the window terms of
// Eq. 12's ranking key (timely prefetches, lifecycle overhead).
#include <algorithm>
#include <mutex>

#include "wf_internal.cuh"

namespace {

constexpr int kEvalThreads = 128;
constexpr int kSampleThreads = 64;
constexpr int64_t kNone = INT64_MIN;

struct PlanRows {
    const uint8_t *place;
    const uint16_t *order;
    const uint32_t *fuse;
    const uint32_t *prefetch;
    const uint32_t *retain;  // NULL = all retained
};

__device__ __forceinline__ bool bit_at(const uint32_t *row, int32_t n)
{
    return (__ldg(row + (n >> 5)) >> (n & 31)) & 1u;
}

__device__ __forceinline__ PlanRows plan_rows(const wf_plans &pl, int64_t p)
{
    PlanRows r;
    r.place = pl.place + p * pl.place_stride;
    r.order = (const uint16_t *)((const uint8_t *)pl.order + p * pl.order_stride);
    r.fuse = (const uint32_t *)((const uint8_t *)pl.fuse + p * pl.bits_stride);
    r.prefetch = (const uint32_t *)((const uint8_t *)pl.prefetch + p * pl.bits_stride);
    r.retain = pl.retain ? (const uint32_t *)((const uint8_t *)pl.retain + p * pl.bits_stride) : nullptr;
    return r;
}

// Scratch row of one simulation.
struct Row {
    int64_t *ctail;   // [N] finish time of chain tails (also holds int32 positions for the status check)
    int64_t *tfree;   // [D] device free time
    int64_t *occ;     // [D] start of the current occupancy interval, kNone if empty
    int64_t *gpu;     // [D] closed occupancy
    int64_t *comp;    // [W] latest finish per session
    int32_t *used;    // [D] resident weights
    int32_t *nres;    // [D] resident model count
    int32_t *stamp;   // [D][M] last dispatch position + 1 using the model, 0 = not resident
    int32_t *loaded;  // [D] bit m: model m was ever resident on the device (Eq. 12 window terms)
    // With a replica batch limit B = dp.batch (only then laid out):
    int64_t *slot_end;  // [D][B] when each slot of the device's current replica frees
    int64_t *slot_kv;   // [D][B] KV need of the unit in each slot
    int64_t *last_adm;  // [D] the device's latest admission
    int32_t *cur;       // [D] model of the device's current replica, -1 for none
};

__device__ __forceinline__ size_t up8(size_t x) { return (x + 7) & ~(size_t)7; }

__device__ __forceinline__ Row row_at(const wf_dev_problem &dp, uint8_t *base)
{
    Row r;
    size_t o = 0;
    r.ctail = (int64_t *)(base + o); o += up8(8 * (size_t)dp.N);
    r.tfree = (int64_t *)(base + o); o += 8 * (size_t)dp.D;
    r.occ = (int64_t *)(base + o); o += 8 * (size_t)dp.D;
    r.gpu = (int64_t *)(base + o); o += 8 * (size_t)dp.D;
    r.comp = (int64_t *)(base + o); o += 8 * (size_t)dp.W;
    r.used = (int32_t *)(base + o); o += up8(4 * (size_t)dp.D);
    r.nres = (int32_t *)(base + o); o += up8(4 * (size_t)dp.D);
    r.stamp = (int32_t *)(base + o); o += up8(4 * (size_t)dp.D * dp.M);
    r.loaded = (int32_t *)(base + o); o += up8(4 * (size_t)dp.D);
    if (dp.batch > 0) {
        r.slot_end = (int64_t *)(base + o); o += 8 * (size_t)dp.D * dp.batch;
        r.slot_kv = (int64_t *)(base + o); o += 8 * (size_t)dp.D * dp.batch;
        r.last_adm = (int64_t *)(base + o); o += 8 * (size_t)dp.D;
        r.cur = (int32_t *)(base + o);
    } else {
        r.slot_end = r.slot_kv = r.last_adm = nullptr;
        r.cur = nullptr;
    }
    return r;
}

// Status bits (Eq. 8-10).  Uses the ctail area as an int32 position table.
__device__ uint32_t plan_status(const wf_dev_problem &dp, const PlanRows &pr, Row &row)
{
    const int32_t N = dp.N, D = dp.D;
    uint32_t st = 0;
    for (int32_t n = 0; n < N; ++n) {
        const int32_t d = pr.place[n];
        if (d >= D) st |= WF_ST_DEVICE;
        else if (dp.peak[(int64_t)n * D + d] > dp.cap[d]) st |= WF_ST_CAPACITY;
    }
    int32_t *pos = (int32_t *)row.ctail;
    for (int32_t n = 0; n < N; ++n) pos[n] = -1;
    for (int32_t i = 0; i < N; ++i) {
        const int32_t h = pr.order[i];
        if (h >= N || pos[h] >= 0) { st |= WF_ST_PERMUTATION; continue; }
        pos[h] = i;
    }
    if (!(st & WF_ST_PERMUTATION)) {
        for (int32_t v = 0; v < N && !(st & WF_ST_TOPOLOGY); ++v)
            for (int32_t e = dp.pred_off[v]; e < dp.pred_off[v + 1]; ++e)
                if (pos[dp.pred_idx[e]] > pos[v]) { st |= WF_ST_TOPOLOGY; break; }
    }
    return st;
}

// SplitMix64 output function (Steele, Lea, Flood 2014).
__device__ __forceinline__ uint64_t splitmix(uint64_t x)
{
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
}

// Run time of activation n on device d; for a latency sample, scaled by the
// multiplier drawn from (plan, sample, n) through the integer Box-Muller
// tables (an arithmetic right shift of the signed product is the floor).
template <bool kStoch>
__device__ __forceinline__ int64_t run_time(const wf_dev_problem &dp, int32_t n, int32_t d, uint64_t key)
{
    const int64_t base = dp.lat[(int64_t)n * dp.D + d];
    if (!kStoch) return base;
    const uint64_t h = splitmix(key ^ (uint64_t)n);
    const int64_t r = dp.bm_r[h & (uint64_t)(dp.bm_rn - 1)];
    const int64_t c = dp.bm_c[(h >> 32) & (uint64_t)(dp.bm_cn - 1)];
    const int64_t zq = (r * c) >> 18;
    const int64_t mult = dp.bm_e[zq + ((dp.bm_en - 1) >> 1)];
    return (base * mult + 32768) >> 16;
}

// One play of a valid plan.  Returns makespan and GPU time; per-session
// completion latencies are left in row.comp.  With phi, also the window
// terms of Eq. 12: phi[0] the timely prefetches (a prefetched load that
// starts before the unit's release and ends by it), phi[1] the lifecycle
// overhead (the delay each load adds to its unit's start, plus the load time
// of every reload of a model the device held before).
template <bool kStoch>
__device__ void play(const wf_dev_problem &dp, const PlanRows &pr, Row &row, uint64_t key,
                     int64_t *makespan, int64_t *gpu_total, int64_t *phi = nullptr)
{
    const int32_t N = dp.N, D = dp.D, M = dp.M, W = dp.W;
    int64_t timely = 0, life = 0;
    for (int32_t d = 0; d < D; ++d) {
        row.tfree[d] = 0; row.occ[d] = kNone; row.gpu[d] = 0; row.used[d] = 0; row.nres[d] = 0;
        row.loaded[d] = 0;
    }
    for (int32_t k = 0; k < D * M; ++k) row.stamp[k] = 0;
    for (int32_t w = 0; w < W; ++w) row.comp[w] = kNone;
    int64_t end = 0;

    for (int32_t i = 0; i < N; ++i) {
        const int32_t h = pr.order[i];
        const int32_t d = pr.place[h];
        // A chain member runs inside its head's unit (Eq. 3, Eq. 9).
        const int32_t fp = dp.fprev[h];
        if (fp >= 0 && bit_at(pr.fuse, h) && pr.place[fp] == d) continue;

        const int32_t m = dp.model[h];
        const int32_t w = dp.session[h];
        const int64_t arr = dp.arrival[w];
        int64_t rel = arr;  // Eq. 2 / Eq. 7: the heads' predecessors are chain tails
        for (int32_t e = dp.pred_off[h]; e < dp.pred_off[h + 1]; ++e)
            rel = max(rel, row.ctail[dp.pred_idx[e]]);

        // Extend the chain; admission KV is the largest on it, run time the sum (Eq. 4).
        const int32_t wm = dp.weight[m];
        int32_t tail = h;
        int64_t kv = dp.peak[(int64_t)h * D + d] - wm;
        int64_t run = run_time<kStoch>(dp, h, d, key);
        for (int32_t s = dp.fnext[h]; s >= 0 && bit_at(pr.fuse, s) && pr.place[s] == d; s = dp.fnext[s]) {
            kv = max(kv, (int64_t)dp.peak[(int64_t)s * D + d] - wm);
            run += run_time<kStoch>(dp, s, d, key);
            tail = s;
        }

        // Eq. 11 with LRU reclamation of other models.
        int32_t *st = row.stamp + d * M;
        const bool hit = st[m] != 0;
        const int64_t need = hit ? kv : wm + kv;
        while (row.used[d] + need > dp.cap[d]) {
            int32_t victim = -1, vs = INT32_MAX;
            for (int32_t k = 0; k < M; ++k)
                if (k != m && st[k] != 0 && st[k] < vs) { vs = st[k]; victim = k; }
            if (victim < 0) { atomicExch(dp.err, 2); break; }  // unreachable for a valid plan
            row.used[d] -= dp.weight[victim];
            row.nres[d] -= 1;
            st[victim] = 0;
        }
        const int64_t tf = row.tfree[d];
        int64_t start;
        if (hit) {
            start = max(tf, rel);
        } else {
            const bool pf = bit_at(pr.prefetch, h);
            const int64_t ls = max(tf, pf ? arr : rel);
            if (row.occ[d] == kNone) row.occ[d] = ls;
            row.used[d] += wm;
            row.nres[d] += 1;
            const int64_t le = ls + dp.load[m * D + d];
            start = max(le, rel);
            if (phi) {
                timely += pf && ls < rel && le <= rel;
                if ((row.loaded[d] >> m) & 1) life += dp.load[m * D + d];
                row.loaded[d] |= 1 << m;
            }
        }
        if (phi) life += start - max(tf, rel);
        const int64_t c = start + dp.grant + run;
        row.ctail[tail] = c;
        row.tfree[d] = c;
        st[m] = i + 1;
        end = max(end, c);
        row.comp[w] = max(row.comp[w], c);
        if (pr.retain && !bit_at(pr.retain, tail)) {
            row.used[d] -= wm;
            row.nres[d] -= 1;
            st[m] = 0;
            if (row.nres[d] == 0) {
                row.gpu[d] += c - row.occ[d];
                row.occ[d] = kNone;
            }
        }
    }
    int64_t g = 0;
    for (int32_t d = 0; d < D; ++d) {
        if (row.occ[d] != kNone) row.gpu[d] += end - row.occ[d];
        g += row.gpu[d];
    }
    for (int32_t w = 0; w < W; ++w) row.comp[w] -= dp.arrival[w];
    *makespan = end - dp.first_arrival;
    *gpu_total = g;
    if (phi) { phi[0] = timely; phi[1] = life; }
}

// One play with the replica batch limit B_q (Eq. 11 over every active unit,
// Section 3.5): a device runs units of one replica (a resident model) at a
// time, up to B = dp.batch of them at once.  Units are admitted in dispatch
// order.  A unit of the device's current replica takes the slot that frees
// earliest, no earlier than its release and the device's latest admission,
// once resident weights + the KV of the units still running + its own KV
// fit (idle least-recently-used models are reclaimed first; if that is not
// enough the unit waits for the next running unit to end).  A unit of
// another model waits for the device to drain and then hits or loads as in
// play<false>; its other slots free when the model is ready.  B = 1 gives
// play<false>'s results.  Deterministic times; retain rows only with B = 1.
__device__ void play_batched(const wf_dev_problem &dp, const PlanRows &pr, Row &row, int64_t *makespan,
                             int64_t *gpu_total)
{
    const int32_t N = dp.N, D = dp.D, M = dp.M, W = dp.W, B = dp.batch;
    for (int32_t d = 0; d < D; ++d) {
        row.occ[d] = kNone; row.gpu[d] = 0; row.used[d] = 0; row.nres[d] = 0;
        row.last_adm[d] = 0; row.cur[d] = -1;
        for (int32_t j = 0; j < B; ++j) { row.slot_end[d * B + j] = 0; row.slot_kv[d * B + j] = 0; }
    }
    for (int32_t k = 0; k < D * M; ++k) row.stamp[k] = 0;
    for (int32_t w = 0; w < W; ++w) row.comp[w] = kNone;
    int64_t end = 0;

    for (int32_t i = 0; i < N; ++i) {
        const int32_t h = pr.order[i];
        const int32_t d = pr.place[h];
        const int32_t fp = dp.fprev[h];
        if (fp >= 0 && bit_at(pr.fuse, h) && pr.place[fp] == d) continue;  // inside its head's unit
        const int32_t m = dp.model[h];
        const int32_t w = dp.session[h];
        const int64_t arr = dp.arrival[w];
        int64_t rel = arr;
        for (int32_t e = dp.pred_off[h]; e < dp.pred_off[h + 1]; ++e)
            rel = max(rel, row.ctail[dp.pred_idx[e]]);
        const int32_t wm = dp.weight[m];
        int32_t tail = h;
        int64_t kv = dp.peak[(int64_t)h * D + d] - wm;
        int64_t run = dp.lat[(int64_t)h * D + d];
        for (int32_t s = dp.fnext[h]; s >= 0 && bit_at(pr.fuse, s) && pr.place[s] == d; s = dp.fnext[s]) {
            kv = max(kv, (int64_t)dp.peak[(int64_t)s * D + d] - wm);
            run += dp.lat[(int64_t)s * D + d];
            tail = s;
        }
        int32_t *st = row.stamp + d * M;
        int64_t *se = row.slot_end + d * B, *sk = row.slot_kv + d * B;
        const int64_t cap = dp.cap[d];
        int64_t adm, start;
        int32_t slot = 0;
        if (m == row.cur[d]) {
            // Join the current replica (Eq. 11 with the running units' KV).
            for (int32_t j = 1; j < B; ++j)
                if (se[j] < se[slot]) slot = j;
            adm = max(max(rel, se[slot]), row.last_adm[d]);
            for (;;) {
                int64_t running = 0;
                for (int32_t j = 0; j < B; ++j) running += se[j] > adm ? sk[j] : 0;
                while (row.used[d] + running + kv > cap) {  // idle models, least recently used first
                    int32_t victim = -1, vs = INT32_MAX;
                    for (int32_t k = 0; k < M; ++k)
                        if (k != m && st[k] != 0 && st[k] < vs) { vs = st[k]; victim = k; }
                    if (victim < 0) break;
                    row.used[d] -= dp.weight[victim];
                    row.nres[d] -= 1;
                    st[victim] = 0;
                }
                if (row.used[d] + running + kv <= cap) break;
                int64_t next = kNone;  // the next running unit to end
                for (int32_t j = 0; j < B; ++j)
                    if (se[j] > adm && (next == kNone || se[j] < next)) next = se[j];
                if (next == kNone) { atomicExch(dp.err, 2); break; }  // unreachable for a valid plan
                adm = next;
            }
            start = adm;
        } else {
            // Another model: the device drains, then the unit hits or loads.
            int64_t drain = 0;
            for (int32_t j = 0; j < B; ++j) drain = max(drain, se[j]);
            const bool hit = st[m] != 0;
            const int64_t need = hit ? kv : wm + kv;
            while (row.used[d] + need > cap) {
                int32_t victim = -1, vs = INT32_MAX;
                for (int32_t k = 0; k < M; ++k)
                    if (k != m && st[k] != 0 && st[k] < vs) { vs = st[k]; victim = k; }
                if (victim < 0) { atomicExch(dp.err, 2); break; }  // unreachable for a valid plan
                row.used[d] -= dp.weight[victim];
                row.nres[d] -= 1;
                st[victim] = 0;
            }
            int64_t ready;
            if (hit) {
                adm = start = max(drain, rel);
                ready = drain;
            } else {
                const int64_t ls = max(drain, bit_at(pr.prefetch, h) ? arr : rel);
                if (row.occ[d] == kNone) row.occ[d] = ls;
                row.used[d] += wm;
                row.nres[d] += 1;
                const int64_t le = ls + dp.load[m * D + d];
                adm = ls;
                start = max(le, rel);
                ready = le;
            }
            for (int32_t j = 0; j < B; ++j) { se[j] = ready; sk[j] = 0; }
            row.cur[d] = m;
        }
        const int64_t c = start + dp.grant + run;
        row.ctail[tail] = c;
        se[slot] = c;
        sk[slot] = kv;
        row.last_adm[d] = adm;
        st[m] = i + 1;
        end = max(end, c);
        row.comp[w] = max(row.comp[w], c);
        if (pr.retain && !bit_at(pr.retain, tail)) {  // B = 1 only
            row.used[d] -= wm;
            row.nres[d] -= 1;
            st[m] = 0;
            row.cur[d] = -1;
            if (row.nres[d] == 0) {
                row.gpu[d] += c - row.occ[d];
                row.occ[d] = kNone;
            }
        }
    }
    int64_t g = 0;
    for (int32_t d = 0; d < D; ++d) {
        if (row.occ[d] != kNone) row.gpu[d] += end - row.occ[d];
        g += row.gpu[d];
    }
    for (int32_t w = 0; w < W; ++w) row.comp[w] -= dp.arrival[w];
    *makespan = end - dp.first_arrival;
    *gpu_total = g;
}

// r-th smallest (0-based) of v[0..n), reordering v (Hoare quickselect).
__device__ int64_t select_rank(int64_t *v, int32_t n, int32_t r)
{
    int32_t lo = 0, hi = n - 1;
    while (lo < hi) {
        const int64_t pivot = v[lo + (hi - lo) / 2];
        int32_t i = lo, j = hi;
        while (i <= j) {
            while (v[i] < pivot) ++i;
            while (v[j] > pivot) --j;
            if (i <= j) { int64_t t = v[i]; v[i] = v[j]; v[j] = t; ++i; --j; }
        }
        if (r <= j) hi = j;
        else if (r >= i) lo = i;
        else return v[r];
    }
    return v[r];
}

__device__ __forceinline__ int32_t p95_rank(int64_t n) { return (int32_t)((95 * n + 99) / 100 - 1); }

__global__ void __launch_bounds__(kEvalThreads)
eval_det_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, uint8_t *scratch, size_t row_bytes,
                int64_t rows)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= rows) return;
    Row row = row_at(dp, scratch + (size_t)t * row_bytes);
    for (int64_t p = t; p < pl.P; p += rows) {
        const PlanRows pr = plan_rows(pl, p);
        const uint32_t st = plan_status(dp, pr, row);
        out.status[p] = st;
        if (st) {
            out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
            if (dp.phi_life) dp.phi_timely[p] = dp.phi_life[p] = WF_INF64;
            continue;
        }
        int64_t mk, g, phi[2];
        if (dp.batch > 0) play_batched(dp, pr, row, &mk, &g);
        else play<false>(dp, pr, row, 0, &mk, &g, dp.phi_life ? phi : nullptr);
        out.makespan_us[p] = mk;
        out.gpu_us[p] = g;
        out.p95_us[p] = select_rank(row.comp, dp.W, p95_rank(dp.W));
        if (dp.phi_life) { dp.phi_timely[p] = phi[0]; dp.phi_life[p] = phi[1]; }
    }
}

// The int64 path for the plans whose times overflow the sweep's u32 slots.
__global__ void __launch_bounds__(kEvalThreads)
eval_list_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, uint8_t *scratch, size_t row_bytes,
                 int64_t rows, const int32_t *list, const int32_t *count)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int32_t n = *count;
    if (t >= rows || t >= n) return;
    Row row = row_at(dp, scratch + (size_t)t * row_bytes);
    for (int64_t k = t; k < n; k += rows) {
        const int64_t p = list[k];
        const PlanRows pr = plan_rows(pl, p);
        const uint32_t st = plan_status(dp, pr, row);
        out.status[p] = st;
        if (st) {
            out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
            if (dp.phi_life) dp.phi_timely[p] = dp.phi_life[p] = WF_INF64;
            continue;
        }
        int64_t mk, g, phi[2];
        if (dp.batch > 0) play_batched(dp, pr, row, &mk, &g);
        else play<false>(dp, pr, row, 0, &mk, &g, dp.phi_life ? phi : nullptr);
        out.makespan_us[p] = mk;
        out.gpu_us[p] = g;
        out.p95_us[p] = select_rank(row.comp, dp.W, p95_rank(dp.W));
        if (dp.phi_life) { dp.phi_timely[p] = phi[0]; dp.phi_life[p] = phi[1]; }
    }
}

// Stochastic latencies: one CTA per plan, one thread per sample; the pooled
// S x W completions of the plan go to a per-CTA pool for the p95 selection.
__global__ void __launch_bounds__(kSampleThreads)
eval_stoch_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, uint8_t *scratch, size_t row_bytes,
                  int64_t *pool_base, int64_t ctas, const int32_t *list, const int32_t *list_len)
{
    __shared__ unsigned long long s_mk, s_gpu;
    __shared__ uint32_t s_status;
    __shared__ uint32_t s_hist[256];
    __shared__ uint64_t s_prefix;
    __shared__ int32_t s_rank;
    const int64_t cta = blockIdx.x;
    const int32_t S = dp.S, W = dp.W;
    Row row = row_at(dp, scratch + (size_t)(cta * blockDim.x + threadIdx.x) * row_bytes);
    int64_t *pool = pool_base + cta * (int64_t)S * W;
    // Every plan of the batch, or only those listed (plans whose times left
    // the 32-bit range of the shared-memory sweep).
    const int64_t total = list ? (int64_t)*list_len : pl.P;
    for (int64_t j = cta; j < total; j += ctas) {
        const int64_t p = list ? (int64_t)list[j] : j;
        const PlanRows pr = plan_rows(pl, p);
        if (threadIdx.x == 0) {
            s_mk = 0; s_gpu = 0;
            s_status = plan_status(dp, pr, row);
        }
        __syncthreads();
        const uint32_t st = s_status;
        if (st) {
            if (threadIdx.x == 0) {
                out.status[p] = st;
                out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
            }
            __syncthreads();
            continue;
        }
        const uint64_t gp = (uint64_t)(pl.plan_base + p);
        for (int32_t s = threadIdx.x; s < S; s += blockDim.x) {
            const uint64_t key = splitmix(splitmix(dp.seed ^ gp) ^ (uint64_t)s);
            int64_t mk, g;
            play<true>(dp, pr, row, key, &mk, &g);
            atomicAdd(&s_mk, (unsigned long long)mk);
            atomicAdd(&s_gpu, (unsigned long long)g);
            for (int32_t w = 0; w < W; ++w) pool[(int64_t)s * W + w] = row.comp[w];
        }
        __syncthreads();
        // Nearest-rank p95 of the pooled non-negative completions: radix
        // select, 8 bits per pass from the most significant byte.
        const int64_t n = (int64_t)S * W;
        if (threadIdx.x == 0) { s_prefix = 0; s_rank = p95_rank(n); }
        __syncthreads();
        for (int shift = 56; shift >= 0; shift -= 8) {
            for (int b = threadIdx.x; b < 256; b += blockDim.x) s_hist[b] = 0;
            __syncthreads();
            const uint64_t hi_mask = shift == 56 ? 0 : (~0ull << (shift + 8));
            for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
                const uint64_t v = (uint64_t)pool[i];
                if ((v & hi_mask) == s_prefix) atomicAdd(&s_hist[(v >> shift) & 255u], 1u);
            }
            __syncthreads();
            if (threadIdx.x == 0) {
                int32_t r = s_rank;
                int b = 0;
                while ((int32_t)s_hist[b] <= r) { r -= s_hist[b]; ++b; }
                s_rank = r;
                s_prefix |= (uint64_t)b << shift;
            }
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            out.status[p] = 0;
            out.makespan_us[p] = (int64_t)(s_mk / (unsigned long long)S);
            out.gpu_us[p] = (int64_t)(s_gpu / (unsigned long long)S);
            out.p95_us[p] = (int64_t)s_prefix;
        }
        __syncthreads();
    }
}

}  // namespace

size_t wf_eval_row_bytes(const wf_dev_problem &dp)
{
    size_t b = ((8 * (size_t)dp.N + 7) & ~(size_t)7) + 8 * 3 * (size_t)dp.D + 8 * (size_t)dp.W +
               2 * ((4 * (size_t)dp.D + 7) & ~(size_t)7) + ((4 * (size_t)dp.D * dp.M + 7) & ~(size_t)7) +
               4 * (size_t)dp.D;
    if (dp.batch > 0) b += 4 + 16 * (size_t)dp.D * dp.batch + 12 * (size_t)dp.D;  // (4: padding after loaded)
    return (b + 127) & ~(size_t)127;
}

static size_t sample_cta_bytes(const wf_dev_problem &dp)
{
    const size_t pool = (8 * (size_t)dp.S * dp.W + 127) & ~(size_t)127;
    return kSampleThreads * wf_eval_row_bytes(dp) + pool;
}

size_t wf_eval_scratch_bytes(const wf_dev_problem &dp, int64_t max_P, int64_t *units)
{
    const size_t budget = (size_t)1 << 30;
    const size_t unit = dp.S == 0 ? wf_eval_row_bytes(dp) : sample_cta_bytes(dp);
    const int64_t floor_units = dp.S == 0 ? 1024 : 16;
    *units = std::min<int64_t>(max_P, std::max<int64_t>((int64_t)(budget / unit), floor_units));
    return unit * (size_t)*units;
}

int wf_launch_eval(wf_ctx *ctx, const wf_plans *plans, const wf_eval_out *out, cudaStream_t st)
{
    const wf_dev_problem &dp = ctx->dp;
    uint8_t *scratch = (uint8_t *)ctx->eval_scratch;
    const int64_t units = std::min<int64_t>(ctx->eval_threads, plans->P);
    if (dp.batch > 1 && plans->retain)
        return wf_set_error(WF_EINVAL, "retain rows are modelled with a replica batch limit of 1 only");
    if (dp.batch > 0 && dp.phi_life)
        return wf_set_error(WF_EINVAL, "the window terms of Eq. 12 are not modelled with a replica batch limit");
    if (dp.S == 0) {
        const int64_t blocks = (units + kEvalThreads - 1) / kEvalThreads;
        // The replica batch limit: its own sweep in shared memory, the int64
        // path for what it hands on (or for everything, when it does not fit).
        const size_t bsm = dp.batch > 0 && !ctx->force_int64 ? wf_batch_smem(dp) : 0;
        if (bsm) {
            int rc = wf_cuda_check(cudaMemsetAsync(ctx->ovf_count, 0, sizeof(int32_t), st), "reset overflow count");
            if (!rc) rc = wf_launch_batch(ctx, plans, out, bsm, ctx->ovf_list, ctx->ovf_count, st);
            if (rc) return rc;
            eval_list_kernel<<<(unsigned)blocks, kEvalThreads, 0, st>>>(dp, *plans, *out, scratch, ctx->eval_row_bytes,
                                                                       units, ctx->ovf_list, ctx->ovf_count);
            return wf_cuda_check(cudaGetLastError(), "int64 pass launch");
        }
        const wf_sweep_cfg cfg = ctx->force_int64 || dp.batch > 0 ? wf_sweep_cfg{} : wf_sweep_config(dp);
        if (dp.reclaim && !cfg.smem64)
            return wf_set_error(WF_EINVAL, "reclamation by next use runs only in the shared-memory sweep");
        if (cfg.smem32 || cfg.smem64) {
            // Under stream capture (a CUDA graph) nothing but launches on the
            // stream may happen: the path choice stays as it is.
            cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
            int rc0 = wf_cuda_check(cudaStreamIsCapturing(st, &cs), "stream capture status");
            if (rc0) return rc0;
            const bool capturing = cs != cudaStreamCaptureStatusNone;
            // Path choice: the u32 sweep's hand-off count of an earlier call,
            // if it has arrived (never waited for).
            if (ctx->wide_pending && !capturing) {
                const cudaError_t q = cudaEventQuery(ctx->ovf_event);
                if (q == cudaSuccess) {
                    ctx->prefer_wide = 2 * (int64_t)*ctx->h_ovf > ctx->wide_P;
                    ctx->wide_pending = false;
                } else if (q == cudaErrorNotReady) {
                    (void)cudaGetLastError();
                } else {
                    return wf_cuda_check(q, "overflow count event");
                }
            }
            const bool wide_first = (ctx->prefer_wide || ctx->start_path >= WF_PATH_WIDE) && cfg.smem64;
            // Two pairs of counts, taken by calls in turn, so that a call
            // issued before an earlier call's read-back has run does not
            // reset the count it reads; a call that comes back to a pair
            // whose read-back is still pending waits for that copy first.
            const int q = capturing ? ctx->ovf_pair : (ctx->ovf_pair ^= 1);
            int32_t *counts = ctx->ovf_count + 2 * q;
            int rc = WF_OK;
            if (!capturing && ctx->wide_pending && ctx->rb_pair == q)
                rc = wf_cuda_check(cudaStreamWaitEvent(st, ctx->ovf_event, 0), "overflow read-back wait");
            if (!rc) rc = wf_cuda_check(cudaMemsetAsync(counts, 0, 2 * sizeof(int32_t), st), "reset overflow counts");
            const int32_t *rest = nullptr, *rest_count = nullptr;
            if (!rc) rc = wf_launch_sweep(ctx, plans, out, cfg, wide_first, counts, ctx->ovf_list, ctx->ovf_list2, st,
                                          &rest, &rest_count);
            if (rc) return rc;
            if (cfg.smem32 && !wide_first && !ctx->wide_pending && !capturing) {
                // The read-back runs on the context's side stream after the
                // sweeps, so the caller's stream never waits for it; the
                // value only picks the path, never a result.
                rc = wf_cuda_check(cudaEventRecord(ctx->sweep_done, st), "sweep event");
                if (!rc) rc = wf_cuda_check(cudaStreamWaitEvent(ctx->side, ctx->sweep_done, 0), "side stream wait");
                if (!rc) rc = wf_cuda_check(cudaMemcpyAsync(ctx->h_ovf, counts, sizeof(int32_t),
                                                            cudaMemcpyDeviceToHost, ctx->side),
                                            "overflow count read-back");
                if (!rc) rc = wf_cuda_check(cudaEventRecord(ctx->ovf_event, ctx->side), "overflow count event");
                if (rc) return rc;
                ctx->wide_pending = true;
                ctx->wide_P = plans->P;
                ctx->rb_pair = q;
            }
            eval_list_kernel<<<(unsigned)blocks, kEvalThreads, 0, st>>>(dp, *plans, *out, scratch,
                                                                       ctx->eval_row_bytes, units,
                                                                       rest, rest_count);
        } else {
            eval_det_kernel<<<(unsigned)blocks, kEvalThreads, 0, st>>>(dp, *plans, *out, scratch,
                                                                        ctx->eval_row_bytes, units);
        }
    } else {
        // Per-thread rows of every CTA first, then one completion pool per CTA.
        int64_t *pool = (int64_t *)(scratch + (size_t)units * kSampleThreads * ctx->eval_row_bytes);
        const size_t smem = ctx->force_int64 ? 0 : wf_stoch_smem(dp);
        if (smem) {
            int rc = wf_cuda_check(cudaMemsetAsync(ctx->ovf_count, 0, sizeof(int32_t), st), "reset overflow count");
            if (!rc) rc = wf_launch_stoch(ctx, plans, out, smem, ctx->ovf_list, ctx->ovf_count, st);
            if (rc) return rc;
            const int64_t lunits = std::min<int64_t>(units, (int64_t)ctx->sms * 4);
            eval_stoch_kernel<<<(unsigned)lunits, kSampleThreads, 0, st>>>(dp, *plans, *out, scratch,
                                                                           ctx->eval_row_bytes, pool, lunits,
                                                                           ctx->ovf_list, ctx->ovf_count);
        } else {
            eval_stoch_kernel<<<(unsigned)units, kSampleThreads, 0, st>>>(dp, *plans, *out, scratch,
                                                                          ctx->eval_row_bytes, pool, units,
                                                                          nullptr, nullptr);
        }
    }
    return wf_cuda_check(cudaGetLastError(), "eval launch");
}

// ---------------------------------------------------------------------------
// Allocation-free entry point: wf_eval_plans_static.
//
// Some callers cannot allocate device memory when they want to score plans:
// a scheduler that runs inside a serving engine which reserved nearly all of
// the GPU's memory up front for model weights and KV cache (an extra
// cudaMalloc there fails, or takes memory the engine's cache counts on), or a
// process whose device memory belongs to another allocator that must not be
// bypassed.  For them this entry point evaluates a deterministic batch with
// no context and no allocation: the caller passes the problem tables, the
// plans and the outputs as device pointers, and every piece of scratch lives
// in the file-scope array below, which each GPU that loads this library holds
// until the process exits.
// ---------------------------------------------------------------------------

namespace {

constexpr size_t kStaticScratchBytes = (size_t)32 << 20;  // 32 MiB
constexpr size_t kStaticHeader = 256;                     // first arrival, error word

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

__host__ __device__ __forceinline__ size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

// Layout: header | succ count [N] | fusible successor [N] | fusible predecessor [N] | rows [P]
struct StaticLayout {
    size_t nsucc, fnext, fprev, rows, total;
};

__host__ __device__ __forceinline__ StaticLayout static_layout(int32_t N, int64_t P, size_t row)
{
    StaticLayout l;
    l.nsucc = kStaticHeader;
    l.fnext = l.nsucc + up256(4 * (size_t)N);
    l.fprev = l.fnext + up256(4 * (size_t)N);
    l.rows = l.fprev + up256(4 * (size_t)N);
    l.total = l.rows + (size_t)P * row;
    return l;
}

// Error word of the static array (header offset 8): 0, or kStaticBadTables
// when the problem tables failed the device check (bits 8.. name the first
// check that failed), or the evaluation's own error codes.
constexpr int kStaticBadTables = 4;

// Everything the derived tables start from: zero successor counts, no links,
// the first arrival at +infinity, a clear error word.
__global__ void static_init_kernel(uint8_t *s, int32_t N, StaticLayout l)
{
    const int32_t n = blockIdx.x * blockDim.x + threadIdx.x;
    if (n == 0) {
        *(int64_t *)s = WF_INF64;
        *(int *)(s + 8) = 0;
    }
    if (n < N) {
        ((int32_t *)(s + l.nsucc))[n] = 0;
        ((int32_t *)(s + l.fnext))[n] = -1;
        ((int32_t *)(s + l.fprev))[n] = -1;
    }
}

// The device check of the caller's tables (one thread per node, model,
// device, session and (model, device) pair), before any of them indexes
// another table.  A failure sets the error word; the kernels after it then
// index nothing.
__global__ void static_check_kernel(uint8_t *s, wf_dev_problem dp)
{
    const int32_t v = blockIdx.x * blockDim.x + threadIdx.x;
    const int32_t N = dp.N, D = dp.D, M = dp.M, W = dp.W;
    int bad = 0;
    if (v < N) {
        const int32_t a = dp.pred_off[v], b = dp.pred_off[v + 1];
        if ((v == 0 && a != 0) || b < a) bad = 1;
        else
            for (int32_t e = a; e < b; ++e) {
                const int32_t u = dp.pred_idx[e];
                if (u < 0 || u >= N || u == v) { bad = 2; break; }
            }
        const uint32_t m = dp.model[v];
        const int32_t w = dp.session[v];
        if (m >= (uint32_t)M) bad = 3;
        else if (w < 0 || w >= W) bad = 4;
        else
            for (int32_t d = 0; d < D; ++d)
                if (dp.lat[(int64_t)v * D + d] < 0 || dp.peak[(int64_t)v * D + d] < dp.weight[m]) { bad = 5; break; }
    }
    if (v < M && dp.weight[v] < 1) bad = 6;
    if (v < D && dp.cap[v] < 1) bad = 7;
    if (v < M * D && dp.load[v] < 0) bad = 8;
    if (v < W && dp.arrival[v] < 0) bad = 9;
    if (bad) atomicCAS((int *)(s + 8), 0, kStaticBadTables | (bad << 8));
}

__global__ void static_count_kernel(uint8_t *s, wf_dev_problem dp, StaticLayout l)
{
    if (*(volatile int *)(s + 8)) return;  // the tables failed the check
    const int32_t v = blockIdx.x * blockDim.x + threadIdx.x;
    if (v < dp.W) atomicMin((long long *)s, (long long)dp.arrival[v]);
    if (v >= dp.N) return;
    int32_t *nsucc = (int32_t *)(s + l.nsucc);
    for (int32_t e = dp.pred_off[v]; e < dp.pred_off[v + 1]; ++e) atomicAdd(&nsucc[dp.pred_idx[e]], 1);
}

// Eq. 3: (u, v) fusible iff succ(u) = {v}, pred(v) = {u}, same model.
__global__ void static_link_kernel(uint8_t *s, wf_dev_problem dp, StaticLayout l)
{
    if (*(volatile int *)(s + 8)) return;  // the tables failed the check
    const int32_t v = blockIdx.x * blockDim.x + threadIdx.x;
    if (v >= dp.N || dp.pred_off[v + 1] - dp.pred_off[v] != 1) return;
    const int32_t u = dp.pred_idx[dp.pred_off[v]];
    if (((const int32_t *)(s + l.nsucc))[u] == 1 && dp.model[u] == dp.model[v]) {
        ((int32_t *)(s + l.fnext))[u] = v;
        ((int32_t *)(s + l.fprev))[v] = u;
    }
}

// The deterministic evaluation with one scratch row per plan and the first
// arrival taken from the static header.
__global__ void __launch_bounds__(kEvalThreads)
eval_static_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, uint8_t *s, StaticLayout l,
                   size_t row_bytes)
{
    const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= pl.P) return;
    if ((*(volatile int *)(s + 8) & 0xFF) == kStaticBadTables) {  // nothing is evaluated
        out.status[p] = WF_ST_TABLES;
        out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
        return;
    }
    wf_dev_problem d = dp;
    d.first_arrival = *(const int64_t *)s;
    Row row = row_at(d, s + l.rows + (size_t)p * row_bytes);
    const PlanRows pr = plan_rows(pl, p);
    const uint32_t st = plan_status(d, pr, row);
    out.status[p] = st;
    if (st) {
        out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
        return;
    }
    int64_t mk, g;
    play<false>(d, pr, row, 0, &mk, &g);
    out.makespan_us[p] = mk;
    out.gpu_us[p] = g;
    out.p95_us[p] = select_rank(row.comp, d.W, p95_rank(d.W));
}

// Device address of the static array per device, from the last lookup
// outside stream capture.
uint8_t *g_static_addr[64];
bool g_static_ready[64];
std::mutex g_static_mu;

}  // namespace

extern "C" int wf_eval_plans_static(const wf_problem *pb, const wf_plans *pl, const wf_eval_out *out,
                                    void *stream)
{
    if (!pb || !pl || !out) return wf_set_error(WF_EINVAL, "NULL argument");
    const int32_t N = pb->N, D = pb->D, M = pb->M, W = pb->W;
    if (N < 1 || N > 65535 || D < 1 || D > 32 || M < 1 || M > 16 || W < 1)
        return wf_set_error(WF_EINVAL, "sizes outside N 1..65535, D 1..32, M 1..16, W >= 1");
    if (pb->S != 0) return wf_set_error(WF_EINVAL, "wf_eval_plans_static evaluates deterministic problems (S = 0) only");
    if (pb->margin_mib != 0)
        return wf_set_error(WF_EINVAL, "wf_eval_plans_static takes no admission margin (fold it into peak_mib)");
    if (!pb->pred_off || !pb->model || !pb->session || !pb->arrival_us || !pb->lat_us || !pb->peak_mib ||
        !pb->weight_mib || !pb->load_us || !pb->cap_mib || pb->grant_us < 0)
        return wf_set_error(WF_EINVAL, "a problem table pointer is NULL or grant_us < 0");
    if (pl->P < 1 || !pl->place || !pl->order || !pl->fuse || !pl->prefetch || pl->plan_base < 0)
        return wf_set_error(WF_EINVAL, "empty batch or NULL plan array");
    if (!out->makespan_us || !out->p95_us || !out->gpu_us || !out->status)
        return wf_set_error(WF_EINVAL, "NULL output array");
    const int64_t words = ((int64_t)N + 31) / 32;
    if (pl->place_stride < N || pl->place_stride % 16 || pl->order_stride < 2 * (int64_t)N ||
        pl->order_stride % 16 || pl->bits_stride < 4 * words || pl->bits_stride % 16)
        return wf_set_error(WF_EINVAL, "plan strides must be multiples of 16 covering N");
    const uintptr_t mis = (uintptr_t)pl->place | (uintptr_t)pl->order | (uintptr_t)pl->fuse |
                          (uintptr_t)pl->prefetch | (uintptr_t)pl->retain;
    if (mis & 15u) return wf_set_error(WF_EINVAL, "plan arrays must be 16-byte aligned");

    wf_dev_problem dp = {};
    dp.N = N; dp.D = D; dp.M = M; dp.W = W;
    dp.grant = pb->grant_us;
    dp.pred_off = pb->pred_off;
    dp.pred_idx = pb->pred_idx;
    dp.model = pb->model;
    dp.session = pb->session;
    dp.arrival = pb->arrival_us;
    dp.lat = pb->lat_us;
    dp.peak = pb->peak_mib;
    dp.weight = pb->weight_mib;
    dp.load = pb->load_us;
    dp.cap = pb->cap_mib;
    const size_t row = wf_eval_row_bytes(dp);
    const StaticLayout l = static_layout(N, pl->P, row);
    if (l.total > kStaticScratchBytes) {
        const int64_t fit = (int64_t)((kStaticScratchBytes - l.rows) / row);
        return wf_set_error(WF_EINVAL,
                            "batch needs %zu bytes of scratch but the static array holds %zu; at most "
                            "%lld plans of this window per call", l.total, kStaticScratchBytes,
                            (long long)fit);
    }

    int dev = 0;
    int rc = wf_cuda_check(cudaGetDevice(&dev), "cudaGetDevice");
    if (rc) return rc;
    if (dev < 0 || dev >= 64) return wf_set_error(WF_EINVAL, "device ordinal %d >= 64", dev);
    cudaStream_t st = (cudaStream_t)stream;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    rc = wf_cuda_check(cudaStreamIsCapturing(st, &cs), "stream capture status");
    if (rc) return rc;
    uint8_t *s = nullptr;
    {
        // Outside capture the address is looked up with the current device
        // (valid in the current context, also after a device reset); under
        // capture the last such lookup on this device is reused.
        std::lock_guard<std::mutex> lock(g_static_mu);
        if (cs == cudaStreamCaptureStatusNone) {
            void *p = nullptr;
            rc = wf_cuda_check(cudaGetSymbolAddress(&p, g_static_scratch), "cudaGetSymbolAddress");
            if (rc) return rc;
            g_static_addr[dev] = (uint8_t *)p;
            g_static_ready[dev] = true;
        } else if (!g_static_ready[dev]) {
            return wf_set_error(WF_EINVAL, "the first wf_eval_plans_static call on a device must not be captured");
        }
        s = g_static_addr[dev];
    }
    dp.fnext = (const int32_t *)(s + l.fnext);
    dp.fprev = (const int32_t *)(s + l.fprev);
    dp.err = (int *)(s + 8);

    const int32_t span = std::max(N, W);
    const unsigned grid = (unsigned)((span + 255) / 256);
    const int32_t cspan = std::max(span, M * D);
    static_init_kernel<<<(unsigned)((N + 255) / 256), 256, 0, st>>>(s, N, l);
    static_check_kernel<<<(unsigned)((cspan + 255) / 256), 256, 0, st>>>(s, dp);
    static_count_kernel<<<grid, 256, 0, st>>>(s, dp, l);
    static_link_kernel<<<(unsigned)((N + 255) / 256), 256, 0, st>>>(s, dp, l);
    eval_static_kernel<<<(unsigned)((pl->P + kEvalThreads - 1) / kEvalThreads), kEvalThreads, 0, st>>>(
        dp, *pl, *out, s, l, row);
    return wf_cuda_check(cudaGetLastError(), "static evaluation launch");
}

extern "C" int wf_static_status(void *stream)
{
    int rc = wf_cuda_check(cudaStreamSynchronize((cudaStream_t)stream), "cudaStreamSynchronize");
    if (rc) return rc;
    int err = 0;
    rc = wf_cuda_check(cudaMemcpyFromSymbol(&err, g_static_scratch, sizeof(int), 8), "read the static error word");
    if (rc) return rc;
    if (!err) return WF_OK;
    const int zero = 0;
    rc = wf_cuda_check(cudaMemcpyToSymbol(g_static_scratch, &zero, sizeof(int), 8), "clear the static error word");
    if (rc) return rc;
    if ((err & 0xFF) == kStaticBadTables) {
        static const char *what[] = {"", "pred_off does not start at 0 or decreases",
                                     "a pred_idx entry is out of range or a self-loop", "a model id is >= M",
                                     "a session id is out of range", "a run time is negative or a peak below its weight",
                                     "a weight is below 1", "a capacity is below 1", "a load time is negative",
                                     "an arrival is negative"};
        const int k = err >> 8;
        return wf_set_error(WF_EINVAL, "the problem tables failed the device check: %s",
                            k >= 1 && k <= 9 ? what[k] : "unknown");
    }
    return wf_set_error(WF_ECUDA, "device error word %d in the static evaluation", err);
}
