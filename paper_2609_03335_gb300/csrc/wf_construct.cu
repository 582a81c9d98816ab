// Plan construction: the paper's per-tick scheduler (Algorithm 1) read as a
// list scheduler over the whole window, one plan per thread.
//
//   RankReady            a node is ready once every graph predecessor is
//                        dispatched; the ready node with the smallest
//                        (release + jitter, id) goes next (aging)
//   BestFeasibleBinding  the device, among those whose capacity holds the
//                        node (Eq. 8), with the smallest predicted finish
//                        (resident model: no load; missing model: loaded on
//                        the device, prefetched if the device would idle
//                        before the release) plus jitter; ties: lower device
//   units                the node's fusible chain (Eq. 3) follows it on that
//                        device while each next member fits (fuse bit 1)
//   PlanPrefetch         the head's prefetch bit when its model is missing
//                        and the device is free before the release
//
// Each unit is played forward with the evaluation rules (admission and LRU
// reclamation, Eq. 11; loads, Eq. 5; starts and finishes, Eq. 2, 7, 10), so
// the constructor's timeline is the one wf_eval_plans reports for its plan.
// State per thread lives in global scratch: finish times (a ready node's
// release until it runs), a binary heap of (rank << 16 | node) keys, the
// pending predecessor counts, and per device the free time, resident weights
// and last-use stamps.
#include <algorithm>

#include "wf_internal.cuh"

namespace {

constexpr int kThreads = 32;     // one warp per CTA, so the plans spread over every SM
constexpr int kPlansPerSm = 128;  // plans built at once per SM (the scratch is sized for them)

__device__ __forceinline__ uint64_t mix64(uint64_t x)  // SplitMix64 output function
{
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
}

struct Scratch {
    int64_t *c;        // [N] finish (release while ready)
    uint64_t *heap;    // [N]
    int32_t *pending;  // [N]
    int64_t *t_free;   // [D]
    int64_t *used;     // [D]
    int64_t *stamp;    // [D][M] last-use sequence number, 0 = not resident
};

__host__ __device__ inline size_t scratch_bytes(int32_t N, int32_t D, int32_t M)
{
    const size_t b = 8 * (size_t)N + 8 * (size_t)N + 4 * (size_t)N + 16 * (size_t)D + 8 * (size_t)D * M;
    return (b + 255) & ~(size_t)255;
}

__device__ __forceinline__ void heap_push(uint64_t *h, int32_t &n, uint64_t key)
{
    int32_t i = n++;
    while (i > 0) {
        const int32_t parent = (i - 1) >> 1;
        const uint64_t pk = h[parent];
        if (pk <= key) break;
        h[i] = pk;
        i = parent;
    }
    h[i] = key;
}

__device__ __forceinline__ uint64_t heap_pop(uint64_t *h, int32_t &n)
{
    const uint64_t top = h[0];
    const uint64_t last = h[--n];
    int32_t i = 0;
    for (;;) {
        int32_t child = 2 * i + 1;
        if (child >= n) break;
        uint64_t ck = h[child];
        if (child + 1 < n) {
            const uint64_t rk = h[child + 1];
            if (rk < ck) { ck = rk; ++child; }
        }
        if (last <= ck) break;
        h[i] = ck;
        i = child;
    }
    if (n > 0) h[i] = last;
    return top;
}

__global__ void __launch_bounds__(kThreads)
construct_kernel(wf_dev_problem dp, wf_plans out, uint64_t seed, int64_t jitter, uint8_t *scratch, int64_t threads)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= threads) return;
    const int32_t N = dp.N, D = dp.D, M = dp.M;
    const int32_t words = (N + 31) / 32;
    uint8_t *base = scratch + (size_t)t * scratch_bytes(N, D, M);
    Scratch s;
    s.c = (int64_t *)base;
    s.heap = (uint64_t *)(s.c + N);
    s.t_free = (int64_t *)(s.heap + N);
    s.used = s.t_free + D;
    s.stamp = s.used + D;
    s.pending = (int32_t *)(s.stamp + (size_t)D * M);
    const uint64_t jmod = (uint64_t)jitter + 1;

    for (int64_t p = t; p < out.P; p += threads) {
        const uint64_t g = (uint64_t)(out.plan_base + p);
        const uint64_t hp = mix64(seed ^ g);
        uint8_t *place = (uint8_t *)out.place + p * out.place_stride;
        uint16_t *order = (uint16_t *)((uint8_t *)out.order + p * out.order_stride);
        uint32_t *fuse = (uint32_t *)((uint8_t *)out.fuse + p * out.bits_stride);
        uint32_t *prefetch = (uint32_t *)((uint8_t *)out.prefetch + p * out.bits_stride);
        for (int32_t k = 0; k < words; ++k) { fuse[k] = 0; prefetch[k] = 0; }
        if (out.retain) {
            uint32_t *retain = (uint32_t *)((uint8_t *)out.retain + p * out.bits_stride);
            for (int32_t k = 0; k < words; ++k)
                retain[k] = (k + 1 < words || (N & 31) == 0) ? 0xFFFFFFFFu : ((1u << (N & 31)) - 1u);
        }
        for (int32_t d = 0; d < D; ++d) { s.t_free[d] = 0; s.used[d] = 0; }
        for (int32_t k = 0; k < D * M; ++k) s.stamp[k] = 0;
        int32_t nheap = 0;
        for (int32_t v = 0; v < N; ++v) {
            const int32_t np = __ldg(dp.pred_off + v + 1) - __ldg(dp.pred_off + v);
            s.pending[v] = np;
            if (np == 0) {
                const int64_t rel = __ldg(dp.arrival + __ldg(dp.session + v));
                s.c[v] = rel;
                const uint64_t j = jitter > 0 ? mix64(hp ^ (uint64_t)v) % jmod : 0;
                heap_push(s.heap, nheap, (((uint64_t)rel + j) << 16) | (uint64_t)v);
            }
        }
        int32_t pos = 0;
        int64_t seq = 0;
        while (nheap > 0) {
            const int32_t u = (int32_t)(heap_pop(s.heap, nheap) & 0xFFFFu);
            const int64_t rel = s.c[u];
            const int32_t m = __ldg(dp.model + u);
            const int64_t arr = __ldg(dp.arrival + __ldg(dp.session + u));
            const uint64_t hu = mix64(hp ^ (uint64_t)u);
            const uint32_t fit_u = __ldg(dp.fitmask + u);

            // BestFeasibleBinding.
            int32_t d = -1;
            int64_t best = 0;
            for (int32_t dd = 0; dd < D; ++dd) {
                if (!((fit_u >> dd) & 1u)) continue;
                const int64_t tf = s.t_free[dd];
                int64_t start;
                if (s.stamp[dd * M + m] != 0) {
                    start = max(tf, rel);
                } else {
                    const int64_t ls = tf < rel ? max(tf, arr) : max(tf, rel);
                    start = max(ls + (int64_t)__ldg(dp.load + m * D + dd), rel);
                }
                const int64_t fin = start + dp.grant + (int64_t)__ldg(&dp.lk[u * D + dd].x);
                const int64_t score = fin + (jitter > 0 ? (int64_t)(mix64(hu ^ (uint64_t)(dd + 1)) % jmod) : 0);
                if (d < 0 || score < best) { d = dd; best = score; }
            }
            if (d < 0) { atomicExch(dp.err, 4); return; }  // unreachable: every node fits somewhere

            // The unit: u and its fusible chain while the members fit on d.
            const bool hit = s.stamp[d * M + m] != 0;
            const int64_t tf = s.t_free[d];
            const bool pf = !hit && tf < rel;
            int64_t kv = __ldg(&dp.lk[u * D + d].y);
            place[u] = (uint8_t)d;
            order[pos++] = (uint16_t)u;
            int32_t tail = u;
            for (int32_t x = __ldg(dp.fnext + u); x >= 0 && ((__ldg(dp.fitmask + x) >> d) & 1u);
                 x = __ldg(dp.fnext + x)) {
                place[x] = (uint8_t)d;
                order[pos++] = (uint16_t)x;
                fuse[x >> 5] |= 1u << (x & 31);
                kv = max(kv, (int64_t)__ldg(&dp.lk[x * D + d].y));
                tail = x;
            }
            if (pf) prefetch[u >> 5] |= 1u << (u & 31);

            // Play it forward: admission with LRU reclamation (Eq. 11), load, run.
            int64_t *st = s.stamp + d * M;
            const int64_t wm = __ldg(dp.weight + m);
            const int64_t need = hit ? kv : wm + kv;
            const int64_t capd = __ldg(dp.cap + d);
            while (s.used[d] + need > capd) {
                int32_t victim = -1;
                for (int32_t k = 0; k < M; ++k)
                    if (k != m && st[k] != 0 && (victim < 0 || st[k] < st[victim])) victim = k;
                if (victim < 0) { atomicExch(dp.err, 4); return; }  // unreachable: the unit fits on d
                s.used[d] -= __ldg(dp.weight + victim);
                st[victim] = 0;
            }
            int64_t start;
            if (hit) {
                start = max(tf, rel);
            } else {
                const int64_t ls = pf ? max(tf, arr) : max(tf, rel);
                start = max(ls + (int64_t)__ldg(dp.load + m * D + d), rel);
                s.used[d] += wm;
            }
            int64_t fin = start + dp.grant;
            for (int32_t x = u;; x = __ldg(dp.fnext + x)) {
                fin += __ldg(&dp.lk[x * D + d].x);
                s.c[x] = fin;
                if (x == tail) break;
            }
            s.t_free[d] = fin;
            st[m] = ++seq;

            // Successors of the unit's last member.
            for (int32_t e = __ldg(dp.succ_off + tail); e < __ldg(dp.succ_off + tail + 1); ++e) {
                const int32_t y = __ldg(dp.succ_idx + e);
                if (--s.pending[y] > 0) continue;
                int64_t r = __ldg(dp.arrival + __ldg(dp.session + y));
                for (int32_t f = __ldg(dp.pred_off + y); f < __ldg(dp.pred_off + y + 1); ++f)
                    r = max(r, s.c[__ldg(dp.pred_idx + f)]);
                s.c[y] = r;
                const uint64_t j = jitter > 0 ? mix64(hp ^ (uint64_t)y) % jmod : 0;
                heap_push(s.heap, nheap, (((uint64_t)r + j) << 16) | (uint64_t)y);
            }
        }
    }
}

}  // namespace

extern "C" int wf_construct_plans(wf_ctx *c, const wf_plans *out, uint64_t seed, int64_t jitter_us, void *stream)
{
    if (!c || !out) return wf_set_error(WF_EINVAL, "NULL argument");
    int rc = wf_check_plans(c, out, "plans");
    if (rc) return rc;
    if (jitter_us < 0) return wf_set_error(WF_EINVAL, "jitter_us < 0");
    // Ranks (release + jitter) are packed above a 16-bit node id.
    if (c->dp.horizon + jitter_us >= ((int64_t)1 << 47))
        return wf_set_error(WF_EINVAL, "window horizon %lld us + jitter exceeds 2^47 us", (long long)c->dp.horizon);
    rc = wf_select_device(c);
    if (rc) return rc;
    const wf_dev_problem &dp = c->dp;
    if (!c->construct_scratch) {
        // First call: per-thread state for up to kPlansPerSm plans per SM at once.
        c->construct_threads = std::min<int64_t>(c->max_P, (int64_t)c->sms * kPlansPerSm);
        rc = wf_cuda_check(cudaMalloc(&c->construct_scratch, scratch_bytes(dp.N, dp.D, dp.M) * c->construct_threads),
                           "cudaMalloc(constructor scratch)");
        if (rc) { c->construct_scratch = nullptr; return rc; }
    }
    const int64_t threads = std::min<int64_t>(out->P, c->construct_threads);
    const unsigned blocks = (unsigned)((threads + kThreads - 1) / kThreads);
    construct_kernel<<<blocks, kThreads, 0, (cudaStream_t)stream>>>(dp, *out, seed, jitter_us,
                                                                    (uint8_t *)c->construct_scratch, threads);
    return wf_cuda_check(cudaGetLastError(), "construct launch");
}
