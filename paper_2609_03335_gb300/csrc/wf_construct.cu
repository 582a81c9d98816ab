// Plan construction: the paper's per-tick scheduler (Algorithm 1) read as a
// list scheduler over the whole window, one plan per warp.
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
// State per plan lives in global scratch: finish times (a ready node's
// release until it runs), the unordered ready keys (rank << 16 | node), the
// pending predecessor counts, and per device the free time, resident weights
// and last-use stamps.
#include <algorithm>

#include "wf_internal.cuh"

namespace {

constexpr int kWarps = 4;          // warps per CTA, a plan per warp
constexpr int kCtasPerSm = 10;     // resident CTAs per SM (48 registers per thread)
constexpr int kSlotsPerSm = kWarps * kCtasPerSm;  // plans built at once per SM (the scratch is sized for them)

__device__ __forceinline__ uint64_t mix64(uint64_t x)  // SplitMix64 output function
{
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
}

// x mod d for d >= 2, exact for every 64-bit x, from the 128-bit reciprocal
// M = floor((2^128 - 1) / d) + 1 (Lemire, Kaser and Kurz, "Faster remainder
// by direct computation", 2019): the remainder is the top 64 bits of
// (M x mod 2^128) d.  A handful of multiplies instead of a 64-bit division.
struct Mod64 {
    uint64_t mh, ml, d;
};

__device__ __forceinline__ uint64_t mod64(uint64_t x, const Mod64 &m)
{
    const uint64_t l0 = m.ml * x;
    const uint64_t l1 = __umul64hi(m.ml, x) + m.mh * x;
    const uint64_t a1 = __umul64hi(l0, m.d);
    const uint64_t s = a1 + l1 * m.d;
    return __umul64hi(l1, m.d) + (s < a1 ? 1u : 0u);
}

// Per-plan state in global scratch.  A node's release is accumulated as its
// predecessors' units finish (every predecessor of a node released this way
// is the last member of its unit), so no finish time is read back.
struct Scratch {
    uint64_t *key;     // [N] ready keys (rank << 16 | node), unordered
    int64_t *rel;      // [N] the release of the ready node beside it
    int64_t *relmax;   // [N] session arrival, raised to each finished predecessor's finish
    int32_t *pending;  // [N] predecessors not yet finished
};

__host__ __device__ inline size_t scratch_bytes(int32_t N)
{
    return ((8 + 8 + 8 + 4) * (size_t)N + 255) & ~(size_t)255;
}

// Per-warp device state in shared memory: free time and resident weight per
// device, last-use stamp per (device, model) (0 = not resident; stamps count
// units, below 2^16).
__host__ __device__ inline size_t warp_smem(int32_t D, int32_t M)
{
    return ((16 * (size_t)D + 2 * (size_t)D * M) + 15) & ~(size_t)15;
}

// Warp-wide minimum of a 64-bit key (two 32-bit warp reductions: high
// halves, then low halves among the lanes holding the smallest high half);
// returns the lowest lane holding it, and every lane gets the minimum.
__device__ __forceinline__ int warp_argmin64(uint64_t &key)
{
    const uint32_t hi = __reduce_min_sync(0xFFFFFFFFu, (uint32_t)(key >> 32));
    const uint32_t lo = __reduce_min_sync(0xFFFFFFFFu, (uint32_t)(key >> 32) == hi ? (uint32_t)key : 0xFFFFFFFFu);
    const uint64_t k = ((uint64_t)hi << 32) | lo;
    const int src = __ffs((int)__ballot_sync(0xFFFFFFFFu, key == k)) - 1;
    key = k;
    return src;
}

// Appends (key, rel) of the lanes with take set to the ready arrays at n.
__device__ __forceinline__ void append(const Scratch &s, int32_t &n, bool take, uint64_t key, int64_t rel,
                                       int lane)
{
    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, take);
    if (take) {
        const int32_t i = n + __popc(bal & ((1u << lane) - 1u));
        s.key[i] = key;
        s.rel[i] = rel;
    }
    n += __popc(bal);
}

// A warp per plan.  The ready set is an unordered array; each step takes its
// smallest key (a warp minimum over the array, the node a heap would give,
// keys being unique), scores every device in its own lane, picks
// reclamation victims as a warp minimum over the device's stamps, and
// releases the unit's successors in parallel lanes.  Lane 0 writes the
// plan's rows and the device state; __syncwarp orders those writes before
// the other lanes read them.
__global__ void __launch_bounds__(32 * kWarps, kCtasPerSm)
construct_kernel(wf_dev_problem dp, wf_plans out, uint64_t seed, int64_t jitter, Mod64 jm, uint8_t *scratch,
                 int64_t slots)
{
    extern __shared__ __align__(16) uint8_t csm[];
    const int lane = threadIdx.x & 31;
    const int64_t w = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (w >= slots) return;
    const int32_t N = dp.N, D = dp.D, M = dp.M;
    const int32_t words = (N + 31) / 32;
    uint8_t *base = scratch + (size_t)w * scratch_bytes(N);
    Scratch s;
    s.key = (uint64_t *)base;
    s.rel = (int64_t *)(s.key + N);
    s.relmax = s.rel + N;
    s.pending = (int32_t *)(s.relmax + N);
    uint8_t *wsm = csm + (size_t)(threadIdx.x >> 5) * warp_smem(D, M);
    int64_t *t_free = (int64_t *)wsm;
    int64_t *used_d = t_free + D;
    uint16_t *stamp = (uint16_t *)(used_d + D);
    // Jitter draws are taken mod (jitter + 1) >= 2 when jitter > 0.
    for (int64_t p = w; p < out.P; p += slots) {
        const uint64_t g = (uint64_t)(out.plan_base + p);
        const uint64_t hp = mix64(seed ^ g);
        uint8_t *place = (uint8_t *)out.place + p * out.place_stride;
        uint16_t *order = (uint16_t *)((uint8_t *)out.order + p * out.order_stride);
        uint32_t *fuse = (uint32_t *)((uint8_t *)out.fuse + p * out.bits_stride);
        uint32_t *prefetch = (uint32_t *)((uint8_t *)out.prefetch + p * out.bits_stride);
        for (int32_t k = lane; k < words; k += 32) { fuse[k] = 0; prefetch[k] = 0; }
        if (out.retain) {
            uint32_t *retain = (uint32_t *)((uint8_t *)out.retain + p * out.bits_stride);
            for (int32_t k = lane; k < words; k += 32)
                retain[k] = (k + 1 < words || (N & 31) == 0) ? 0xFFFFFFFFu : ((1u << (N & 31)) - 1u);
        }
        for (int32_t d = lane; d < D; d += 32) { t_free[d] = 0; used_d[d] = 0; }
        for (int32_t k = lane; k < D * M; k += 32) stamp[k] = 0;
        int32_t nready = 0;
        for (int32_t v0 = 0; v0 < N; v0 += 32) {
            const int32_t v = v0 + lane;
            bool take = false;
            uint64_t key = 0;
            int64_t arr = 0;
            if (v < N) {
                const int32_t np = __ldg(dp.pred_off + v + 1) - __ldg(dp.pred_off + v);
                arr = __ldg(dp.arrival + __ldg(dp.session + v));
                s.pending[v] = np;
                s.relmax[v] = arr;
                if (np == 0) {
                    const uint64_t j = jitter > 0 ? mod64(mix64(hp ^ (uint64_t)v), jm) : 0;
                    key = (((uint64_t)arr + j) << 16) | (uint64_t)v;
                    take = true;
                }
            }
            append(s, nready, take, key, arr, lane);
        }
        __syncwarp();
        int32_t pos = 0;
        uint32_t seq = 0;
        while (nready > 0) {
            // RankReady: the smallest key, with its release.
            uint64_t best = ~0ull;
            int32_t at = 0;
            for (int32_t i = lane; i < nready; i += 32) {
                const uint64_t k = s.key[i];
                if (k < best) { best = k; at = i; }
            }
            const int src = warp_argmin64(best);  // keys are unique
            at = __shfl_sync(0xFFFFFFFFu, at, src);
            const int64_t rel = s.rel[at];
            const int32_t u = (int32_t)(best & 0xFFFFu);
            const uint64_t last_k = s.key[nready - 1];
            const int64_t last_r = s.rel[nready - 1];
            __syncwarp();
            if (lane == 0) { s.key[at] = last_k; s.rel[at] = last_r; }
            --nready;
            const int32_t m = __ldg(dp.model + u);
            const int64_t arr = __ldg(dp.arrival + __ldg(dp.session + u));
            const uint32_t fit_u = __ldg(dp.fitmask + u);

            // BestFeasibleBinding: device lane by lane, then the smallest
            // (score, device).
            uint64_t score = ~0ull;
            int64_t tf_l = 0;
            if (lane < D && ((fit_u >> lane) & 1u)) {
                tf_l = t_free[lane];
                int64_t start;
                if (stamp[lane * M + m] != 0) {
                    start = max(tf_l, rel);
                } else {
                    const int64_t ls = tf_l < rel ? max(tf_l, arr) : max(tf_l, rel);
                    start = max(ls + (int64_t)__ldg(dp.load + m * D + lane), rel);
                }
                const int64_t fin = start + dp.grant + (int64_t)__ldg(&dp.lk[u * D + lane].x);
                const uint64_t hu = mix64(hp ^ (uint64_t)u);
                score = (uint64_t)(fin + (jitter > 0 ? (int64_t)mod64(mix64(hu ^ (uint64_t)(lane + 1)), jm) : 0));
            }
            const int32_t d = warp_argmin64(score);  // ties: the lower device
            if (score == ~0ull) {  // unreachable: every node fits somewhere
                if (lane == 0) atomicExch(dp.err, 4);
                return;
            }
            const int64_t tf = __shfl_sync(0xFFFFFFFFu, tf_l, d);
            uint16_t *st = stamp + d * M;
            const bool hit = st[m] != 0;

            // The unit: u and its fusible chain while the members fit on d.
            const bool pf = !hit && tf < rel;
            int64_t kv = __ldg(&dp.lk[u * D + d].y);
            if (lane == 0) { place[u] = (uint8_t)d; order[pos] = (uint16_t)u; }
            ++pos;
            int32_t tail = u;
            for (int32_t x = __ldg(dp.fnext + u); x >= 0 && ((__ldg(dp.fitmask + x) >> d) & 1u);
                 x = __ldg(dp.fnext + x)) {
                if (lane == 0) {
                    place[x] = (uint8_t)d;
                    order[pos] = (uint16_t)x;
                    fuse[x >> 5] |= 1u << (x & 31);
                }
                ++pos;
                kv = max(kv, (int64_t)__ldg(&dp.lk[x * D + d].y));
                tail = x;
            }
            if (pf && lane == 0) prefetch[u >> 5] |= 1u << (u & 31);

            // Play it forward: admission with LRU reclamation (Eq. 11), load, run.
            const int64_t wm = __ldg(dp.weight + m);
            const int64_t need = hit ? kv : wm + kv;
            const int64_t capd = __ldg(dp.cap + d);
            int64_t used = used_d[d];
            while (used + need > capd) {
                const uint32_t sk = (lane < M && lane != m && st[lane] != 0) ? st[lane] : 0xFFFFFFFFu;
                const uint32_t smin = __reduce_min_sync(0xFFFFFFFFu, sk);
                if (smin == 0xFFFFFFFFu) {  // unreachable: the unit fits on d
                    if (lane == 0) atomicExch(dp.err, 4);
                    return;
                }
                const int32_t victim = __ffs((int)__ballot_sync(0xFFFFFFFFu, sk == smin)) - 1;
                used -= __ldg(dp.weight + victim);
                __syncwarp();
                if (lane == 0) st[victim] = 0;
                __syncwarp();
            }
            int64_t start;
            if (hit) {
                start = max(tf, rel);
            } else {
                const int64_t ls = pf ? max(tf, arr) : max(tf, rel);
                start = max(ls + (int64_t)__ldg(dp.load + m * D + d), rel);
                used += wm;
            }
            int64_t fin = start + dp.grant;
            for (int32_t x = u;; x = __ldg(dp.fnext + x)) {
                fin += __ldg(&dp.lk[x * D + d].x);
                if (x == tail) break;
            }
            ++seq;
            __syncwarp();
            if (lane == 0) {
                used_d[d] = used;
                t_free[d] = fin;
                st[m] = (uint16_t)seq;
            }
            __syncwarp();

            // Successors of the unit's last member, one per lane: each takes
            // this finish into its release; the last predecessor makes it ready.
            const int32_t e0 = __ldg(dp.succ_off + tail), e1 = __ldg(dp.succ_off + tail + 1);
            for (int32_t eb = e0; eb < e1; eb += 32) {
                const int32_t e = eb + lane;
                bool take = false;
                uint64_t key = 0;
                int64_t r = 0;
                if (e < e1) {
                    const int32_t y = __ldg(dp.succ_idx + e);
                    const int32_t left = s.pending[y] - 1;
                    r = max(s.relmax[y], fin);
                    s.pending[y] = left;
                    s.relmax[y] = r;
                    if (left == 0) {
                        const uint64_t j = jitter > 0 ? mod64(mix64(hp ^ (uint64_t)y), jm) : 0;
                        key = (((uint64_t)r + j) << 16) | (uint64_t)y;
                        take = true;
                    }
                }
                append(s, nready, take, key, r, lane);
            }
            __syncwarp();
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
        // First call: per-plan state for up to kSlotsPerSm plans per SM at once.
        c->construct_threads = std::min<int64_t>(c->max_P, (int64_t)c->sms * kSlotsPerSm);
        rc = wf_cuda_check(cudaMalloc(&c->construct_scratch, scratch_bytes(dp.N) * c->construct_threads),
                           "cudaMalloc(constructor scratch)");
        if (rc) { c->construct_scratch = nullptr; return rc; }
    }
    const int64_t slots = std::min<int64_t>(out->P, c->construct_threads);
    const unsigned blocks = (unsigned)((slots + kWarps - 1) / kWarps);
    const size_t smem = kWarps * warp_smem(dp.D, dp.M);
    Mod64 jm = {0, 0, (uint64_t)jitter_us + 1};
    if (jitter_us > 0) {
        const unsigned __int128 r = ~(unsigned __int128)0 / jm.d + 1;
        jm.mh = (uint64_t)(r >> 64);
        jm.ml = (uint64_t)r;
    }
    construct_kernel<<<blocks, 32 * kWarps, smem, (cudaStream_t)stream>>>(dp, *out, seed, jitter_us, jm,
                                                                          (uint8_t *)c->construct_scratch, slots);
    return wf_cuda_check(cudaGetLastError(), "construct launch");
}
