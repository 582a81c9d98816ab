// Local search around the best plans: the scheduler re-ranks its uncommitted
// decisions when new information arrives (Section 3.5); here the k best
// evaluated plans (the elite) spawn children with a few point changes each,
// the children are evaluated by the sweep, and the elite keeps the k best of
// itself and its children.
//
//   mutate_kernel   a CTA per child: copy the parent's rows in 16-byte
//                   pieces, then apply the child's changes (one thread)
//   union_kernel    elite and child results side by side for the top-k key
//   pairs_kernel    one CTA: which elite slots leave, which children enter
//   replace_kernel  a CTA per entering child: its rows and results into the
//                   slot it takes
#include <algorithm>

#include "wf_internal.cuh"

namespace {

constexpr int kCopyThreads = 128;
constexpr int kMaxK = 1024;

__device__ __forceinline__ uint64_t mix64(uint64_t x)  // SplitMix64 output function
{
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
}

__host__ __device__ inline int64_t pad16(int64_t bytes) { return (bytes + 15) & ~(int64_t)15; }

// bytes (a multiple of 16) from src to dst, both 16-byte aligned, by the CTA.
__device__ __forceinline__ void copy_row(void *dst, const void *src, int64_t bytes)
{
    const uint4 *s = (const uint4 *)src;
    uint4 *d = (uint4 *)dst;
    for (int64_t i = threadIdx.x; i < bytes / 16; i += blockDim.x) d[i] = __ldg(s + i);
}

struct Row {
    uint8_t *place;
    uint16_t *order;
    uint32_t *fuse, *prefetch, *retain;
};

__device__ __forceinline__ Row row_of(const wf_plans &pl, int64_t p)
{
    Row r;
    r.place = (uint8_t *)pl.place + p * pl.place_stride;
    r.order = (uint16_t *)((uint8_t *)pl.order + p * pl.order_stride);
    r.fuse = (uint32_t *)((uint8_t *)pl.fuse + p * pl.bits_stride);
    r.prefetch = (uint32_t *)((uint8_t *)pl.prefetch + p * pl.bits_stride);
    r.retain = pl.retain ? (uint32_t *)((uint8_t *)pl.retain + p * pl.bits_stride) : nullptr;
    return r;
}

// Every row of plan b of `from` into plan a of `to` (padding to 16 bytes included).
__device__ __forceinline__ void copy_plan(const wf_dev_problem &dp, const wf_plans &to, int64_t a,
                                          const wf_plans &from, int64_t b)
{
    const int64_t N = dp.N, wbytes = pad16(4 * ((N + 31) / 32));
    const Row d = row_of(to, a), s = row_of(from, b);
    copy_row(d.place, s.place, pad16(N));
    copy_row(d.order, s.order, pad16(2 * N));
    copy_row(d.fuse, s.fuse, wbytes);
    copy_row(d.prefetch, s.prefetch, wbytes);
    if (d.retain && s.retain) copy_row(d.retain, s.retain, wbytes);
}

__device__ bool is_pred(const wf_dev_problem &dp, int32_t u, int32_t v)
{
    for (int32_t e = __ldg(dp.pred_off + v); e < __ldg(dp.pred_off + v + 1); ++e)
        if (__ldg(dp.pred_idx + e) == u) return true;
    return false;
}

// Child c copies parent c mod n_par; change s is decoded from
// h = mix(mix(mix(seed ^ round) ^ c) ^ s): h mod 4 picks a move to a fitting
// device (Eq. 8), a fuse flip (Eq. 3), a prefetch flip (Eq. 5) or an adjacent
// swap that never crosses a graph edge (Eq. 10).
__global__ void __launch_bounds__(kCopyThreads)
mutate_kernel(wf_dev_problem dp, wf_plans par, int64_t n_par, wf_plans ch, uint64_t seed, int64_t round,
              int32_t n_ops)
{
    const int32_t N = dp.N;
    for (int64_t c = blockIdx.x; c < ch.P; c += gridDim.x) {
        copy_plan(dp, ch, c, par, c % n_par);
        __syncthreads();
        if (threadIdx.x == 0) {
            const Row r = row_of(ch, c);
            for (int32_t s = 0; s < n_ops; ++s) {
                const uint64_t h = mix64(mix64(mix64(seed ^ (uint64_t)round) ^ (uint64_t)c) ^ (uint64_t)s);
                const uint32_t x = (uint32_t)(h >> 8), y = (uint32_t)(h >> 40);
                const uint32_t op = (uint32_t)h & 3u;
                if (op == 3u) {
                    if (N < 2) continue;
                    const int32_t i = (int32_t)(x % (uint32_t)(N - 1));
                    const int32_t u = r.order[i], v = r.order[i + 1];
                    if (v < N && !(u < N && is_pred(dp, u, v))) {
                        r.order[i] = (uint16_t)v;
                        r.order[i + 1] = (uint16_t)u;
                    }
                    continue;
                }
                const int32_t n = (int32_t)(x % (uint32_t)N);
                if (op == 0u) {
                    uint32_t fit = __ldg(dp.fitmask + n);
                    const int32_t f = __popc(fit);
                    if (f == 0) continue;
                    for (int32_t k = (int32_t)(y % (uint32_t)f); k > 0; --k) fit &= fit - 1;  // drop the lowest k
                    r.place[n] = (uint8_t)(__ffs((int)fit) - 1);
                } else if (op == 1u) {
                    r.fuse[n >> 5] ^= 1u << (n & 31);
                } else {
                    r.prefetch[n >> 5] ^= 1u << (n & 31);
                }
            }
        }
        __syncthreads();
    }
}

// Elite results (index < k) and child results (index k + c) side by side.
__global__ void union_kernel(wf_eval_out u, wf_eval_out elite, int32_t k, wf_eval_out child, int64_t C)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < k + C; i += (int64_t)gridDim.x * blockDim.x) {
        const wf_eval_out &s = i < k ? elite : child;
        const int64_t j = i < k ? i : i - k;
        u.makespan_us[i] = s.makespan_us[j];
        u.p95_us[i] = s.p95_us[j];
        u.gpu_us[i] = s.gpu_us[j];
        u.status[i] = s.status[j];
    }
}

// Exclusive prefix sum over the CTA (one value per thread, blockDim <= 1024).
__device__ int32_t block_exclusive_scan(int32_t v, int32_t *buf, int32_t *total)
{
    const int t = threadIdx.x;
    buf[t] = v;
    __syncthreads();
    for (int off = 1; off < (int)blockDim.x; off <<= 1) {
        const int32_t add = t >= off ? buf[t - off] : 0;
        __syncthreads();
        buf[t] += add;
        __syncthreads();
    }
    const int32_t incl = buf[t];
    if (t == (int)blockDim.x - 1) *total = incl;
    __syncthreads();
    return incl - v;
}

// ids: the k best of the union in key order.  Slots (ascending) whose plan
// left take the entering children (in key order): pairs[t] = {slot, child}.
__global__ void __launch_bounds__(kMaxK) pairs_kernel(const int32_t *ids, int32_t k, int2 *pairs, int32_t *npairs)
{
    __shared__ int32_t stays[kMaxK];
    __shared__ int32_t buf[kMaxK];
    __shared__ int32_t tot;
    const int t = threadIdx.x;
    if (t < k) stays[t] = 0;
    __syncthreads();
    const int32_t id = t < k ? ids[t] : 0;
    if (t < k && id < k) stays[id] = 1;
    __syncthreads();
    const int32_t enter = (t < k && id >= k) ? 1 : 0;
    const int32_t leave = (t < k && !stays[t]) ? 1 : 0;
    const int32_t e_at = block_exclusive_scan(enter, buf, &tot);
    const int32_t n_enter = tot;
    const int32_t l_at = block_exclusive_scan(leave, buf, &tot);
    if (enter) pairs[e_at].y = id - k;
    if (leave) pairs[l_at].x = t;
    if (t == 0) *npairs = n_enter;
}

__global__ void __launch_bounds__(kCopyThreads)
replace_kernel(wf_dev_problem dp, wf_plans elite, wf_eval_out elite_res, wf_plans ch, wf_eval_out ch_res,
               const int2 *pairs, const int32_t *npairs)
{
    const int32_t j = blockIdx.x;
    if (j >= *npairs) return;
    const int2 pr = pairs[j];
    copy_plan(dp, elite, pr.x, ch, pr.y);
    if (threadIdx.x == 0) {
        elite_res.makespan_us[pr.x] = ch_res.makespan_us[pr.y];
        elite_res.p95_us[pr.x] = ch_res.p95_us[pr.y];
        elite_res.gpu_us[pr.x] = ch_res.gpu_us[pr.y];
        elite_res.status[pr.x] = ch_res.status[pr.y];
    }
}

struct SearchScratch {
    wf_eval_out u;
    int32_t *ids;
    int2 *pairs;
    int32_t *npairs;
};

SearchScratch scratch_of(const wf_ctx *c)
{
    uint8_t *b = (uint8_t *)c->search_scratch;
    const int64_t n = c->max_P;
    SearchScratch s;
    s.u.makespan_us = (int64_t *)b;
    s.u.p95_us = s.u.makespan_us + n;
    s.u.gpu_us = s.u.p95_us + n;
    s.u.status = (uint32_t *)(s.u.gpu_us + n);
    uint8_t *t = b + ((24 * n + 4 * n + 255) & ~(int64_t)255);
    s.ids = (int32_t *)t;
    s.pairs = (int2 *)(t + 4 * kMaxK);
    s.npairs = (int32_t *)(t + 12 * kMaxK);
    return s;
}

int launch_mutate(wf_ctx *c, const wf_plans *par, const wf_plans *ch, uint64_t seed, int64_t round, int32_t n_ops,
                  cudaStream_t st)
{
    const int64_t blocks = std::min<int64_t>(ch->P, (int64_t)c->sms * 64);
    mutate_kernel<<<(unsigned)blocks, kCopyThreads, 0, st>>>(c->dp, *par, par->P, *ch, seed, round, n_ops);
    return wf_cuda_check(cudaGetLastError(), "mutate launch");
}

int launch_merge(wf_ctx *c, const wf_plans *elite, const wf_eval_out *elite_res, const wf_plans *ch,
                 const wf_eval_out *ch_res, cudaStream_t st)
{
    const SearchScratch s = scratch_of(c);
    const int32_t k = (int32_t)elite->P;
    const int64_t total = k + ch->P;
    const int64_t ublocks = std::min<int64_t>((total + 255) / 256, (int64_t)c->sms * 8);
    union_kernel<<<(unsigned)ublocks, 256, 0, st>>>(s.u, *elite_res, k, *ch_res, ch->P);
    int rc = wf_cuda_check(cudaGetLastError(), "union launch");
    if (!rc) rc = wf_launch_topk(c, &s.u, total, k, s.ids, nullptr, st);
    if (rc) return rc;
    pairs_kernel<<<1, ((k + 31) / 32) * 32, 0, st>>>(s.ids, k, s.pairs, s.npairs);
    rc = wf_cuda_check(cudaGetLastError(), "pairs launch");
    if (rc) return rc;
    replace_kernel<<<(unsigned)k, kCopyThreads, 0, st>>>(c->dp, *elite, *elite_res, *ch, *ch_res, s.pairs,
                                                         s.npairs);
    return wf_cuda_check(cudaGetLastError(), "replace launch");
}

int check_pair(const wf_ctx *c, const wf_plans *a, const wf_plans *b)
{
    if ((a->retain == nullptr) != (b->retain == nullptr))
        return wf_set_error(WF_EINVAL, "parents and children must both have retain rows or neither");
    (void)c;
    return WF_OK;
}

}  // namespace

size_t wf_search_scratch_bytes(int64_t max_P)
{
    return (size_t)((28 * max_P + 255) & ~(int64_t)255) + 16 * kMaxK + 256;
}

extern "C" int wf_mutate_plans(wf_ctx *c, const wf_plans *parents, const wf_plans *children, uint64_t seed,
                               int64_t round, int32_t n_ops, void *stream)
{
    if (!c || !parents || !children) return wf_set_error(WF_EINVAL, "NULL argument");
    int rc = wf_check_plans(c, parents, "parents");
    if (!rc) rc = wf_check_plans(c, children, "children");
    if (!rc) rc = check_pair(c, parents, children);
    if (rc) return rc;
    if (n_ops < 0 || n_ops > 4096) return wf_set_error(WF_EINVAL, "n_ops=%d outside 0..4096", n_ops);
    rc = wf_select_device(c);
    if (rc) return rc;
    return launch_mutate(c, parents, children, seed, round, n_ops, (cudaStream_t)stream);
}

static int check_merge(const wf_ctx *c, const wf_plans *elite, const wf_eval_out *elite_res,
                       const wf_plans *children, const wf_eval_out *child_res)
{
    if (!c || !elite || !elite_res || !children || !child_res) return wf_set_error(WF_EINVAL, "NULL argument");
    int rc = wf_check_plans(c, elite, "elite");
    if (!rc) rc = wf_check_plans(c, children, "children");
    if (!rc) rc = wf_check_out(elite_res, "elite results");
    if (!rc) rc = wf_check_out(child_res, "child results");
    if (!rc) rc = check_pair(c, elite, children);
    if (rc) return rc;
    if (elite->P > kMaxK) return wf_set_error(WF_EINVAL, "elite of %lld plans exceeds 1024", (long long)elite->P);
    if (elite->P + children->P > c->max_P)
        return wf_set_error(WF_EINVAL, "elite + children = %lld exceeds max_P=%lld",
                            (long long)(elite->P + children->P), (long long)c->max_P);
    return WF_OK;
}

extern "C" int wf_merge_elite(wf_ctx *c, const wf_plans *elite, const wf_eval_out *elite_res,
                              const wf_plans *children, const wf_eval_out *child_res, void *stream)
{
    int rc = check_merge(c, elite, elite_res, children, child_res);
    if (!rc) rc = wf_select_device(c);
    if (rc) return rc;
    return launch_merge(c, elite, elite_res, children, child_res, (cudaStream_t)stream);
}

extern "C" int wf_local_search(wf_ctx *c, const wf_plans *elite, const wf_eval_out *elite_res,
                               const wf_plans *children, const wf_eval_out *child_res, uint64_t seed,
                               int64_t round0, int32_t rounds, int32_t n_ops, void *stream)
{
    int rc = check_merge(c, elite, elite_res, children, child_res);
    if (rc) return rc;
    if (rounds < 0) return wf_set_error(WF_EINVAL, "rounds < 0");
    if (n_ops < 0 || n_ops > 4096) return wf_set_error(WF_EINVAL, "n_ops=%d outside 0..4096", n_ops);
    rc = wf_select_device(c);
    if (rc) return rc;
    const cudaStream_t st = (cudaStream_t)stream;
    for (int32_t r = 0; r < rounds && !rc; ++r) {
        rc = launch_mutate(c, elite, children, seed, round0 + r, n_ops, st);
        if (!rc) rc = wf_launch_eval(c, children, child_res, st);
        if (!rc) rc = launch_merge(c, elite, elite_res, children, child_res, st);
    }
    return rc;
}
