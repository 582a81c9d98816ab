// Local search around the best plans: the scheduler re-ranks its uncommitted
// decisions when new information arrives (Section 3.5); here the k best
// evaluated plans (the elite) spawn children with a few point changes each,
// the children are evaluated by the sweep, and the elite keeps the k best of
// itself and its children.
//
//   mutate_kernel   a CTA per child: the parent's rows copied to the child
//                   in 16-byte pieces, then the child's changes applied by
//                   one thread; for short rows mutate_staged_kernel, a warp
//                   per child, stages the rows in shared memory with bulk
//                   copies and decodes the changes on all lanes
//   union_kernel    elite and child results side by side for the top-k key
//   pairs_kernel    one CTA: which elite slots leave, which children enter
//   replace_kernel  a CTA per entering child: its rows and results into the
//                   slot it takes
#include <algorithm>

#include "wf_internal.cuh"

namespace {

constexpr int kCopyThreads = 128;
constexpr int kMutWarps = 8;                // children a staged mutate CTA works on at once, a warp each
constexpr int64_t kStagedMax = 96 * 1024;  // shared memory of a staged mutate CTA, at most
constexpr int kMaxK = 1024;

__device__ __forceinline__ uint64_t mix64(uint64_t x)  // SplitMix64 output function
{
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
}

__host__ __device__ inline int64_t pad16(int64_t bytes) { return (bytes + 15) & ~(int64_t)15; }

// bytes (a multiple of 16) from src to dst, both 16-byte aligned, by `lanes`
// threads (this one is `lane`), four pieces a thread in flight (kWide) or one.
// src is global memory that no thread writes during the kernel (read through
// the non-coherent path).
template <bool kWide = true>
__device__ __forceinline__ void copy_row(void *dst, const void *src, int64_t bytes, int lane, int lanes)
{
    const uint4 *s = (const uint4 *)src;
    uint4 *d = (uint4 *)dst;
    const int64_t n = bytes / 16;
    int64_t i = lane;
    for (; kWide && i + 3 * lanes < n; i += 4 * lanes) {
        const uint4 a = __ldg(s + i), b = __ldg(s + i + lanes), c = __ldg(s + i + 2 * lanes),
                    e = __ldg(s + i + 3 * lanes);
        d[i] = a;
        d[i + lanes] = b;
        d[i + 2 * lanes] = c;
        d[i + 3 * lanes] = e;
    }
    for (; i < n; i += lanes) d[i] = __ldg(s + i);
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
                                          const wf_plans &from, int64_t b, int lane, int lanes)
{
    const int64_t N = dp.N, wbytes = pad16(4 * ((N + 31) / 32));
    const Row d = row_of(to, a), s = row_of(from, b);
    copy_row(d.place, s.place, pad16(N), lane, lanes);
    copy_row(d.order, s.order, pad16(2 * N), lane, lanes);
    copy_row(d.fuse, s.fuse, wbytes, lane, lanes);
    copy_row(d.prefetch, s.prefetch, wbytes, lane, lanes);
    if (d.retain && s.retain) copy_row(d.retain, s.retain, wbytes, lane, lanes);
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
// swap that never crosses a graph edge (Eq. 10).  The changes apply in turn.
struct Change {
    uint32_t kind;  // 0 none, 1 move node a to device b, 2 fuse flip of a, 3 prefetch flip of a,
                    // 4 swap of positions a and a + 1 (when legal at that point)
    int32_t a, b;
};

// hc = mix(mix(seed ^ round) ^ c), shared by the child's changes.
__device__ __forceinline__ Change decode_change(const wf_dev_problem &dp, uint64_t hc, int32_t s)
{
    const int32_t N = dp.N;
    const uint64_t h = mix64(hc ^ (uint64_t)s);
    const uint32_t x = (uint32_t)(h >> 8), y = (uint32_t)(h >> 40);
    const uint32_t op = (uint32_t)h & 3u;
    Change g{0u, 0, 0};
    if (op == 3u) {
        if (N >= 2) g = Change{4u, (int32_t)(x % (uint32_t)(N - 1)), 0};
        return g;
    }
    const int32_t n = (int32_t)(x % (uint32_t)N);
    if (op == 0u) {
        uint32_t fit = __ldg(dp.fitmask + n);
        const int32_t f = __popc(fit);
        if (f == 0) return g;
        for (int32_t k = (int32_t)(y % (uint32_t)f); k > 0; --k) fit &= fit - 1;  // drop the lowest k
        return Change{1u, n, __ffs((int)fit) - 1};
    }
    return Change{op == 1u ? 2u : 3u, n, 0};
}

__device__ __forceinline__ void apply_change(const wf_dev_problem &dp, const Row &r, const Change &g)
{
    const int32_t N = dp.N, a = g.a;
    if (g.kind == 4u) {
        const int32_t u = r.order[a], v = r.order[a + 1];
        if (v < N && !(u < N && is_pred(dp, u, v))) {
            r.order[a] = (uint16_t)v;
            r.order[a + 1] = (uint16_t)u;
        }
    } else if (g.kind == 1u) {
        r.place[a] = (uint8_t)g.b;
    } else if (g.kind == 2u) {
        r.fuse[a >> 5] ^= 1u << (a & 31);
    } else if (g.kind == 3u) {
        r.prefetch[a >> 5] ^= 1u << (a & 31);
    }
}

__device__ __forceinline__ uint64_t child_hash(uint64_t seed, int64_t round, int64_t c)
{
    return mix64(mix64(seed ^ (uint64_t)round) ^ (uint64_t)c);
}

// Long rows: a CTA per child, the changes applied to the child's rows in
// global memory.
__global__ void __launch_bounds__(kCopyThreads)
mutate_kernel(wf_dev_problem dp, wf_plans par, int64_t n_par, wf_plans ch, uint64_t seed, int64_t round,
              int32_t n_ops)
{
    for (int64_t c = blockIdx.x; c < ch.P; c += gridDim.x) {
        copy_plan(dp, ch, c, par, c % n_par, (int)threadIdx.x, (int)blockDim.x);
        __syncthreads();
        if (threadIdx.x == 0) {
            const Row r = row_of(ch, c);
            const uint64_t hc = child_hash(seed, round, c);
            for (int32_t s = 0; s < n_ops; ++s) apply_change(dp, r, decode_change(dp, hc, s));
        }
        __syncthreads();
    }
}

// Shared-memory address of a generic pointer into this CTA's shared memory.
__device__ __forceinline__ uint32_t smem_addr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t *bar)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Arms bar for one phase that completes when `bytes` have landed.
__device__ __forceinline__ void mbar_expect(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

// Waits for bar's phase of the given parity: at most 2^20 polls, each with a
// suspend-time hint of 1 us; one poll takes about 4 us on a GB300, so the
// wait gives up after about 4 s.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity)
{
    for (uint32_t it = 0; it < (1u << 20); ++it) {
        uint32_t done;
        asm volatile("{\n\t.reg .pred p;\n\t"
                     "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
                     "selp.u32 %0, 1, 0, p;\n\t}"
                     : "=r"(done)
                     : "r"(smem_addr(bar)), "r"(parity), "r"(1000u)
                     : "memory");
        if (done) return true;
    }
    return false;
}

// 1-D bulk copy (TMA) of `bytes` (a multiple of 16, both ends 16-byte
// aligned) from global memory into this CTA's shared memory, counted on bar.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_addr(dst)),
                 "l"(src), "r"(bytes), "r"(smem_addr(bar))
                 : "memory");
}

// 1-D bulk copy from shared memory to global memory, in the thread's open
// bulk group.
__device__ __forceinline__ void bulk_store(void *dst, const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_addr(src)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// The thread's bulk stores have read their shared-memory sources.
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// The thread's bulk stores are complete.
__device__ __forceinline__ void bulk_wait() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// Orders this thread's shared-memory accesses before later bulk copies.
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Bytes of one warp's staged rows: place, order, fuse, prefetch and, when
// both batches carry one, retain, each padded to 16 bytes.
__host__ __device__ inline int64_t staged_row_bytes(int64_t N, bool retain)
{
    return pad16(N) + pad16(2 * N) + (retain ? 3 : 2) * pad16(4 * ((N + 31) / 32));
}

// Short rows: a warp per child.  Lane 0 stages the parent's rows in the
// warp's slice of shared memory with bulk copies while the lanes decode the
// child's changes (lane t the t-th of each group of 32); lane 0 then applies
// them on chip, in turn, and writes the rows to the child with bulk copies.
// The slice is reloaded only after those stores have read it.  A bulk load
// that has not landed after the bounded wait sets error word 3; the warp then
// waits once more, with the same bound, for the copies it issued (an issued
// bulk copy cannot be withdrawn, and an unbounded wait could hang the GPU),
// stops taking children, and drains its own bulk stores before the CTA
// exits.
__global__ void __launch_bounds__(32 * kMutWarps, 4)
mutate_staged_kernel(wf_dev_problem dp, wf_plans par, int64_t n_par, wf_plans ch, uint64_t seed, int64_t round,
                     int32_t n_ops)
{
    extern __shared__ __align__(16) uint8_t msm[];
    __shared__ uint64_t bars[kMutWarps];
    const int64_t N = dp.N, pl = pad16(N), ol = pad16(2 * N), wb = pad16(4 * ((N + 31) / 32));
    const bool ret = par.retain != nullptr && ch.retain != nullptr;
    const int lane = (int)(threadIdx.x & 31), warp = (int)(threadIdx.x >> 5);
    uint8_t *base = msm + warp * staged_row_bytes(N, ret);
    uint64_t *bar = &bars[warp];
    Row sm;
    sm.place = base;
    sm.order = (uint16_t *)(base + pl);
    sm.fuse = (uint32_t *)(base + pl + ol);
    sm.prefetch = (uint32_t *)(base + pl + ol + wb);
    sm.retain = ret ? (uint32_t *)(base + pl + ol + 2 * wb) : nullptr;
    const uint32_t bytes = (uint32_t)staged_row_bytes(N, ret);
    if (lane == 0) mbar_init(bar);
    __syncwarp();
    uint32_t parity = 0;
    for (int64_t c = (int64_t)blockIdx.x * kMutWarps + warp; c < ch.P; c += (int64_t)gridDim.x * kMutWarps) {
        const Row s = row_of(par, c % n_par), d = row_of(ch, c);
        if (lane == 0) {
            bulk_wait_read();  // the previous child's stores are done with the slice
            fence_async_shared();
            mbar_expect(bar, bytes);
            bulk_load(sm.place, s.place, (uint32_t)pl, bar);
            bulk_load(sm.order, s.order, (uint32_t)ol, bar);
            bulk_load(sm.fuse, s.fuse, (uint32_t)wb, bar);
            bulk_load(sm.prefetch, s.prefetch, (uint32_t)wb, bar);
            if (ret) bulk_load(sm.retain, s.retain, (uint32_t)wb, bar);
        }
        const uint64_t hc = child_hash(seed, round, c);
        Change g = lane < n_ops ? decode_change(dp, hc, lane) : Change{0u, 0, 0};
        bool landed = true;
        if (lane == 0) {
            landed = mbar_wait(bar, parity);
            if (!landed) {
                atomicExch(dp.err, 3);
                mbar_wait(bar, parity);
            }
        }
        parity ^= 1u;
        if (!__shfl_sync(0xFFFFFFFFu, landed, 0)) break;
        for (int32_t g0 = 0; g0 < n_ops; g0 += 32) {
            if (g0 > 0) g = g0 + lane < n_ops ? decode_change(dp, hc, g0 + lane) : Change{0u, 0, 0};
            const int cnt = min(32, n_ops - g0);
            for (int t = 0; t < cnt; ++t) {
                const Change e{__shfl_sync(0xFFFFFFFFu, g.kind, t), __shfl_sync(0xFFFFFFFFu, g.a, t),
                               __shfl_sync(0xFFFFFFFFu, g.b, t)};
                if (lane == 0) apply_change(dp, sm, e);
            }
        }
        if (lane == 0) {
            fence_async_shared();  // lane 0's changes are seen by the bulk stores
            bulk_store(d.place, sm.place, (uint32_t)pl);
            bulk_store(d.order, sm.order, (uint32_t)ol);
            bulk_store(d.fuse, sm.fuse, (uint32_t)wb);
            bulk_store(d.prefetch, sm.prefetch, (uint32_t)wb);
            if (ret) bulk_store(d.retain, sm.retain, (uint32_t)wb);
            bulk_commit();
        }
    }
    if (lane == 0) bulk_wait();
}

// The bounded wait's expiry path: an mbarrier armed for 16 bytes that no copy
// delivers, so the wait gives up and sets error word 3.
__global__ void wait_expiry_kernel(int *err)
{
    __shared__ uint64_t bar;
    mbar_init(&bar);
    mbar_expect(&bar, 16);
    if (!mbar_wait(&bar, 0)) atomicExch(err, 3);
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
    copy_plan(dp, elite, pr.x, ch, pr.y, (int)threadIdx.x, (int)blockDim.x);
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
    const int64_t staged = kMutWarps * staged_row_bytes(c->dp.N, par->retain && ch->retain);
    if (staged <= kStagedMax) {
        // One wave of resident CTAs, each warp striding over the children.
        int rc = wf_cuda_check(cudaFuncSetAttribute(mutate_staged_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                    (int)staged), "mutate smem attribute");
        int per_sm = 0;
        if (!rc) rc = wf_cuda_check(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, mutate_staged_kernel,
                                                                                    32 * kMutWarps, (size_t)staged),
                                    "mutate occupancy");
        if (rc) return rc;
        const int64_t blocks = std::min<int64_t>((ch->P + kMutWarps - 1) / kMutWarps,
                                                 (int64_t)c->sms * std::max(per_sm, 1));
        mutate_staged_kernel<<<(unsigned)blocks, 32 * kMutWarps, (size_t)staged, st>>>(c->dp, *par, par->P, *ch,
                                                                                       seed, round, n_ops);
    } else {
        const int64_t blocks = std::min<int64_t>(ch->P, (int64_t)c->sms * 64);
        mutate_kernel<<<(unsigned)blocks, kCopyThreads, 0, st>>>(c->dp, *par, par->P, *ch, seed, round, n_ops);
    }
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

extern "C" int wf_ctx_check_wait_expiry(wf_ctx *c, void *stream)
{
    if (!c) return wf_set_error(WF_EINVAL, "NULL context");
    int rc = wf_select_device(c);
    if (rc) return rc;
    wait_expiry_kernel<<<1, 1, 0, (cudaStream_t)stream>>>(c->dp.err);
    return wf_cuda_check(cudaGetLastError(), "wait expiry launch");
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
