// Top-k of evaluated plans (row a12) by the key (status != 0, makespan, p95,
// gpu, plan index), ascending.
//
//  1. threshold: T, a 64-bit key (status != 0) << 63 | makespan that at
//     least k plans' keys do not exceed;
//  2. compact: every plan whose 64-bit key is at most T becomes a candidate
//     (all ties with T included, so the full key decides among them);
//  3. final: one CTA sorts the candidates by the full key in shared memory
//     (bitonic network) and writes the first k; more candidates than one
//     tile (massive ties) are folded tile by tile into the running best k.
//
// Up to kOneCta plans, one CTA does all three with the keys staged in shared
// memory (one launch): T is the exact k-th smallest key, found by radix
// selection (8 bits a pass, the digit found by a warp scan of the
// histogram), so usually about k candidates reach the sort.  Beyond, T is
// first the smallest of the tiles' own k-th keys (kth_kernel, one CTA a
// tile); the final CTA then runs the same exact selection over those
// candidates before sorting.
#include <algorithm>

#include "wf_internal.cuh"

namespace {

constexpr int kTile = 2048;
constexpr int kThreads = 1024;

struct Cand {
    int64_t mk, p95, gpu;
    int32_t id;
    uint32_t bad;  // 0 valid, 1 invalid plan, 2 padding
};

__device__ __forceinline__ bool before(const Cand &a, const Cand &b)
{
    if (a.bad != b.bad) return a.bad < b.bad;
    if (a.mk != b.mk) return a.mk < b.mk;
    if (a.p95 != b.p95) return a.p95 < b.p95;
    if (a.gpu != b.gpu) return a.gpu < b.gpu;
    return a.id < b.id;
}

__device__ __forceinline__ Cand padding()
{
    Cand c;
    c.mk = c.p95 = c.gpu = WF_INF64;
    c.id = INT32_MAX;
    c.bad = 2;
    return c;
}

__device__ __forceinline__ uint64_t key64(const wf_eval_out &res, int64_t p)
{
    return ((uint64_t)(res.status[p] != 0) << 63) | (uint64_t)res.makespan_us[p];
}

// Scratch words: [0] T (u64), [1] candidate count, then the candidates.
struct TopkScratch {
    unsigned long long *T;
    unsigned int *count;
    Cand *cand;
};

__device__ __forceinline__ TopkScratch scratch_of(void *base)
{
    TopkScratch s;
    s.T = (unsigned long long *)base;
    s.count = (unsigned int *)((uint8_t *)base + 8);
    s.cand = (Cand *)((uint8_t *)base + 64);
    return s;
}

// Warp-wide minimum / maximum of 64-bit values (two 32-bit reductions each).
__device__ __forceinline__ uint64_t warp_min64(uint64_t v)
{
    const uint32_t hi = __reduce_min_sync(0xFFFFFFFFu, (uint32_t)(v >> 32));
    const uint32_t lo = __reduce_min_sync(0xFFFFFFFFu, (uint32_t)(v >> 32) == hi ? (uint32_t)v : 0xFFFFFFFFu);
    return ((uint64_t)hi << 32) | lo;
}

__device__ __forceinline__ uint64_t warp_max64(uint64_t v)
{
    const uint32_t hi = __reduce_max_sync(0xFFFFFFFFu, (uint32_t)(v >> 32));
    const uint32_t lo = __reduce_max_sync(0xFFFFFFFFu, (uint32_t)(v >> 32) == hi ? (uint32_t)v : 0u);
    return ((uint64_t)hi << 32) | lo;
}

// The radix passes can start at the highest byte in which the keys differ:
// the bytes above it are the same in every key (those of the smallest).
// From this thread's smallest and largest keys, the block's range gives
// prefix and the first pass's shift (-8: all keys are equal, no pass).
__device__ void first_pass(uint64_t mn, uint64_t mx, unsigned long long *wmin, unsigned long long *wmax,
                           unsigned long long &prefix, int &first)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    mn = warp_min64(mn);
    mx = warp_max64(mx);
    if (lane == 0) { wmin[warp] = mn; wmax[warp] = mx; }
    __syncthreads();
    if (warp == 0) {
        const int nw = (int)(blockDim.x >> 5);
        mn = warp_min64(lane < nw ? wmin[lane] : ~0ull);
        mx = warp_max64(lane < nw ? wmax[lane] : 0ull);
        if (lane == 0) {
            const uint64_t diff = mn ^ mx;
            if (diff == 0) {
                prefix = mn;
                first = -8;
            } else {
                const int shift = ((63 - __clzll((long long)diff)) / 8) * 8;
                prefix = shift == 56 ? 0ull : (mn & (~0ull << (shift + 8)));
                first = shift;
            }
        }
    }
    __syncthreads();
}

// The digit of the k-th smallest key in this radix pass: warp 0 scans the
// 256-bucket histogram (8 buckets a lane), finds the bucket holding rank,
// and narrows prefix and rank to it.
__device__ __forceinline__ void pick_digit(const unsigned int *hist, int shift, unsigned long long &prefix,
                                           long long &rank)
{
    const int lane = threadIdx.x & 31;
    unsigned int h[8], sum = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) { h[j] = hist[8 * lane + j]; sum += h[j]; }
    unsigned int inc = sum;  // inclusive prefix over lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int v = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += v;
    }
    const long long r = rank;
    const unsigned int over = __ballot_sync(0xFFFFFFFFu, (long long)inc > r);
    const int src = __ffs((int)over) - 1;  // the lane whose buckets hold rank (rank < count)
    if (lane == src) {
        long long left = r - (long long)(inc - sum);
        int b = 0;
        while ((long long)h[b] <= left) { left -= h[b]; ++b; }
        rank = left;
        prefix |= (unsigned long long)(8 * lane + b) << shift;
    }
}


// The second and third terms of the key: p95 and GPU time, or (Eq. 12's
// window terms) minus the timely prefetches and the lifecycle overhead.
struct Terms {
    const int64_t *a, *b;
    int64_t sa;  // +1, or -1 for a term ranked largest first
};

__device__ __forceinline__ Cand cand_of(const wf_eval_out &res, const Terms &tm, int64_t p)
{
    Cand c;
    c.mk = res.makespan_us[p];
    c.p95 = tm.sa * tm.a[p];
    c.gpu = tm.b[p];
    c.id = (int32_t)p;
    c.bad = res.status[p] != 0 ? 1u : 0u;
    return c;
}

__global__ void compact_kernel(wf_eval_out res, Terms tm, int64_t P, void *scr)
{
    const TopkScratch s = scratch_of(scr);
    const unsigned long long T = *s.T;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x) {
        if (key64(res, p) > T) continue;
        s.cand[atomicAdd(s.count, 1u)] = cand_of(res, tm, p);
    }
}

// The k-th smallest of kk[0, n) (shared memory, k <= n), by radix selection
// from the highest byte in which the keys differ.  Every thread of the CTA
// calls it with the smallest and largest of the keys it wrote.
__device__ unsigned long long radix_kth(const unsigned long long *kk, int64_t n, int32_t k, uint64_t mn,
                                        uint64_t mx)
{
    __shared__ unsigned int hist[256];
    __shared__ unsigned long long prefix;
    __shared__ long long rank;
    __shared__ unsigned long long wmin[32], wmax[32];
    __shared__ int shift0;
    if (threadIdx.x == 0) rank = k - 1;
    first_pass(mn, mx, wmin, wmax, prefix, shift0);
    for (int shift = shift0; shift >= 0; shift -= 8) {
        for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        const unsigned long long hi = shift == 56 ? 0ull : (~0ull << (shift + 8));
        const unsigned long long pre = prefix;
        for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
            const uint64_t v = kk[i];
            if ((v & hi) == pre) atomicAdd(&hist[(v >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (threadIdx.x < 32) pick_digit(hist, shift, prefix, rank);
        __syncthreads();
    }
    return prefix;
}

// Beyond kOneCta plans: each CTA finds the k-th smallest 64-bit key of a
// tile of kKth plans and lowers T to it.  Every tile's k-th key bounds the
// batch's k-th from above, so the keys at most T (the smallest bound) hold
// the k best, ties included; compact and final take it from there.  T starts
// at all ones and the candidate count at 0 (host memsets).
constexpr int kKth = 4096;

__global__ void __launch_bounds__(kThreads)
kth_kernel(wf_eval_out res, int64_t P, int32_t k, void *scr)
{
    __shared__ unsigned long long v[kKth];
    const TopkScratch s = scratch_of(scr);
    const int64_t base = (int64_t)blockIdx.x * kKth;
    const int n = P - base < kKth ? (int)(P - base) : kKth;
    if (n < k) return;  // a short last tile bounds nothing
    uint64_t mn = ~0ull, mx = 0;
    for (int u = threadIdx.x; u < n; u += blockDim.x) {
        const uint64_t x = key64(res, base + u);
        v[u] = x;
        mn = min(mn, x);
        mx = max(mx, x);
    }
    const unsigned long long T = radix_kth(v, n, k, mn, mx);
    if (threadIdx.x == 0) atomicMin(s.T, T);
}

// Sorts t[0, len) ascending; len is a power of two, at most kTile.
__device__ void bitonic_sort(Cand *t, int len)
{
    for (int size = 2; size <= len; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncthreads();
            for (int u = threadIdx.x; u < len / 2; u += blockDim.x) {
                const int i = 2 * stride * (u / stride) + (u % stride);
                const int j = i + stride;
                const bool up = (i & size) == 0;
                const Cand a = t[i], b = t[j];
                if (before(b, a) == up) { t[i] = b; t[j] = a; }
            }
        }
    }
    __syncthreads();
}

__device__ void write_first(const Cand *t, int32_t k, int32_t *ids, int64_t *keys, int64_t sa)
{
    for (int u = threadIdx.x; u < k; u += blockDim.x) {
        ids[u] = t[u].id;
        if (keys) {
            keys[3 * u] = t[u].mk;
            keys[3 * u + 1] = sa * t[u].p95;
            keys[3 * u + 2] = t[u].gpu;
        }
    }
}

// Items to rank: the plans of an evaluated batch, or the candidates
// compacted into scratch.
struct PlanSrc {
    wf_eval_out res;
    Terms tm;
    __device__ uint64_t key(int64_t i) const { return key64(res, i); }
    __device__ Cand get(int64_t i) const { return cand_of(res, tm, i); }
};

struct CandSrc {
    const Cand *cand;
    __device__ uint64_t key(int64_t i) const { return ((uint64_t)cand[i].bad << 63) | (uint64_t)cand[i].mk; }
    __device__ Cand get(int64_t i) const { return cand[i]; }
};

// Sorts the items of src[0, n) that qualify (all when kk is null, else those
// with kk[i] <= T) by the full key, a tile at a time: the running best k stay
// in t[0, k) and each round fills the rest of the tile; writes the first k.
template <class Src>
__device__ void fold_sort(const Src &src, int64_t n, int32_t k, const unsigned long long *kk,
                          unsigned long long T, Cand *t, int32_t *ids, int64_t *keys, int64_t sa)
{
    int len = 64;
    while (len < n && len < kTile) len <<= 1;
    int64_t next = 0;
    bool first = true;
    while (first || next < n) {
        const int base = first ? 0 : k;
        for (int u = threadIdx.x; u < len - base; u += blockDim.x) {
            const int64_t c = next + u;
            t[base + u] = c < n && (!kk || kk[c] <= T) ? src.get(c) : padding();
        }
        next += len - base;
        first = false;
        bitonic_sort(t, len);
    }
    write_first(t, k, ids, keys, sa);
}

// The k best of src[0, n) (k <= n <= kOneCta): the 64-bit keys staged in kk,
// T the exact k-th smallest of them, the items with keys at most T gathered
// into t and sorted there by the full key.
template <class Src>
__device__ void select_and_sort(const Src &src, int64_t n, int32_t k, unsigned long long *kk, Cand *t,
                                int32_t *ids, int64_t *keys, int64_t sa)
{
    __shared__ unsigned int m;
    if (threadIdx.x == 0) m = 0;
    uint64_t mn = ~0ull, mx = 0;
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
        const uint64_t v = src.key(i);
        kk[i] = v;
        mn = min(mn, v);
        mx = max(mx, v);
    }
    const unsigned long long T = radix_kth(kk, n, k, mn, mx);
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
        if (kk[i] > T) continue;
        const unsigned int slot = atomicAdd(&m, 1u);
        if (slot < (unsigned)kTile) t[slot] = src.get(i);
    }
    __syncthreads();
    const unsigned int cnt = m;
    if (cnt > (unsigned)kTile) {  // massive ties with T
        fold_sort(src, n, k, kk, T, t, ids, keys, sa);
        return;
    }
    int len = 64;
    while (len < (int)cnt) len <<= 1;
    for (int u = (int)cnt + threadIdx.x; u < len; u += blockDim.x) t[u] = padding();
    bitonic_sort(t, len);
    write_first(t, k, ids, keys, sa);
}

constexpr int64_t kOneCta = 16384;  // keys staged in shared memory by one CTA

__global__ void __launch_bounds__(kThreads)
final_kernel(int32_t k, void *scr, int32_t *ids, int64_t *keys, int64_t sa)
{
    extern __shared__ __align__(16) uint8_t tsm[];
    Cand *t = (Cand *)tsm;
    unsigned long long *kk = (unsigned long long *)(tsm + kTile * sizeof(Cand));  // [kOneCta]
    const TopkScratch s = scratch_of(scr);
    const int64_t n = *s.count;
    const CandSrc src{s.cand};
    if (n <= kOneCta) select_and_sort(src, n, k, kk, t, ids, keys, sa);
    else fold_sort(src, n, k, nullptr, 0ull, t, ids, keys, sa);
}

__global__ void __launch_bounds__(kThreads)
topk_one_kernel(wf_eval_out res, Terms tm, int64_t P, int32_t k, int32_t *ids, int64_t *keys)
{
    extern __shared__ __align__(16) uint8_t tsm[];
    Cand *t = (Cand *)tsm;
    unsigned long long *kk = (unsigned long long *)(tsm + kTile * sizeof(Cand));  // [P]
    select_and_sort(PlanSrc{res, tm}, P, k, kk, t, ids, keys, tm.sa);
}

}  // namespace

size_t wf_topk_scratch_bytes(int64_t max_P)
{
    return 64 + sizeof(Cand) * (size_t)max_P;
}

int wf_launch_topk(wf_ctx *ctx, const wf_eval_out *res, int64_t P, int32_t k, int32_t *ids,
                   int64_t *keys, cudaStream_t st, const int64_t *term2, const int64_t *term3, int64_t sign2)
{
    const Terms tm{term2 ? term2 : res->p95_us, term3 ? term3 : res->gpu_us, term2 ? sign2 : 1};
    const size_t smem = kTile * sizeof(Cand) + 8 * (size_t)std::min<int64_t>(P, kOneCta);
    if (P <= kOneCta) {
        int rc = wf_cuda_check(cudaFuncSetAttribute(topk_one_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                    (int)smem), "topk smem attribute");
        if (rc) return rc;
        topk_one_kernel<<<1, kThreads, smem, st>>>(*res, tm, P, k, ids, keys);
        return wf_cuda_check(cudaGetLastError(), "topk launch");
    }
    int rc = wf_cuda_check(cudaFuncSetAttribute(final_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)smem), "topk smem attribute");
    if (rc) return rc;
    // T = all ones, candidate count = 0 (scratch words 0 and 1).
    rc = wf_cuda_check(cudaMemsetAsync(ctx->topk_scratch, 0xFF, 8, st), "topk reset");
    if (!rc) rc = wf_cuda_check(cudaMemsetAsync((uint8_t *)ctx->topk_scratch + 8, 0, 4, st), "topk reset");
    if (rc) return rc;
    kth_kernel<<<(unsigned)((P + kKth - 1) / kKth), kThreads, 0, st>>>(*res, P, k, ctx->topk_scratch);
    const int64_t blocks = std::min<int64_t>((P + 255) / 256, (int64_t)ctx->sms * 8);
    compact_kernel<<<(unsigned)blocks, 256, 0, st>>>(*res, tm, P, ctx->topk_scratch);
    final_kernel<<<1, kThreads, smem, st>>>(k, ctx->topk_scratch, ids, keys, tm.sa);
    return wf_cuda_check(cudaGetLastError(), "topk launch");
}
