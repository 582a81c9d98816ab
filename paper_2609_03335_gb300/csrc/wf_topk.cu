// Top-k of evaluated plans (row a12) by the key (status != 0, makespan, p95,
// gpu, plan index), ascending.
//
//  1. select: one CTA finds T, the k-th smallest of the 64-bit keys
//     (status != 0) << 63 | makespan, by radix selection (8 bits a pass);
//  2. compact: every plan whose 64-bit key is at most T becomes a candidate
//     (all ties with T included, so the full key decides among them);
//  3. final: one CTA sorts the candidates by the full key in shared memory
//     (bitonic network) and writes the first k; more candidates than one
//     tile (massive ties) are folded tile by tile into the running best k.
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

constexpr int64_t kSelectShared = 20480;  // keys staged in shared memory up to this many plans

template <bool kStaged>
__global__ void __launch_bounds__(kThreads)
select_kernel(wf_eval_out res, int64_t P, int32_t k, void *scr)
{
    extern __shared__ unsigned long long keys[];
    __shared__ unsigned int hist[256];
    __shared__ unsigned long long prefix;
    __shared__ long long rank;
    const TopkScratch s = scratch_of(scr);
    if (threadIdx.x == 0) { prefix = 0; rank = k - 1; *s.count = 0; }
    if (kStaged)
        for (int64_t p = threadIdx.x; p < P; p += blockDim.x) keys[p] = key64(res, p);
    __syncthreads();
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        const unsigned long long hi = shift == 56 ? 0ull : (~0ull << (shift + 8));
        const unsigned long long pre = prefix;
        for (int64_t p = threadIdx.x; p < P; p += blockDim.x) {
            const uint64_t v = kStaged ? keys[p] : key64(res, p);
            if ((v & hi) == pre) atomicAdd(&hist[(v >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            long long r = rank;
            int b = 0;
            while ((long long)hist[b] <= r) { r -= hist[b]; ++b; }
            rank = r;
            prefix |= (unsigned long long)b << shift;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) *s.T = prefix;
}

__global__ void compact_kernel(wf_eval_out res, int64_t P, void *scr)
{
    const TopkScratch s = scratch_of(scr);
    const unsigned long long T = *s.T;
    for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < P; p += (int64_t)gridDim.x * blockDim.x) {
        if (key64(res, p) > T) continue;
        Cand c;
        c.mk = res.makespan_us[p];
        c.p95 = res.p95_us[p];
        c.gpu = res.gpu_us[p];
        c.id = (int32_t)p;
        c.bad = res.status[p] != 0 ? 1u : 0u;
        s.cand[atomicAdd(s.count, 1u)] = c;
    }
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

__global__ void __launch_bounds__(kThreads)
final_kernel(int32_t k, void *scr, int32_t *ids, int64_t *keys)
{
    extern __shared__ Cand t[];
    const TopkScratch s = scratch_of(scr);
    const int64_t n = *s.count;
    // One network of the smallest power-of-two size that holds every candidate
    // when they fit a tile; otherwise the running best k occupy t[0, k) and
    // each round fills the rest of a full tile with new candidates.
    int len = 64;
    while (len < n && len < kTile) len <<= 1;
    int64_t next = 0;
    bool first = true;
    while (first || next < n) {
        const int base = first ? 0 : k;
        for (int u = threadIdx.x; u < len - base; u += blockDim.x) {
            const int64_t c = next + u;
            t[base + u] = c < n ? s.cand[c] : padding();
        }
        next += len - base;
        first = false;
        bitonic_sort(t, len);
    }
    for (int u = threadIdx.x; u < k; u += blockDim.x) {
        ids[u] = t[u].id;
        if (keys) {
            keys[3 * u] = t[u].mk;
            keys[3 * u + 1] = t[u].p95;
            keys[3 * u + 2] = t[u].gpu;
        }
    }
}

}  // namespace

size_t wf_topk_scratch_bytes(int64_t max_P)
{
    return 64 + sizeof(Cand) * (size_t)max_P;
}

int wf_launch_topk(wf_ctx *ctx, const wf_eval_out *res, int64_t P, int32_t k, int32_t *ids,
                   int64_t *keys, cudaStream_t st)
{
    const size_t smem = kTile * sizeof(Cand);
    int rc = wf_cuda_check(cudaFuncSetAttribute(final_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)smem), "topk smem attribute");
    if (rc) return rc;
    if (P <= kSelectShared) {
        const size_t ks = 8 * (size_t)P;
        rc = wf_cuda_check(cudaFuncSetAttribute(select_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)ks), "topk select smem attribute");
        if (rc) return rc;
        select_kernel<true><<<1, kThreads, ks, st>>>(*res, P, k, ctx->topk_scratch);
    } else {
        select_kernel<false><<<1, kThreads, 0, st>>>(*res, P, k, ctx->topk_scratch);
    }
    const int64_t blocks = std::min<int64_t>((P + 255) / 256, (int64_t)ctx->sms * 8);
    compact_kernel<<<(unsigned)blocks, 256, 0, st>>>(*res, P, ctx->topk_scratch);
    final_kernel<<<1, kThreads, smem, st>>>(k, ctx->topk_scratch, ids, keys);
    return wf_cuda_check(cudaGetLastError(), "topk launch");
}
