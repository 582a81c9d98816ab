// Top-k of evaluated plans (row a12) by the key (status != 0, makespan, p95,
// gpu, plan index): each CTA sorts a tile of candidates in shared memory
// (bitonic network) and keeps its k best; passes repeat until one tile holds
// every survivor.
#include <algorithm>

#include "wf_internal.cuh"

namespace {

constexpr int kTile = 2048;          // candidates per CTA
constexpr int kTopkThreads = 1024;   // two candidates per thread

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

__device__ void bitonic_sort(Cand *s)
{
    for (int size = 2; size <= kTile; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncthreads();
            for (int t = threadIdx.x; t < kTile / 2; t += blockDim.x) {
                const int i = 2 * stride * (t / stride) + (t % stride);
                const int j = i + stride;
                const bool up = (i & size) == 0;
                Cand a = s[i], b = s[j];
                if (before(b, a) == up) { s[i] = b; s[j] = a; }
            }
        }
    }
    __syncthreads();
}

// First pass: candidates straight from the result arrays.
__global__ void __launch_bounds__(kTopkThreads)
topk_from_results(wf_eval_out res, int64_t P, int32_t k, Cand *dst)
{
    extern __shared__ Cand s[];
    const int64_t base = (int64_t)blockIdx.x * kTile;
    for (int t = threadIdx.x; t < kTile; t += blockDim.x) {
        const int64_t p = base + t;
        Cand c = padding();
        if (p < P) {
            c.mk = res.makespan_us[p];
            c.p95 = res.p95_us[p];
            c.gpu = res.gpu_us[p];
            c.id = (int32_t)p;
            c.bad = res.status[p] != 0 ? 1u : 0u;
        }
        s[t] = c;
    }
    bitonic_sort(s);
    for (int t = threadIdx.x; t < k; t += blockDim.x) dst[(int64_t)blockIdx.x * k + t] = s[t];
}

// Later passes: candidates from the previous pass.
__global__ void __launch_bounds__(kTopkThreads)
topk_from_cands(const Cand *src, int64_t n, int32_t k, Cand *dst, int32_t *ids, int64_t *keys)
{
    extern __shared__ Cand s[];
    const int64_t base = (int64_t)blockIdx.x * kTile;
    for (int t = threadIdx.x; t < kTile; t += blockDim.x)
        s[t] = base + t < n ? src[base + t] : padding();
    bitonic_sort(s);
    if (ids) {  // final pass: one CTA
        for (int t = threadIdx.x; t < k; t += blockDim.x) {
            ids[t] = s[t].id;
            if (keys) {
                keys[3 * t] = s[t].mk;
                keys[3 * t + 1] = s[t].p95;
                keys[3 * t + 2] = s[t].gpu;
            }
        }
    } else {
        for (int t = threadIdx.x; t < k; t += blockDim.x) dst[(int64_t)blockIdx.x * k + t] = s[t];
    }
}

}  // namespace

size_t wf_topk_scratch_bytes(int64_t max_P)
{
    const int64_t tiles = (max_P + kTile - 1) / kTile + 1;
    return 2 * (size_t)tiles * 1024 * sizeof(Cand);
}

int wf_launch_topk(wf_ctx *ctx, const wf_eval_out *res, int64_t P, int32_t k, int32_t *ids,
                   int64_t *keys, cudaStream_t st)
{
    const size_t smem = kTile * sizeof(Cand);
    static bool attr_set = false;
    if (!attr_set) {
        int rc = wf_cuda_check(cudaFuncSetAttribute(topk_from_results,
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                               "topk smem attribute");
        if (!rc) rc = wf_cuda_check(cudaFuncSetAttribute(topk_from_cands,
                                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                                    "topk smem attribute");
        if (rc) return rc;
        attr_set = true;
    }
    Cand *buf[2];
    const int64_t half = (int64_t)(ctx->topk_scratch_bytes / 2 / sizeof(Cand));
    buf[0] = (Cand *)ctx->topk_scratch;
    buf[1] = buf[0] + half;
    int64_t tiles = (P + kTile - 1) / kTile;
    if (tiles == 1) {
        // One tile: sort the results directly into the output.
        topk_from_results<<<1, kTopkThreads, smem, st>>>(*res, P, k, buf[0]);
        topk_from_cands<<<1, kTopkThreads, smem, st>>>(buf[0], k, k, nullptr, ids, keys);
        return wf_cuda_check(cudaGetLastError(), "topk launch");
    }
    topk_from_results<<<(unsigned)tiles, kTopkThreads, smem, st>>>(*res, P, k, buf[0]);
    int64_t n = tiles * k;
    int cur = 0;
    while (n > kTile) {
        tiles = (n + kTile - 1) / kTile;
        topk_from_cands<<<(unsigned)tiles, kTopkThreads, smem, st>>>(buf[cur], n, k, buf[cur ^ 1],
                                                                      nullptr, nullptr);
        cur ^= 1;
        n = tiles * k;
    }
    topk_from_cands<<<1, kTopkThreads, smem, st>>>(buf[cur], n, k, nullptr, ids, keys);
    return wf_cuda_check(cudaGetLastError(), "topk launch");
}
