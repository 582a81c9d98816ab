// Readiness forecast (Eq. 2) over the whole window, free of contention and of
// loading: one CTA sweeps the topological levels; the activations of a level
// are independent and processed in parallel.  The shortest feasible run time
// of every activation is found first (all activations in parallel); when the
// window fits, finish times then live in shared memory for the level sweep,
// and when the predecessor lists, arrivals and level order fit too, they are
// staged there as well.
#include "wf_internal.cuh"

namespace {

constexpr int kForecastThreads = 1024;
constexpr int32_t kSharedMaxN = 12288;  // 2 x 8 B per activation in shared memory

// Fastest device whose capacity admits the activation's peak (Eq. 8).
__device__ __forceinline__ int64_t fastest(const wf_dev_problem &dp, int32_t n)
{
    int64_t lmin = WF_INF64;
    const int32_t *lat = dp.lat + (int64_t)n * dp.D;
    const int32_t *pk = dp.peak + (int64_t)n * dp.D;
    for (int32_t d = 0; d < dp.D; ++d)
        if (__ldg(pk + d) <= __ldg(dp.cap + d)) lmin = min(lmin, (int64_t)__ldg(lat + d));
    return lmin;
}

// Shared-memory layout of the staged sweep: finish times, fastest run times
// and session arrivals (8 B each per activation), the predecessor CSR, the
// level order and the level offsets (4 B entries).
__host__ __device__ inline size_t staged_bytes(int32_t N, int32_t E, int32_t nlev)
{
    return 24 * (size_t)N + 4 * ((size_t)N + 1) + 4 * (size_t)E + 4 * (size_t)N + 4 * ((size_t)nlev + 1);
}

template <bool kShared, bool kStaged>
__global__ void __launch_bounds__(kForecastThreads)
forecast_kernel(wf_dev_problem dp, int64_t *__restrict__ rel, int64_t *__restrict__ comp)
{
    extern __shared__ int64_t fs[];
    const int32_t N = dp.N, E = dp.E;
    int64_t *c = kShared ? fs : comp;            // finish times read by later levels
    int64_t *lmin = kShared ? fs + N : rel;      // rel[] doubles as scratch on the global path
    // Staged: every table the level sweep reads is copied to shared memory
    // first (all activations at once), so each level costs shared-memory
    // latencies only.
    int64_t *arr_s = fs + 2 * N;
    int32_t *poff_s = (int32_t *)(fs + 3 * N);
    int32_t *pidx_s = poff_s + N + 1;
    int32_t *lev_s = pidx_s + E;
    int32_t *loff_s = lev_s + N;
    for (int32_t n = threadIdx.x; n < N; n += blockDim.x) {
        lmin[n] = fastest(dp, n);
        if (kStaged) {
            arr_s[n] = __ldg(dp.arrival + __ldg(dp.session + n));
            poff_s[n] = __ldg(dp.pred_off + n);
            lev_s[n] = __ldg(dp.lev_nodes + n);
        }
    }
    if (kStaged) {
        if (threadIdx.x == 0) poff_s[N] = __ldg(dp.pred_off + N);
        for (int32_t e = threadIdx.x; e < E; e += blockDim.x) pidx_s[e] = __ldg(dp.pred_idx + e);
        for (int32_t l = threadIdx.x; l <= dp.nlev; l += blockDim.x) loff_s[l] = __ldg(dp.lev_off + l);
    }
    __syncthreads();
    for (int32_t l = 0; l < dp.nlev; ++l) {
        const int32_t lo = kStaged ? loff_s[l] : __ldg(dp.lev_off + l);
        const int32_t hi = kStaged ? loff_s[l + 1] : __ldg(dp.lev_off + l + 1);
        for (int32_t i = lo + (int32_t)threadIdx.x; i < hi; i += blockDim.x) {
            const int32_t n = kStaged ? lev_s[i] : __ldg(dp.lev_nodes + i);
            int64_t r = kStaged ? arr_s[n] : __ldg(dp.arrival + __ldg(dp.session + n));
            const int32_t e0 = kStaged ? poff_s[n] : __ldg(dp.pred_off + n);
            const int32_t e1 = kStaged ? poff_s[n + 1] : __ldg(dp.pred_off + n + 1);
            for (int32_t e = e0; e < e1; ++e) r = max(r, c[kStaged ? pidx_s[e] : __ldg(dp.pred_idx + e)]);
            const int64_t f = r + lmin[n];
            c[n] = f;
            if (kShared) { rel[n] = r; comp[n] = f; }
            else rel[n] = r;  // the node's own lmin slot is no longer needed
        }
        __syncthreads();  // level l's finish times are read by level l + 1
    }
}

}  // namespace

int wf_launch_forecast(wf_ctx *ctx, int64_t *rel, int64_t *comp, cudaStream_t st)
{
    const wf_dev_problem &dp = ctx->dp;
    const size_t staged = staged_bytes(dp.N, dp.E, dp.nlev);
    if (staged <= 227 * 1024) {
        int rc = wf_cuda_check(cudaFuncSetAttribute(forecast_kernel<true, true>,
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)staged),
                               "forecast smem attribute");
        if (rc) return rc;
        forecast_kernel<true, true><<<1, kForecastThreads, staged, st>>>(dp, rel, comp);
    } else if (dp.N <= kSharedMaxN) {
        const size_t smem = 16 * (size_t)dp.N;
        int rc = wf_cuda_check(cudaFuncSetAttribute(forecast_kernel<true, false>,
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                               "forecast smem attribute");
        if (rc) return rc;
        forecast_kernel<true, false><<<1, kForecastThreads, smem, st>>>(dp, rel, comp);
    } else {
        forecast_kernel<false, false><<<1, kForecastThreads, 0, st>>>(dp, rel, comp);
    }
    return wf_cuda_check(cudaGetLastError(), "forecast launch");
}
