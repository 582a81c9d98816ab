// Readiness forecast (Eq. 2) over the whole window, free of contention and of
// loading: one CTA sweeps the topological levels; the activations of a level
// are independent and processed in parallel.  The shortest feasible run time
// of every activation is found first (all activations in parallel); when the
// window fits, finish times then live in shared memory for the level sweep.
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

template <bool kShared>
__global__ void __launch_bounds__(kForecastThreads)
forecast_kernel(wf_dev_problem dp, int64_t *__restrict__ rel, int64_t *__restrict__ comp)
{
    extern __shared__ int64_t fs[];
    int64_t *c = kShared ? fs : comp;            // finish times read by later levels
    int64_t *lmin = kShared ? fs + dp.N : rel;   // rel[] doubles as scratch on the global path
    for (int32_t n = threadIdx.x; n < dp.N; n += blockDim.x) lmin[n] = fastest(dp, n);
    __syncthreads();
    for (int32_t l = 0; l < dp.nlev; ++l) {
        const int32_t lo = __ldg(dp.lev_off + l), hi = __ldg(dp.lev_off + l + 1);
        for (int32_t i = lo + (int32_t)threadIdx.x; i < hi; i += blockDim.x) {
            const int32_t n = __ldg(dp.lev_nodes + i);
            int64_t r = __ldg(dp.arrival + __ldg(dp.session + n));
            for (int32_t e = __ldg(dp.pred_off + n); e < __ldg(dp.pred_off + n + 1); ++e)
                r = max(r, c[__ldg(dp.pred_idx + e)]);
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
    if (ctx->dp.N <= kSharedMaxN) {
        const size_t smem = 16 * (size_t)ctx->dp.N;
        int rc = wf_cuda_check(cudaFuncSetAttribute(forecast_kernel<true>,
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                               "forecast smem attribute");
        if (rc) return rc;
        forecast_kernel<true><<<1, kForecastThreads, smem, st>>>(ctx->dp, rel, comp);
    } else {
        forecast_kernel<false><<<1, kForecastThreads, 0, st>>>(ctx->dp, rel, comp);
    }
    return wf_cuda_check(cudaGetLastError(), "forecast launch");
}
