// Readiness forecast (Eq. 2) over the whole window, free of contention and of
// loading: one CTA sweeps the topological levels; the activations of a level
// are independent and processed in parallel.
#include "wf_internal.cuh"

namespace {

constexpr int kForecastThreads = 1024;

__global__ void __launch_bounds__(kForecastThreads)
forecast_kernel(wf_dev_problem dp, int64_t *__restrict__ rel, int64_t *__restrict__ comp)
{
    for (int32_t l = 0; l < dp.nlev; ++l) {
        const int32_t lo = dp.lev_off[l], hi = dp.lev_off[l + 1];
        for (int32_t i = lo + (int32_t)threadIdx.x; i < hi; i += blockDim.x) {
            const int32_t n = dp.lev_nodes[i];
            int64_t r = dp.arrival[dp.session[n]];
            for (int32_t e = dp.pred_off[n]; e < dp.pred_off[n + 1]; ++e)
                r = max(r, comp[dp.pred_idx[e]]);
            // Fastest device whose capacity admits the activation's peak (Eq. 8).
            int64_t lmin = WF_INF64;
            const int32_t *lat = dp.lat + (int64_t)n * dp.D;
            const int32_t *pk = dp.peak + (int64_t)n * dp.D;
            for (int32_t d = 0; d < dp.D; ++d)
                if (pk[d] <= dp.cap[d]) lmin = min(lmin, (int64_t)lat[d]);
            rel[n] = r;
            comp[n] = r + lmin;
        }
        __syncthreads();  // level l's comp[] is read by level l+1
    }
}

}  // namespace

int wf_launch_forecast(wf_ctx *ctx, int64_t *rel, int64_t *comp, cudaStream_t st)
{
    forecast_kernel<<<1, kForecastThreads, 0, st>>>(ctx->dp, rel, comp);
    return wf_cuda_check(cudaGetLastError(), "forecast launch");
}
