// One step of the hot path from and to host memory (wf_eval_topk_host):
// host plan rows -> a device staging slot -> evaluation / top-k on the
// caller's stream (the forecast beside them) -> results back to the host.
//
// The context holds two staging slots and a copy stream.  A call takes the
// slot the previous call did not use, so its copy (on the copy stream) runs
// while the previous call evaluates (on the caller's stream); the copy first
// waits for the event recorded at the end of the call that last used the slot,
// and the evaluation waits for the event recorded after the copy.  The
// forecast (which depends on the window only) runs on the copy stream too,
// into the slot's own buffer.  The results and top-k buffers are single:
// everything that touches them runs in order on the caller's stream.
#include <cstdint>
#include <cstdlib>

#include "wf_internal.cuh"

struct wf_host_stage {
    int64_t P;                           // plans per slot (the context's max_P)
    int64_t place_stride, order_stride, bits_stride;  // bytes per staged row
    uint8_t *slot[2];                    // place | order | fuse | prefetch | retain rows
    int64_t *metrics;                    // makespan, p95, gpu: [3][P]
    uint32_t *status;                    // [P]
    int32_t *ids;                        // [1024]
    int64_t *keys;                       // [1024][3]
    int64_t *fc[2];                      // per slot: rel, comp [2][N]
    cudaStream_t copy;
    cudaEvent_t copied[2], freed[2];
    int next;
};

namespace {

int64_t round16(int64_t x) { return (x + 15) & ~(int64_t)15; }

int fail(int code, const char *what)
{
    return wf_set_error(code, "%s", what);
}

// The five row arrays of slot s for P plans.
wf_plans slot_plans(const wf_host_stage *h, int s, int64_t P, int64_t plan_base, bool retain)
{
    uint8_t *b = h->slot[s];
    wf_plans d;
    d.P = P;
    d.plan_base = plan_base;
    d.place_stride = h->place_stride;
    d.order_stride = h->order_stride;
    d.bits_stride = h->bits_stride;
    d.place = b;
    b += h->place_stride * h->P;
    d.order = (const uint16_t *)b;
    b += h->order_stride * h->P;
    d.fuse = (const uint32_t *)b;
    b += h->bits_stride * h->P;
    d.prefetch = (const uint32_t *)b;
    b += h->bits_stride * h->P;
    d.retain = retain ? (const uint32_t *)b : nullptr;
    return d;
}

int reserve(wf_ctx *c)
{
    if (c->host) return WF_OK;
    wf_host_stage *h = (wf_host_stage *)calloc(1, sizeof(wf_host_stage));
    if (!h) return fail(WF_ENOMEM, "host allocation of the staging record");
    const int64_t N = c->dp.N, P = c->max_P;
    h->P = P;
    h->place_stride = round16(N);
    h->order_stride = round16(2 * N);
    h->bits_stride = round16(4 * ((N + 31) / 32));
    const size_t slot_bytes = (size_t)P * (size_t)(h->place_stride + h->order_stride + 3 * h->bits_stride);
    c->host = h;  // wf_host_release frees whatever was made below
    int rc = WF_OK;
    for (int s = 0; s < 2 && !rc; ++s)
        rc = wf_cuda_check(cudaMalloc(&h->slot[s], slot_bytes), "cudaMalloc(host staging slot)");
    if (!rc) rc = wf_cuda_check(cudaMalloc(&h->metrics, sizeof(int64_t) * 3 * (size_t)P), "cudaMalloc(host results)");
    if (!rc) rc = wf_cuda_check(cudaMalloc(&h->status, sizeof(uint32_t) * (size_t)P), "cudaMalloc(host status)");
    if (!rc) rc = wf_cuda_check(cudaMalloc(&h->ids, sizeof(int32_t) * 1024), "cudaMalloc(host top-k)");
    if (!rc) rc = wf_cuda_check(cudaMalloc(&h->keys, sizeof(int64_t) * 3 * 1024), "cudaMalloc(host top-k keys)");
    for (int s = 0; s < 2 && !rc; ++s)
        rc = wf_cuda_check(cudaMalloc(&h->fc[s], sizeof(int64_t) * 2 * (size_t)N), "cudaMalloc(host forecast)");
    if (!rc) rc = wf_cuda_check(cudaStreamCreateWithFlags(&h->copy, cudaStreamNonBlocking), "cudaStreamCreate");
    for (int s = 0; s < 2 && !rc; ++s) {
        rc = wf_cuda_check(cudaEventCreateWithFlags(&h->copied[s], cudaEventDisableTiming), "cudaEventCreate");
        if (!rc) rc = wf_cuda_check(cudaEventCreateWithFlags(&h->freed[s], cudaEventDisableTiming), "cudaEventCreate");
    }
    if (rc) {
        wf_host_release(c);
        return rc;
    }
    return WF_OK;
}

// Row copies of one host array into the slot: width bytes of each of P rows.
// Rows laid out with the slot's own stride go as one flat copy (a pitched
// copy of short rows moves far slower); others row by row.
int copy_rows(void *dst, int64_t dpitch, const void *src, int64_t spitch, int64_t width, int64_t P,
              cudaStream_t st)
{
    if (spitch == dpitch && width == dpitch)
        return wf_cuda_check(cudaMemcpyAsync(dst, src, (size_t)(dpitch * P), cudaMemcpyHostToDevice, st),
                             "plan rows host to device");
    return wf_cuda_check(cudaMemcpy2DAsync(dst, (size_t)dpitch, src, (size_t)spitch, (size_t)width, (size_t)P,
                                           cudaMemcpyHostToDevice, st),
                         "plan rows host to device");
}

}  // namespace

void wf_host_release(wf_ctx *c)
{
    wf_host_stage *h = c->host;
    if (!h) return;
    if (h->copy) cudaStreamSynchronize(h->copy);
    for (int s = 0; s < 2; ++s) {
        if (h->slot[s]) cudaFree(h->slot[s]);
        if (h->copied[s]) cudaEventDestroy(h->copied[s]);
        if (h->freed[s]) cudaEventDestroy(h->freed[s]);
        if (h->fc[s]) cudaFree(h->fc[s]);
    }
    if (h->metrics) cudaFree(h->metrics);
    if (h->status) cudaFree(h->status);
    if (h->ids) cudaFree(h->ids);
    if (h->keys) cudaFree(h->keys);
    if (h->copy) cudaStreamDestroy(h->copy);
    free(h);
    c->host = nullptr;
}

extern "C" int wf_ctx_reserve_host(wf_ctx *c)
{
    if (!c) return fail(WF_EINVAL, "NULL context");
    int rc = wf_select_device(c);
    return rc ? rc : reserve(c);
}

extern "C" int wf_eval_topk_host(wf_ctx *c, const wf_plans *hp, int32_t k, int32_t *ids_host, int64_t *keys_host,
                                 const wf_eval_out *out_host, int64_t *rel_host, int64_t *comp_host, void *stream)
{
    if (!c || !hp || !ids_host) return fail(WF_EINVAL, "NULL argument");
    const int64_t N = c->dp.N, P = hp->P;
    if (P < 1 || P > c->max_P) return fail(WF_EINVAL, "host plans: P outside 1..max_P");
    if (k < 1 || k > 1024 || k > P) return fail(WF_EINVAL, "k outside 1..min(P, 1024)");
    if (!hp->place || !hp->order || !hp->fuse || !hp->prefetch) return fail(WF_EINVAL, "host plans: NULL plan array");
    if (hp->plan_base < 0) return fail(WF_EINVAL, "host plans: plan_base < 0");
    if (out_host) {
        const int bad = wf_check_out(out_host, "host results");
        if (bad) return bad;
    }
    if (!rel_host != !comp_host) return fail(WF_EINVAL, "rel_host and comp_host: both or neither");
    int rc = wf_select_device(c);
    if (!rc) rc = reserve(c);
    if (rc) return rc;
    wf_host_stage *h = c->host;
    if (hp->place_stride < h->place_stride || hp->place_stride % 16 || hp->order_stride < h->order_stride ||
        hp->order_stride % 16 || hp->bits_stride < h->bits_stride || hp->bits_stride % 16)
        return fail(WF_EINVAL, "host plans: a stride below its row size or not a multiple of 16 bytes");

    const cudaStream_t st = (cudaStream_t)stream;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    rc = wf_cuda_check(cudaStreamIsCapturing(st, &cs), "stream capture status");
    if (rc) return rc;
    // Under capture the copies go on the caller's stream (no events from
    // outside the capture are waited for).
    const bool capturing = cs != cudaStreamCaptureStatusNone;
    const int s = h->next;
    h->next ^= 1;
    const wf_plans d = slot_plans(h, s, P, hp->plan_base, hp->retain != nullptr);
    const cudaStream_t cp = capturing ? st : h->copy;
    if (!capturing) rc = wf_cuda_check(cudaStreamWaitEvent(cp, h->freed[s], 0), "wait for the slot");
    // The forecast depends on the window only: it runs on the copy stream
    // too, before the copies, beside the previous call's evaluation.
    if (!rc && rel_host) rc = wf_launch_forecast(c, h->fc[s], h->fc[s] + N, cp);
    if (!rc) rc = copy_rows((void *)d.place, d.place_stride, hp->place, hp->place_stride, d.place_stride, P, cp);
    if (!rc) rc = copy_rows((void *)d.order, d.order_stride, hp->order, hp->order_stride, d.order_stride, P, cp);
    if (!rc) rc = copy_rows((void *)d.fuse, d.bits_stride, hp->fuse, hp->bits_stride, d.bits_stride, P, cp);
    if (!rc) rc = copy_rows((void *)d.prefetch, d.bits_stride, hp->prefetch, hp->bits_stride, d.bits_stride, P, cp);
    if (!rc && hp->retain)
        rc = copy_rows((void *)d.retain, d.bits_stride, hp->retain, hp->bits_stride, d.bits_stride, P, cp);
    if (!rc && !capturing) {
        rc = wf_cuda_check(cudaEventRecord(h->copied[s], cp), "record the copy");
        if (!rc) rc = wf_cuda_check(cudaStreamWaitEvent(st, h->copied[s], 0), "wait for the copy");
    }
    if (rc) return rc;

    wf_eval_out dout;
    dout.makespan_us = h->metrics;
    dout.p95_us = h->metrics + P;
    dout.gpu_us = h->metrics + 2 * P;
    dout.status = h->status;
    if (!rc) rc = wf_launch_eval(c, &d, &dout, st);
    if (!rc) rc = wf_launch_topk(c, &dout, P, k, h->ids, h->keys, st);
    if (rc) return rc;

    const cudaMemcpyKind dh = cudaMemcpyDeviceToHost;
    rc = wf_cuda_check(cudaMemcpyAsync(ids_host, h->ids, sizeof(int32_t) * (size_t)k, dh, st), "top-k to host");
    if (!rc && keys_host)
        rc = wf_cuda_check(cudaMemcpyAsync(keys_host, h->keys, sizeof(int64_t) * 3 * (size_t)k, dh, st),
                           "top-k keys to host");
    if (!rc && out_host) {
        const size_t b = sizeof(int64_t) * (size_t)P;
        rc = wf_cuda_check(cudaMemcpyAsync(out_host->makespan_us, dout.makespan_us, b, dh, st), "results to host");
        if (!rc) rc = wf_cuda_check(cudaMemcpyAsync(out_host->p95_us, dout.p95_us, b, dh, st), "results to host");
        if (!rc) rc = wf_cuda_check(cudaMemcpyAsync(out_host->gpu_us, dout.gpu_us, b, dh, st), "results to host");
        if (!rc)
            rc = wf_cuda_check(cudaMemcpyAsync(out_host->status, dout.status, sizeof(uint32_t) * (size_t)P, dh, st),
                               "status to host");
    }
    if (!rc && rel_host) {
        const size_t b = sizeof(int64_t) * (size_t)N;
        rc = wf_cuda_check(cudaMemcpyAsync(rel_host, h->fc[s], b, dh, st), "forecast to host");
        if (!rc) rc = wf_cuda_check(cudaMemcpyAsync(comp_host, h->fc[s] + N, b, dh, st), "forecast to host");
    }
    // The slot (its rows and its forecast) may be refilled once this call's
    // evaluation and copies back have run.
    if (!rc && !capturing) rc = wf_cuda_check(cudaEventRecord(h->freed[s], st), "record the slot's release");
    return rc;
}
