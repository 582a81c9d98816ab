// Context build (host side of the library): validation of a problem,
// derivation of the fusible edges (Eq. 3) and of topological levels, and the
// upload of every table to the device.  Also the C-ABI entry points, which
// check their arguments and hand over to the kernel launchers.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <vector>

#include "wf_internal.cuh"

static thread_local char g_last_error[512];

int wf_set_error(int code, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
    return code;
}

int wf_cuda_check(cudaError_t e, const char *what)
{
    if (e == cudaSuccess) return WF_OK;
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return wf_set_error(WF_ENOMEM, "%s: %s", what, cudaGetErrorString(e));
    }
    return wf_set_error(WF_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

extern "C" const char *wf_last_error(void) { return g_last_error; }

extern "C" const char *wf_strerror(int code)
{
    switch (code) {
    case WF_OK: return "ok";
    case WF_EINVAL: return "invalid argument";
    case WF_ENOMEM: return "out of memory";
    case WF_ECUDA: return "CUDA error";
    case WF_ETIMEOUT: return "device wait timed out";
    default: return "unknown error";
    }
}

#define REQUIRE(cond, ...) \
    do { if (!(cond)) return wf_set_error(WF_EINVAL, __VA_ARGS__); } while (0)

static bool is_pow2(int32_t x) { return x > 0 && (x & (x - 1)) == 0; }

// Derived host-side tables.
struct wf_derived {
    std::vector<int32_t> fnext, fprev, lev_off, lev_nodes;
};

// Checks every precondition of a problem; on success fills the derived tables.
static int validate(const wf_problem *pb, wf_derived *dv)
{
    REQUIRE(pb != nullptr, "problem is NULL");
    const int32_t N = pb->N, D = pb->D, M = pb->M, W = pb->W;
    REQUIRE(N >= 1 && N <= 65535, "N=%d outside 1..65535", N);
    REQUIRE(D >= 1 && D <= 32, "D=%d outside 1..32", D);
    REQUIRE(M >= 1 && M <= 16, "M=%d outside 1..16", M);
    REQUIRE(W >= 1, "W=%d < 1", W);
    REQUIRE(pb->pred_off && pb->model && pb->session && pb->arrival_us && pb->lat_us &&
                pb->peak_mib && pb->weight_mib && pb->load_us && pb->cap_mib,
            "a problem table pointer is NULL");
    REQUIRE(pb->pred_off[0] == 0, "pred_off[0] != 0");
    for (int32_t v = 0; v < N; ++v)
        REQUIRE(pb->pred_off[v + 1] >= pb->pred_off[v], "pred_off not monotone at %d", v);
    const int32_t E = pb->pred_off[N];
    REQUIRE(E == 0 || pb->pred_idx, "pred_idx is NULL with E=%d", E);
    REQUIRE(pb->grant_us >= 0, "grant_us < 0");
    REQUIRE(pb->margin_mib >= 0, "margin_mib < 0");
    for (int32_t m = 0; m < M; ++m) REQUIRE(pb->weight_mib[m] >= 1, "weight_mib[%d] < 1", m);
    for (int32_t d = 0; d < D; ++d) REQUIRE(pb->cap_mib[d] >= 1, "cap_mib[%d] < 1", d);
    for (int64_t i = 0; i < (int64_t)M * D; ++i) REQUIRE(pb->load_us[i] >= 0, "load_us < 0");
    for (int32_t w = 0; w < W; ++w) REQUIRE(pb->arrival_us[w] >= 0, "arrival_us[%d] < 0", w);

    std::vector<int32_t> per_session(W, 0), nsucc(N, 0), only(N, -1), mark(N, -1);
    for (int32_t v = 0; v < N; ++v) {
        REQUIRE(pb->model[v] < M, "model[%d] >= M", v);
        REQUIRE(pb->session[v] >= 0 && pb->session[v] < W, "session[%d] out of range", v);
        per_session[pb->session[v]] += 1;
        bool fits = false;
        for (int32_t d = 0; d < D; ++d) {
            int64_t i = (int64_t)v * D + d;
            REQUIRE(pb->lat_us[i] >= 0, "lat_us[%d][%d] < 0", v, d);
            REQUIRE(pb->peak_mib[i] >= pb->weight_mib[pb->model[v]],
                    "peak_mib[%d][%d] below the model weight", v, d);
            REQUIRE((int64_t)pb->peak_mib[i] + pb->margin_mib <= INT32_MAX, "peak_mib + margin_mib overflows");
            fits |= (int64_t)pb->peak_mib[i] + pb->margin_mib <= pb->cap_mib[d];
        }
        REQUIRE(fits, "activation %d fits on no device", v);
        for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) {
            int32_t u = pb->pred_idx[e];
            REQUIRE(u >= 0 && u < N, "pred_idx out of range at edge %d", e);
            REQUIRE(u != v, "self-loop at %d", v);
            REQUIRE(mark[u] != v, "duplicate edge %d -> %d", u, v);
            mark[u] = v;
            REQUIRE(pb->session[u] == pb->session[v], "edge %d -> %d crosses sessions", u, v);
            nsucc[u] += 1;
            only[u] = v;
        }
    }
    for (int32_t w = 0; w < W; ++w) REQUIRE(per_session[w] > 0, "session %d has no activation", w);

    if (pb->S != 0) {
        REQUIRE(pb->S > 0, "S < 0");
        REQUIRE(pb->bm_r && pb->bm_c && pb->bm_e, "stochastic tables are NULL");
        REQUIRE(is_pow2(pb->bm_rn) && is_pow2(pb->bm_cn), "bm_rn / bm_cn not powers of two");
        REQUIRE(pb->bm_en >= 1 && (pb->bm_en & 1), "bm_en must be odd");
        int64_t rmax = 0, cmax = 0;
        for (int32_t i = 0; i < pb->bm_rn; ++i) rmax = std::max<int64_t>(rmax, std::llabs(pb->bm_r[i]));
        for (int32_t i = 0; i < pb->bm_cn; ++i) cmax = std::max<int64_t>(cmax, std::llabs(pb->bm_c[i]));
        for (int32_t i = 0; i < pb->bm_en; ++i) REQUIRE(pb->bm_e[i] >= 0, "bm_e[%d] < 0", i);
        const int64_t zmax = (rmax * cmax + (1 << 18) - 1) >> 18;
        REQUIRE(zmax <= (pb->bm_en - 1) / 2, "bm_e too short for the largest |zq|=%lld",
                (long long)zmax);
    }

    // Topological levels (Kahn by levels) -> acyclicity.
    std::vector<int32_t> soff(N + 1, 0), sidx(E > 0 ? E : 1), fill(N), indeg(N);
    for (int32_t u = 0; u < N; ++u) soff[u + 1] = soff[u] + nsucc[u];
    for (int32_t u = 0; u < N; ++u) fill[u] = soff[u];
    for (int32_t v = 0; v < N; ++v) {
        indeg[v] = pb->pred_off[v + 1] - pb->pred_off[v];
        for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) sidx[fill[pb->pred_idx[e]]++] = v;
    }
    std::vector<int32_t> cur, nxt;
    for (int32_t v = 0; v < N; ++v) if (indeg[v] == 0) cur.push_back(v);
    dv->lev_off.assign(1, 0);
    dv->lev_nodes.clear();
    while (!cur.empty()) {
        nxt.clear();
        for (int32_t u : cur) {
            dv->lev_nodes.push_back(u);
            for (int32_t e = soff[u]; e < soff[u + 1]; ++e)
                if (--indeg[sidx[e]] == 0) nxt.push_back(sidx[e]);
        }
        dv->lev_off.push_back((int32_t)dv->lev_nodes.size());
        cur.swap(nxt);
    }
    REQUIRE((int32_t)dv->lev_nodes.size() == N, "the DAG has a cycle");

    // Eq. 3: (u, v) fusible iff succ(u) = {v}, pred(v) = {u}, same model.
    dv->fnext.assign(N, -1);
    dv->fprev.assign(N, -1);
    for (int32_t u = 0; u < N; ++u) {
        if (nsucc[u] != 1) continue;
        int32_t v = only[u];
        if (pb->pred_off[v + 1] - pb->pred_off[v] == 1 && pb->model[u] == pb->model[v]) {
            dv->fnext[u] = v;
            dv->fprev[v] = u;
        }
    }
    return WF_OK;
}

extern "C" int wf_problem_check(const wf_problem *prob)
{
    wf_derived dv;
    return validate(prob, &dv);
}

// Appends a host array to the staging image at a 256-byte aligned offset.
struct Image {
    std::vector<uint8_t> bytes;
    size_t add(const void *src, size_t n)
    {
        size_t off = (bytes.size() + 255) & ~(size_t)255;
        bytes.resize(off + (n > 0 ? n : 1), 0);
        if (n && src) memcpy(bytes.data() + off, src, n);
        return off;
    }
};

extern "C" int wf_ctx_create(const wf_problem *pb, int device, int64_t max_P, wf_ctx **out)
{
    if (!out) return wf_set_error(WF_EINVAL, "out is NULL");
    *out = nullptr;
    REQUIRE(max_P >= 1, "max_P < 1");
    wf_derived dv;
    int rc = validate(pb, &dv);
    if (rc) return rc;
    int ndev = 0;
    rc = wf_cuda_check(cudaGetDeviceCount(&ndev), "cudaGetDeviceCount");
    if (rc) return rc;
    REQUIRE(device >= 0 && device < ndev, "device %d not present", device);
    rc = wf_cuda_check(cudaSetDevice(device), "cudaSetDevice");
    if (rc) return rc;

    const int32_t N = pb->N, D = pb->D, M = pb->M, W = pb->W, E = pb->pred_off[N];
    Image img;
    size_t o_poff = img.add(pb->pred_off, sizeof(int32_t) * (N + 1));
    size_t o_pidx = img.add(pb->pred_idx, sizeof(int32_t) * E);
    size_t o_fnext = img.add(dv.fnext.data(), sizeof(int32_t) * N);
    size_t o_fprev = img.add(dv.fprev.data(), sizeof(int32_t) * N);
    size_t o_model = img.add(pb->model, N);
    size_t o_sess = img.add(pb->session, sizeof(int32_t) * N);
    size_t o_arr = img.add(pb->arrival_us, sizeof(int64_t) * W);
    size_t o_lat = img.add(pb->lat_us, sizeof(int32_t) * (size_t)N * D);
    // Admission memory (Section 3.3): predicted peak + margin, used wherever a
    // capacity is checked.
    std::vector<int32_t> adm((size_t)N * D);
    for (size_t i = 0; i < adm.size(); ++i) adm[i] = pb->peak_mib[i] + pb->margin_mib;
    size_t o_peak = img.add(adm.data(), sizeof(int32_t) * (size_t)N * D);
    size_t o_w = img.add(pb->weight_mib, sizeof(int32_t) * M);
    size_t o_load = img.add(pb->load_us, sizeof(int32_t) * (size_t)M * D);
    size_t o_cap = img.add(pb->cap_mib, sizeof(int32_t) * D);
    size_t o_loff = img.add(dv.lev_off.data(), sizeof(int32_t) * dv.lev_off.size());
    size_t o_lnodes = img.add(dv.lev_nodes.data(), sizeof(int32_t) * N);
    const bool stoch = pb->S > 0;
    size_t o_br = img.add(stoch ? pb->bm_r : nullptr, stoch ? sizeof(int32_t) * pb->bm_rn : 0);
    size_t o_bc = img.add(stoch ? pb->bm_c : nullptr, stoch ? sizeof(int32_t) * pb->bm_cn : 0);
    size_t o_be = img.add(stoch ? pb->bm_e : nullptr, stoch ? sizeof(int32_t) * pb->bm_en : 0);
    // The radius and angle tables again as int16 when every value fits: half
    // the L1 footprint for the stochastic sweep's per-sample lookups.
    std::vector<int16_t> br16, bc16;
    bool t16 = stoch;
    for (int32_t i = 0; t16 && i < pb->bm_rn; ++i) t16 = pb->bm_r[i] >= -32768 && pb->bm_r[i] <= 32767;
    for (int32_t i = 0; t16 && i < pb->bm_cn; ++i) t16 = pb->bm_c[i] >= -32768 && pb->bm_c[i] <= 32767;
    if (t16) {
        br16.assign(pb->bm_r, pb->bm_r + pb->bm_rn);
        bc16.assign(pb->bm_c, pb->bm_c + pb->bm_cn);
    }
    size_t o_br16 = img.add(t16 ? br16.data() : nullptr, t16 ? sizeof(int16_t) * br16.size() : 0);
    size_t o_bc16 = img.add(t16 ? bc16.data() : nullptr, t16 ? sizeof(int16_t) * bc16.size() : 0);
    size_t o_err = img.add(nullptr, 256);
    // Slot tables of the shared-memory sweep.
    std::vector<int32_t> rslot(N), wl_off;
    std::vector<uint16_t> wl;
    const int32_t nslots = wf_assign_slots(N, W, pb->pred_off, pb->pred_idx, pb->session, dv.fprev.data(),
                                           dv.fnext.data(), rslot.data(), wl_off, wl);
    std::vector<int4> noderec(2 * (size_t)N);
    std::vector<int2> lk((size_t)N * D);
    for (int32_t n = 0; n < N; ++n) {
        noderec[2 * n] = make_int4(dv.fprev[n], dv.fnext[n], rslot[n], (int32_t)pb->model[n] | (pb->session[n] << 8));
        // Write list of n as a unit's last member: start, length, first two codes inline.
        const int32_t a = wl_off[n], len = wl_off[n + 1] - wl_off[n];
        const uint32_t c0 = len > 0 ? wl[a] : 0u, c1 = len > 1 ? wl[a + 1] : 0u;
        noderec[2 * n + 1] = make_int4(a, len, (int32_t)(c0 | (c1 << 16)), 0);
        for (int32_t d = 0; d < D; ++d) {
            const int64_t i = (int64_t)n * D + d;
            // KV admission, or -1 where the activation does not fit the device
            // (Eq. 8): the sweep's producers read the pair for every unit anyway.
            lk[i] = make_int2(pb->lat_us[i],
                              adm[i] <= pb->cap_mib[d] ? adm[i] - pb->weight_mib[pb->model[n]] : -1);
        }
    }
    size_t o_rec = img.add(noderec.data(), sizeof(int4) * noderec.size());
    std::vector<uint32_t> links(N);
    for (int32_t n = 0; n < N; ++n)
        links[n] = ((uint32_t)dv.fprev[n] & 0xFFFFu) | ((uint32_t)dv.fnext[n] << 16);  // -1 -> 0xFFFF
    size_t o_links = img.add(links.data(), sizeof(uint32_t) * N);
    // Per-node record of the sweep's producers: links; release slot code
    // (slot | accumulator << 15; the zero slot nslots + 1 without
    // predecessors) | model << 16 | write-list length (max 7) << 20; session
    // arrival (u32: the sweep runs only with arrivals below 2^32); the first
    // two write codes, the sink slot nslots standing in for absent ones.
    std::vector<uint4> hrec(N);
    std::vector<uint32_t> wc23(N, 0);
    if (nslots > 0) {
        const uint32_t trash = (uint32_t)nslots, zero = trash + 1;
        for (int32_t n = 0; n < N; ++n) {
            const uint32_t rs = rslot[n] < 0 ? zero
                                             : (((uint32_t)rslot[n] & 0x7FFFu) | ((rslot[n] & WF_RSLOT_ACC) ? 0x8000u : 0u));
            const int32_t a = wl_off[n], len = wl_off[n + 1] - wl_off[n];
            const uint32_t c0 = len > 0 ? wl[a] : trash, c1 = len > 1 ? wl[a + 1] : trash;
            hrec[n] = make_uint4(links[n], rs | ((uint32_t)pb->model[n] << 16) | ((uint32_t)std::min(len, 7) << 20),
                                 (uint32_t)pb->arrival_us[pb->session[n]], c0 | (c1 << 16));
            wc23[n] = (len > 2 ? wl[a + 2] : trash) | ((uint32_t)(len > 3 ? wl[a + 3] : trash) << 16);
        }
    }
    size_t o_hrec = img.add(hrec.data(), sizeof(uint4) * N);
    size_t o_wc23 = img.add(wc23.data(), sizeof(uint32_t) * N);
    size_t o_wloff = img.add(wl_off.data(), sizeof(int32_t) * (N + 1));
    size_t o_wl = img.add(wl.data(), sizeof(uint16_t) * wl.size());
    size_t o_lk = img.add(lk.data(), sizeof(int2) * lk.size());
    // Status tables: the devices each activation fits on (Eq. 8), padded to a
    // multiple of four entries, and every edge packed as pred | succ << 16.
    std::vector<uint32_t> fitmask(((size_t)N + 15) & ~(size_t)15, 0u);  // read 16 at a time
    for (int32_t n = 0; n < N; ++n)
        for (int32_t d = 0; d < D; ++d)
            if (adm[(int64_t)n * D + d] <= pb->cap_mib[d]) fitmask[n] |= 1u << d;
    size_t o_fit = img.add(fitmask.data(), sizeof(uint32_t) * fitmask.size());
    // The same masks a byte each when every device index fits a byte's bits.
    std::vector<uint8_t> fit8(fitmask.size(), 0u);
    for (size_t n = 0; n < fitmask.size(); ++n) fit8[n] = (uint8_t)(fitmask[n] & 0xFFu);
    size_t o_fit8 = img.add(fit8.data(), fit8.size());
    std::vector<uint32_t> edges(((size_t)E + 3) & ~(size_t)3, 0u);  // read 4 at a time
    for (int32_t v = 0; v < N; ++v)
        for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e)
            edges[e] = (uint32_t)pb->pred_idx[e] | ((uint32_t)v << 16);
    size_t o_edges = img.add(edges.data(), sizeof(uint32_t) * edges.size());
    // Successor lists (the transpose of pred CSR) for the plan constructor,
    // and a bound on any time a plan of the window can reach.
    std::vector<int32_t> succ_off(N + 1, 0), succ_idx(E > 0 ? E : 1);
    for (int32_t e = 0; e < E; ++e) succ_off[pb->pred_idx[e] + 1] += 1;
    for (int32_t v = 0; v < N; ++v) succ_off[v + 1] += succ_off[v];
    {
        std::vector<int32_t> fill(succ_off.begin(), succ_off.end() - 1);
        for (int32_t v = 0; v < N; ++v)
            for (int32_t e = pb->pred_off[v]; e < pb->pred_off[v + 1]; ++e) succ_idx[fill[pb->pred_idx[e]]++] = v;
    }
    size_t o_soff = img.add(succ_off.data(), sizeof(int32_t) * (N + 1));
    size_t o_sidx = img.add(succ_idx.data(), sizeof(int32_t) * succ_idx.size());
    int64_t max_chain = 0;
    for (int32_t h = 0; h < N; ++h) {
        if (dv.fprev[h] >= 0) continue;
        int64_t sum = pb->grant_us;
        for (int32_t x = h; x >= 0; x = dv.fnext[x]) {
            int64_t worst = 0;
            for (int32_t d = 0; d < D; ++d) worst = std::max(worst, (int64_t)pb->lat_us[(int64_t)x * D + d]);
            sum += worst;
        }
        max_chain = std::max(max_chain, sum);
    }
    int64_t horizon = 0;
    for (int32_t w = 0; w < W; ++w) horizon = std::max(horizon, pb->arrival_us[w]);
    for (int32_t n = 0; n < N; ++n) {
        int64_t worst = 0;
        for (int32_t d = 0; d < D; ++d)
            worst = std::max(worst, (int64_t)pb->lat_us[(int64_t)n * D + d] +
                                        pb->load_us[(int64_t)pb->model[n] * D + d]);
        horizon += worst + pb->grant_us;
    }
    size_t o_ovf = img.add(nullptr, sizeof(int32_t) * (2 * (size_t)max_P + 64));

    wf_ctx *c = (wf_ctx *)calloc(1, sizeof(wf_ctx));
    if (!c) return wf_set_error(WF_ENOMEM, "host allocation of the context");
    c->device = device;
    c->max_P = max_P;
    c->force_int64 = false;
    c->tables_bytes = img.bytes.size();
    rc = wf_cuda_check(cudaMalloc(&c->tables, c->tables_bytes), "cudaMalloc(tables)");
    if (!rc) rc = wf_cuda_check(cudaMemcpy(c->tables, img.bytes.data(), c->tables_bytes,
                                           cudaMemcpyHostToDevice), "upload tables");
    if (rc) { wf_ctx_destroy(c); return rc; }
    uint8_t *base = (uint8_t *)c->tables;
    wf_dev_problem &dp = c->dp;
    dp.N = N; dp.D = D; dp.M = M; dp.W = W; dp.E = E;
    dp.grant = pb->grant_us;
    dp.S = pb->S;
    dp.seed = pb->seed;
    dp.bm_rn = stoch ? pb->bm_rn : 0;
    dp.bm_cn = stoch ? pb->bm_cn : 0;
    dp.bm_en = stoch ? pb->bm_en : 0;
    int64_t first = INT64_MAX;
    for (int32_t w = 0; w < W; ++w) first = std::min(first, pb->arrival_us[w]);
    dp.first_arrival = first;
    dp.pred_off = (const int32_t *)(base + o_poff);
    dp.pred_idx = (const int32_t *)(base + o_pidx);
    dp.fnext = (const int32_t *)(base + o_fnext);
    dp.fprev = (const int32_t *)(base + o_fprev);
    dp.model = (const uint8_t *)(base + o_model);
    dp.session = (const int32_t *)(base + o_sess);
    dp.arrival = (const int64_t *)(base + o_arr);
    dp.lat = (const int32_t *)(base + o_lat);
    dp.peak = (const int32_t *)(base + o_peak);
    dp.weight = (const int32_t *)(base + o_w);
    dp.load = (const int32_t *)(base + o_load);
    dp.cap = (const int32_t *)(base + o_cap);
    dp.lev_off = (const int32_t *)(base + o_loff);
    dp.lev_nodes = (const int32_t *)(base + o_lnodes);
    dp.nlev = (int32_t)dv.lev_off.size() - 1;
    dp.bm_r = (const int32_t *)(base + o_br);
    dp.bm_c = (const int32_t *)(base + o_bc);
    dp.bm_e = (const int32_t *)(base + o_be);
    dp.bm_r16 = t16 ? (const int16_t *)(base + o_br16) : nullptr;
    dp.bm_c16 = t16 ? (const int16_t *)(base + o_bc16) : nullptr;
    dp.err = (int *)(base + o_err);
    c->err = dp.err;
    dp.nslots = nslots > 0 ? nslots : 0;
    dp.noderec = (const int4 *)(base + o_rec);
    dp.wl_off = (const int32_t *)(base + o_wloff);
    dp.wl = (const uint16_t *)(base + o_wl);
    dp.lk = (const int2 *)(base + o_lk);
    dp.links = (const uint32_t *)(base + o_links);
    dp.hrec = (const uint4 *)(base + o_hrec);
    dp.wc23 = (const uint32_t *)(base + o_wc23);
    dp.fitmask = (const uint32_t *)(base + o_fit);
    dp.fit8 = (const uint8_t *)(base + o_fit8);
    dp.edges = (const uint32_t *)(base + o_edges);
    dp.succ_off = (const int32_t *)(base + o_soff);
    dp.succ_idx = (const int32_t *)(base + o_sidx);
    dp.horizon = horizon;
    dp.max_chain_run = max_chain;
    dp.reclaim = 0;
    dp.nextuse = nullptr;
    int64_t amax = 0;
    for (int32_t w = 0; w < W; ++w) amax = std::max(amax, pb->arrival_us[w]);
    dp.max_arrival = amax;
    c->ovf_count = (int32_t *)(base + o_ovf);
    c->ovf_list = c->ovf_count + 64;
    c->ovf_list2 = c->ovf_list + max_P;
    rc = wf_cuda_check(cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, device), "SM count");
    if (rc) { wf_ctx_destroy(c); return rc; }

    // Scratch for the evaluation kernels, bounded by a budget; a call with
    // more plans than the scratch holds walks over it in rounds.
    c->eval_row_bytes = wf_eval_row_bytes(dp);
    c->eval_scratch_bytes = wf_eval_scratch_bytes(dp, max_P, &c->eval_threads);
    rc = wf_cuda_check(cudaMalloc(&c->eval_scratch, c->eval_scratch_bytes), "cudaMalloc(eval scratch)");
    if (!rc) {
        c->topk_scratch_bytes = wf_topk_scratch_bytes(max_P);
        rc = wf_cuda_check(cudaMalloc(&c->topk_scratch, c->topk_scratch_bytes), "cudaMalloc(topk scratch)");
    }
    if (!rc) rc = wf_cuda_check(cudaMalloc(&c->search_scratch, wf_search_scratch_bytes(max_P)),
                                "cudaMalloc(search scratch)");
    if (!rc) rc = wf_cuda_check(cudaMallocHost(&c->h_ovf, sizeof(int32_t)), "cudaMallocHost(overflow count)");
    if (!rc) rc = wf_cuda_check(cudaEventCreateWithFlags(&c->ovf_event, cudaEventDisableTiming), "cudaEventCreate");
    if (!rc) rc = wf_cuda_check(cudaEventCreateWithFlags(&c->sweep_done, cudaEventDisableTiming), "cudaEventCreate");
    if (!rc) rc = wf_cuda_check(cudaStreamCreateWithFlags(&c->side, cudaStreamNonBlocking), "cudaStreamCreate");
    if (rc) { wf_ctx_destroy(c); return rc; }
    *out = c;
    return WF_OK;
}

extern "C" void wf_ctx_destroy(wf_ctx *c)
{
    if (!c) return;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(c->device);
    wf_host_release(c);
    if (c->tables) cudaFree(c->tables);
    if (c->eval_scratch) cudaFree(c->eval_scratch);
    if (c->topk_scratch) cudaFree(c->topk_scratch);
    if (c->search_scratch) cudaFree(c->search_scratch);
    if (c->construct_scratch) cudaFree(c->construct_scratch);
    if (c->dp.nextuse) cudaFree(c->dp.nextuse);
    if (c->side) cudaStreamSynchronize(c->side);
    if (c->side) cudaStreamDestroy(c->side);
    if (c->ovf_event) cudaEventDestroy(c->ovf_event);
    if (c->sweep_done) cudaEventDestroy(c->sweep_done);
    if (c->h_ovf) cudaFreeHost(c->h_ovf);
    if (prev >= 0) cudaSetDevice(prev);
    free(c);
}

static int select_device(wf_ctx *c)
{
    return wf_cuda_check(cudaSetDevice(c->device), "cudaSetDevice");
}

extern "C" int wf_forecast_readiness(wf_ctx *c, int64_t *rel, int64_t *comp, void *stream)
{
    REQUIRE(c && rel && comp, "NULL argument");
    int rc = select_device(c);
    if (rc) return rc;
    return wf_launch_forecast(c, rel, comp, (cudaStream_t)stream);
}

static bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

int wf_check_plans(const wf_ctx *c, const wf_plans *pl, const char *what)
{
    REQUIRE(pl, "%s: NULL plans", what);
    REQUIRE(pl->P >= 1 && pl->P <= c->max_P, "%s: P=%lld outside 1..max_P=%lld", what,
            (long long)pl->P, (long long)c->max_P);
    REQUIRE(pl->place && pl->order && pl->fuse && pl->prefetch, "%s: NULL plan array", what);
    const int64_t N = c->dp.N;
    const int64_t words = (N + 31) / 32;
    REQUIRE(pl->place_stride >= N && pl->place_stride % 16 == 0, "%s: place_stride", what);
    REQUIRE(pl->order_stride >= 2 * N && pl->order_stride % 16 == 0, "%s: order_stride", what);
    REQUIRE(pl->bits_stride >= 4 * words && pl->bits_stride % 16 == 0, "%s: bits_stride", what);
    REQUIRE(pl->plan_base >= 0, "%s: plan_base < 0", what);
    REQUIRE(aligned16(pl->place) && aligned16(pl->order) && aligned16(pl->fuse) &&
                aligned16(pl->prefetch) && (pl->retain == nullptr || aligned16(pl->retain)),
            "%s: plan arrays must be 16-byte aligned", what);
    return WF_OK;
}

int wf_check_out(const wf_eval_out *out, const char *what)
{
    REQUIRE(out, "%s: NULL results", what);
    REQUIRE(out->makespan_us && out->p95_us && out->gpu_us && out->status, "%s: NULL result array", what);
    return WF_OK;
}

int wf_select_device(const wf_ctx *c)
{
    return wf_cuda_check(cudaSetDevice(c->device), "cudaSetDevice");
}

extern "C" int wf_eval_plans(wf_ctx *c, const wf_plans *pl, const wf_eval_out *out, void *stream)
{
    REQUIRE(c && pl && out, "NULL argument");
    int rc = wf_check_plans(c, pl, "plans");
    if (!rc) rc = wf_check_out(out, "results");
    if (!rc) rc = select_device(c);
    if (rc) return rc;
    return wf_launch_eval(c, pl, out, (cudaStream_t)stream);
}

extern "C" int wf_topk(wf_ctx *c, const wf_eval_out *res, int64_t P, int32_t k, int32_t *ids,
                       int64_t *keys, void *stream)
{
    REQUIRE(c && res && ids, "NULL argument");
    REQUIRE(res->makespan_us && res->p95_us && res->gpu_us && res->status, "NULL result array");
    REQUIRE(P >= 1 && P <= c->max_P, "P outside 1..max_P");
    REQUIRE(k >= 1 && k <= 1024 && k <= P, "k=%d outside 1..min(P, 1024)", k);
    int rc = select_device(c);
    if (rc) return rc;
    return wf_launch_topk(c, res, P, k, ids, keys, (cudaStream_t)stream);
}

extern "C" int wf_eval_plans_phi(wf_ctx *c, const wf_plans *pl, const wf_eval_out *out, int64_t *timely,
                                 int64_t *life, void *stream)
{
    REQUIRE(c && pl && out && timely && life, "NULL argument");
    REQUIRE(c->dp.S == 0, "the window terms of Eq. 12 need deterministic latencies (S = 0)");
    int rc = wf_check_plans(c, pl, "plans");
    if (!rc) rc = wf_check_out(out, "results");
    if (!rc) rc = select_device(c);
    if (rc) return rc;
    // The kernels take the outputs from the problem they are launched with;
    // the context carries them for this call only.
    c->dp.phi_timely = timely;
    c->dp.phi_life = life;
    rc = wf_launch_eval(c, pl, out, (cudaStream_t)stream);
    c->dp.phi_timely = nullptr;
    c->dp.phi_life = nullptr;
    return rc;
}

extern "C" int wf_topk_phi(wf_ctx *c, const wf_eval_out *res, const int64_t *timely, const int64_t *life,
                           int64_t P, int32_t k, int32_t *ids, int64_t *keys, void *stream)
{
    REQUIRE(c && res && timely && life && ids, "NULL argument");
    REQUIRE(res->makespan_us && res->status, "NULL result array");
    REQUIRE(P >= 1 && P <= c->max_P, "P outside 1..max_P");
    REQUIRE(k >= 1 && k <= 1024 && k <= P, "k=%d outside 1..min(P, 1024)", k);
    int rc = select_device(c);
    if (rc) return rc;
    return wf_launch_topk(c, res, P, k, ids, keys, (cudaStream_t)stream, timely, life, -1);
}

extern "C" int wf_ctx_set_reclaim(wf_ctx *c, int32_t policy)
{
    REQUIRE(c, "NULL context");
    REQUIRE(policy == WF_RECLAIM_LRU || policy == WF_RECLAIM_NEXT_USE, "unknown reclamation policy %d", policy);
    if (policy == WF_RECLAIM_LRU) {
        c->dp.reclaim = 0;
        return WF_OK;
    }
    REQUIRE(c->dp.S == 0, "reclamation by next use needs deterministic latencies (S = 0)");
    REQUIRE(c->dp.batch == 0, "reclamation by next use is not modelled with a replica batch limit");
    REQUIRE(c->dp.max_chain_run < (int64_t)UINT32_MAX,
            "a fusible chain may run %lld us, beyond the shared-memory sweep", (long long)c->dp.max_chain_run);
    int rc = select_device(c);
    if (rc) return rc;
    wf_dev_problem probe = c->dp;
    probe.reclaim = 1;
    const wf_sweep_cfg cfg = wf_sweep_config(probe);
    REQUIRE(cfg.smem64, "reclamation by next use needs the 64-bit shared-memory sweep, "
                        "which this window does not fit");
    if (!c->dp.nextuse) {
        rc = wf_cuda_check(cudaMalloc(&c->dp.nextuse, sizeof(uint16_t) * (size_t)c->max_P * (size_t)c->dp.N),
                           "cudaMalloc(next-use table)");
        if (rc) { c->dp.nextuse = nullptr; return rc; }
    }
    c->dp.reclaim = 1;
    return WF_OK;
}

extern "C" int wf_ctx_status(wf_ctx *c, void *stream)
{
    REQUIRE(c, "NULL context");
    int rc = select_device(c);
    if (rc) return rc;
    rc = wf_cuda_check(cudaStreamSynchronize((cudaStream_t)stream), "cudaStreamSynchronize");
    if (rc) return rc;
    int err = 0;
    rc = wf_cuda_check(cudaMemcpy(&err, c->err, sizeof(int), cudaMemcpyDeviceToHost), "read error word");
    if (rc) return rc;
    if (err) {
        int zero = 0;
        cudaMemcpy(c->err, &zero, sizeof(int), cudaMemcpyHostToDevice);
        return wf_set_error(WF_ETIMEOUT, "device error word %d", err);
    }
    return WF_OK;
}

extern "C" int wf_ctx_set_eval_path(wf_ctx *c, int32_t path)
{
    REQUIRE(c, "NULL context");
    REQUIRE(path >= WF_PATH_AUTO && path <= WF_PATH_RELATIVE, "unknown eval path %d", path);
    if (path == WF_PATH_WIDE || path == WF_PATH_RELATIVE) {
        const int rc = select_device(c);
        if (rc) return rc;
        const wf_sweep_cfg cfg = wf_sweep_config(c->dp);
        REQUIRE(cfg.smem64, "this window does not fit the 64-bit sweep");
        REQUIRE(path == WF_PATH_WIDE || cfg.smemRel, "this window does not fit the relative-time sweep");
    }
    c->force_int64 = path == WF_PATH_INT64;
    c->start_path = path;
    return WF_OK;
}

extern "C" int wf_ctx_set_batch(wf_ctx *c, int32_t batch)
{
    REQUIRE(c, "NULL context");
    REQUIRE(batch >= 0 && batch <= 64, "replica batch limit %d outside 0..64", batch);
    if (batch > 0) {
        REQUIRE(c->dp.S == 0, "the replica batch limit needs deterministic latencies (S = 0)");
        REQUIRE(c->dp.reclaim == 0, "the replica batch limit is modelled with least-recently-used reclamation");
    }
    wf_dev_problem probe = c->dp;
    probe.batch = batch;
    const size_t row = wf_eval_row_bytes(probe);
    if (row > c->eval_row_bytes) {  // a longer state row: the evaluation scratch is rebuilt
        int rc = select_device(c);
        if (rc) return rc;
        int64_t threads = 0;
        const size_t bytes = wf_eval_scratch_bytes(probe, c->max_P, &threads);
        void *fresh = nullptr;
        rc = wf_cuda_check(cudaMalloc(&fresh, bytes), "cudaMalloc(eval scratch)");
        if (rc) return rc;
        rc = wf_cuda_check(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
        if (rc) { cudaFree(fresh); return rc; }
        cudaFree(c->eval_scratch);
        c->eval_scratch = fresh;
        c->eval_scratch_bytes = bytes;
        c->eval_threads = threads;
        c->eval_row_bytes = row;
    }
    c->dp.batch = batch;
    return WF_OK;
}
