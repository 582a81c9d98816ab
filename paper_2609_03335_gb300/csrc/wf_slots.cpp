// Static assignment of finish-time slots for the per-plan sweep.
//
// The sweep needs, when it starts a unit with head h, the latest finish among
// h's graph predecessors (Eq. 2, Eq. 7), and at the end every session's last
// finish (Section 4.2).  Storing one finish time per activation costs N words
// per plan; this pass assigns far fewer words, valid for EVERY plan
// (every placement, dispatch order and fusion pattern), from the DAG alone:
//
//  * pull slot O(u): written with u's finish when u ends a unit; read by each
//    successor whose only predecessor is u;
//  * accumulator A(s) for s with two or more predecessors: every predecessor
//    max-accumulates its finish into it, s reads it and resets it to 0;
//  * session slot w (indices 0..W-1): every sink of session w max-accumulates.
//
// Two pull slots (or two accumulators) may share a word when, in every
// topological order, all reads of one precede every write of the other.  A
// write by node y happens when y's unit starts, which is at or after the
// first node of y's maximal fusible run (Eq. 3) -- or at or after the reader
// itself when the reader lies on y's run before y.  Sessions are independent
// (no edges between them), so their slots never share.
#include <algorithm>
#include <cstdint>
#include <vector>

#include "wf_internal.cuh"

namespace {

struct Logical {
    int32_t key;                   // u for a pull slot, s for an accumulator
    std::vector<int32_t> writers;  // nodes that write it
    std::vector<int32_t> readers;  // nodes that read it
};

}  // namespace

int32_t wf_assign_slots(int32_t N, int32_t W, const int32_t *pred_off, const int32_t *pred_idx,
                        const int32_t *session, const int32_t *fprev, const int32_t *fnext,
                        int32_t *rslot, std::vector<int32_t> &wl_off, std::vector<uint16_t> &wl)
{
    std::vector<int32_t> nsucc(N, 0), soff(N + 1, 0), sidx, fill(N), indeg(N);
    for (int32_t v = 0; v < N; ++v)
        for (int32_t e = pred_off[v]; e < pred_off[v + 1]; ++e) nsucc[pred_idx[e]] += 1;
    for (int32_t u = 0; u < N; ++u) soff[u + 1] = soff[u] + nsucc[u];
    sidx.resize(std::max(soff[N], 1));
    for (int32_t u = 0; u < N; ++u) fill[u] = soff[u];
    for (int32_t v = 0; v < N; ++v) {
        indeg[v] = pred_off[v + 1] - pred_off[v];
        for (int32_t e = pred_off[v]; e < pred_off[v + 1]; ++e) sidx[fill[pred_idx[e]]++] = v;
    }
    auto npred = [&](int32_t v) { return pred_off[v + 1] - pred_off[v]; };

    // Topological order, and the first node of each maximal fusible run.
    std::vector<int32_t> topo;
    topo.reserve(N);
    for (int32_t v = 0; v < N; ++v) if (indeg[v] == 0) topo.push_back(v);
    for (size_t k = 0; k < topo.size(); ++k) {
        int32_t u = topo[k];
        for (int32_t e = soff[u]; e < soff[u + 1]; ++e)
            if (--indeg[sidx[e]] == 0) topo.push_back(sidx[e]);
    }
    std::vector<int32_t> run(N);
    for (int32_t n : topo) run[n] = fprev[n] >= 0 ? run[fprev[n]] : n;

    // Nodes of each session in topological order.
    std::vector<std::vector<int32_t>> members(W);
    for (int32_t n : topo) members[session[n]].push_back(n);

    std::vector<std::vector<std::pair<int32_t, int>>> writes(N);  // (slot, max-accumulate)
    for (int32_t v = 0; v < N; ++v) rslot[v] = -1;
    int32_t next = W;  // slots 0..W-1 are the session slots
    std::vector<int32_t> local(N, -1);
    const size_t kMaxColoured = 2048;

    for (int32_t w = 0; w < W; ++w) {
        const std::vector<int32_t> &nodes = members[w];
        const size_t n = nodes.size();
        for (size_t i = 0; i < n; ++i) local[nodes[i]] = (int32_t)i;
        const size_t words = (n + 63) / 64;
        const bool colour = n <= kMaxColoured;
        // anc[i]: bitset of nodes that are ancestors of nodes[i], or nodes[i] itself.
        std::vector<uint64_t> anc(colour ? n * words : 0, 0);
        if (colour) {
            for (size_t i = 0; i < n; ++i) {
                uint64_t *a = &anc[i * words];
                a[i / 64] |= 1ull << (i % 64);
                int32_t v = nodes[i];
                for (int32_t e = pred_off[v]; e < pred_off[v + 1]; ++e) {
                    const uint64_t *b = &anc[(size_t)local[pred_idx[e]] * words];
                    for (size_t k = 0; k < words; ++k) a[k] |= b[k];
                }
            }
        }
        auto aoe = [&](int32_t r, int32_t x) {  // r is x or an ancestor of x
            size_t ri = local[r], xi = local[x];
            return (anc[xi * words + ri / 64] >> (ri % 64)) & 1ull;
        };
        auto write_floor = [&](int32_t r, int32_t y) {  // earliest unit head that can write y's slot
            return (run[r] == run[y] && aoe(r, y)) ? r : run[y];
        };
        auto before = [&](const Logical &x, const Logical &y) {
            for (int32_t r : x.readers)
                for (int32_t wr : y.writers)
                    if (!aoe(r, write_floor(r, wr))) return false;
            return true;
        };
        auto assign = [&](std::vector<Logical> &L) {
            std::vector<std::vector<int32_t>> colours;  // indices into L
            std::vector<int32_t> of(L.size());
            for (size_t i = 0; i < L.size(); ++i) {
                int32_t c = -1;
                if (colour) {
                    for (size_t k = 0; k < colours.size() && c < 0; ++k) {
                        bool ok = true;
                        for (int32_t j : colours[k])
                            if (!before(L[i], L[j]) && !before(L[j], L[i])) { ok = false; break; }
                        if (ok) c = (int32_t)k;
                    }
                }
                if (c < 0) { c = (int32_t)colours.size(); colours.emplace_back(); }
                colours[c].push_back((int32_t)i);
                of[i] = c;
            }
            int32_t base = next;
            next += (int32_t)colours.size();
            for (auto &x : of) x += base;
            return of;
        };

        std::vector<Logical> pull, acc;
        for (int32_t u : nodes) {
            Logical x;
            x.key = u;
            x.writers = {u};
            for (int32_t e = soff[u]; e < soff[u + 1]; ++e)
                if (npred(sidx[e]) == 1) x.readers.push_back(sidx[e]);
            if (!x.readers.empty()) pull.push_back(std::move(x));
        }
        for (int32_t s : nodes) {
            if (npred(s) < 2) continue;
            Logical x;
            x.key = s;
            x.readers = {s};
            for (int32_t e = pred_off[s]; e < pred_off[s + 1]; ++e) x.writers.push_back(pred_idx[e]);
            acc.push_back(std::move(x));
        }
        std::vector<int32_t> po = assign(pull), pa = assign(acc);
        for (size_t i = 0; i < pull.size(); ++i) {
            writes[pull[i].key].push_back({po[i], 0});
            for (int32_t r : pull[i].readers) rslot[r] = po[i];
        }
        for (size_t i = 0; i < acc.size(); ++i) {
            rslot[acc[i].key] = pa[i] | WF_RSLOT_ACC;
            for (int32_t wr : acc[i].writers) writes[wr].push_back({pa[i], 1});
        }
        for (int32_t v : nodes)
            if (soff[v + 1] == soff[v]) writes[v].push_back({w, 1});
        if (next > 32767) {  // too many slots: the sweep does not apply (empty write lists)
            wl_off.assign(N + 1, 0);
            wl.clear();
            for (int32_t v = 0; v < N; ++v) rslot[v] = -1;
            return -1;
        }
    }
    wl_off.assign(N + 1, 0);
    wl.clear();
    for (int32_t v = 0; v < N; ++v) {
        for (auto &pr : writes[v]) wl.push_back((uint16_t)(pr.first | (pr.second << 15)));
        wl_off[v + 1] = (int32_t)wl.size();
    }
    (void)fnext;
    return next;
}
