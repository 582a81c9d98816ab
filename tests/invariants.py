"""Replay checker for one oracle trace.

It re-derives nothing from the oracle's code: it checks the equations the
paper states as constraints on any feasible graph-schedule plan.
"""
from fractions import Fraction

import numpy as np

from randprob import preds_of


def bit(row, n):
    n = int(n)
    return (int(row[n >> 5]) >> (n & 31)) & 1


def check_trace(prob, plans, p, res, fnext, forecast=None):
    """Raise AssertionError if the trace of plan p violates an invariant."""
    tr = res["trace"]
    N, D = prob.N, prob.D
    L = prob.lat_us.reshape(N, D).astype(np.int64)
    peak = prob.peak_mib.reshape(N, D).astype(np.int64)
    W = prob.weight_mib.astype(np.int64)
    place = plans.place[p, :N].astype(int)
    order = plans.order[p, :N].astype(int)
    fuse, pref = plans.fuse[p], plans.prefetch[p]
    retain = None if plans.retain is None else plans.retain[p]
    arr = prob.arrival_us
    g = prob.grant_us
    start, fin, head_of = tr["start"], tr["finish"], tr["head_of"]
    heads = [int(h) for h in tr["unit_head"]]

    # Every node executed exactly once, for its own run time on its device (Eq. 7).
    assert (head_of >= 0).all()
    for n in range(N):
        assert fin[n] == start[n] + L[n, place[n]], ("c = s + T", n)

    # Units: heads in dispatch order; chains are Eq. 3 edges with the fuse
    # bit set, on one device (Eq. 9), executed back to back.
    pos = np.empty(N, int)
    pos[order] = np.arange(N)
    assert heads == sorted(heads, key=lambda h: pos[h])
    members = {h: [] for h in heads}
    for n in range(N):
        members[int(head_of[n])].append(n)
    for h in heads:
        ch = sorted(members[h], key=lambda n: start[n])
        assert ch[0] == h
        for a, b in zip(ch, ch[1:]):
            assert fnext[a] == b and bit(fuse, b) == 1 and place[b] == place[h]
            assert start[b] == fin[a]
        last = ch[-1]
        nxt = fnext[last]
        assert nxt < 0 or bit(fuse, nxt) == 0 or place[nxt] != place[h], "chain not maximal"
        members[h] = ch
    # Release and graph precedence (Eq. 2, Eq. 7).
    for h in heads:
        w = prob.session[h]
        rel = tr["rel"][h]
        lower = [arr[w]] + [fin[v] for v in preds_of(prob, h)]
        assert rel == max(lower)
        assert start[h] >= rel + g
        le = tr["load_end"][h]
        if le >= 0:
            assert start[h] >= le + g          # load precedes its consumer (Eq. 9)
            ls = tr["load_start"][h]
            assert le - ls == prob.load_us[int(prob.model[h]) * D + place[h]]
            assert ls >= arr[w]
            if not bit(pref, h):
                assert ls >= rel              # only prefetch may start before release
    for n in range(N):
        for v in preds_of(prob, n):
            assert start[n] >= fin[v]

    # Resource order (Eq. 10): per device, units and their loads in dispatch
    # order never overlap; each unit starts as early as its constraints allow.
    t_free = np.zeros(D, np.int64)
    for h in heads:
        d = place[h]
        last = members[h][-1]
        ls = tr["load_start"][h]
        busy_from = ls if ls >= 0 else start[h] - g
        assert busy_from >= t_free[d]
        lb = max(t_free[d], tr["rel"][h])
        if ls >= 0:
            lb = max(lb, tr["load_end"][h])
        assert start[h] == lb + g, "unit starts later than its constraints"
        t_free[d] = fin[last]

    # Cumulative memory (Eq. 11) with least-recently-used reclamation.
    resident = [dict() for _ in range(D)]   # model -> last dispatch position
    for h in heads:
        d, m = place[h], int(prob.model[h])
        ch = members[h]
        kv = max(peak[j, d] - W[m] for j in ch)
        assert kv == tr["kv_adm"][h]
        ev = [k for k in range(prob.M) if (int(tr["evicted"][h]) >> k) & 1]
        hit = m in resident[d]
        assert (tr["load_start"][h] < 0) == hit
        need = kv if hit else W[m] + kv
        used = sum(W[k] for k in resident[d])
        # evictions are exactly the first others in reclamation order, taken
        # until it fits: least recent first, or (next-use reclamation)
        # redundant copies, then farthest next use per unit of reload cost,
        # then least recent
        if getattr(prob, "reclaim", 0):
            def order_key(k):
                red = any(k in resident[e] for e in range(D) if e != d)
                later = [pos[x] for x in heads if pos[x] > pos[h] and place[x] == d and int(prob.model[x]) == k]
                cost = int(prob.load_us[k * D + d])
                if not later or cost == 0:
                    return (not red, 0, 0, resident[d][k])
                return (not red, 1, Fraction(-(min(later) - pos[h]), cost), resident[d][k])
            others = sorted((order_key(k), k) for k in resident[d] if k != m)
        else:
            others = sorted((t, k) for k, t in resident[d].items() if k != m)
        taken = 0
        expect_ev = []
        while used - taken + need > prob.cap_mib[d]:
            _, k = others[len(expect_ev)]
            expect_ev.append(k)
            taken += W[k]
        assert sorted(ev) == sorted(expect_ev), ("reclamation victims", h, ev, expect_ev)
        for k in ev:
            del resident[d][k]
        resident[d][m] = pos[h]
        used = sum(W[k] for k in resident[d])
        assert used == tr["used_after"][h]
        assert used + kv <= prob.cap_mib[d], "Eq. 11 violated"
        if retain is not None and not bit(retain, ch[-1]):
            assert tr["reclaimed"][h] == 1
            del resident[d][m]
        else:
            assert tr["reclaimed"][h] == 0

    # GPU time: occupancy intervals per device are disjoint, cover every load
    # and execution on the device, and sum to the reported total.
    end = int(fin.max())
    occ = list(zip(tr["occ_dev"].tolist(), tr["occ_start"].tolist(), tr["occ_end"].tolist()))
    assert sum(e - s for _, s, e in occ) == res["gpu"]
    for d in range(D):
        iv = sorted((s, e) for dd, s, e in occ if dd == d)
        for (s0, e0), (s1, e1) in zip(iv, iv[1:]):
            assert e0 <= s1
        for h in heads:
            if place[h] != d:
                continue
            a = tr["load_start"][h] if tr["load_start"][h] >= 0 else start[h]
            b = fin[members[h][-1]]
            assert any(s <= a and b <= e for s, e in iv), ("activity outside occupancy", h)
    busy = sum(L[n, place[n]] for n in range(N)) + sum(
        tr["load_end"][h] - tr["load_start"][h] for h in heads if tr["load_start"][h] >= 0)
    assert busy <= res["gpu"] <= D * (end - int(arr.min()))

    # Metrics (Section 4.2).
    assert res["makespan"] == end - int(arr.min())
    comp = [max(fin[n] for n in range(N) if prob.session[n] == w) - arr[w] for w in range(prob.W)]
    assert res["p95"] == int(np.percentile(np.array(comp), 95, method="inverted_cdf"))

    # The release forecast (Eq. 2) is a lower bound on every plan.
    if forecast is not None:
        frel, fcomp = forecast
        for n in range(N):
            assert start[n] >= frel[n] and fin[n] >= fcomp[n]
        assert res["makespan"] >= int(fcomp.max()) - int(arr.min())
    return True
