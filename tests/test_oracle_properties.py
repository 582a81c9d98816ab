"""Oracle pins that do not depend on the oracle's own code.

* textbook routines: longest path in a DAG (networkx), an LRU cache
  (functools.lru_cache), the nearest-rank percentile (numpy inverted_cdf);
* closed forms: serial chains, partitions of independent work;
* exhaustive enumeration on tiny windows;
* the paper's constraint equations replayed from the oracle's trace
  (tests/invariants.py) on random windows;
* monotonicity of prefetch.
"""
import functools
import itertools

import networkx as nx
import numpy as np
import pytest

import oracle
import wfgen
from invariants import check_trace
from randprob import preds_of, random_problem


def one_plan(N, place, order, fuse=(), prefetch=(), retain_off=None):
    pl = wfgen.Plans.empty(1, N, with_retain=retain_off is not None)
    pl.place[0, :N] = place
    pl.order[0, :N] = order
    for n in fuse:
        pl.fuse[0, n >> 5] |= np.uint32(1 << (n & 31))
    for n in prefetch:
        pl.prefetch[0, n >> 5] |= np.uint32(1 << (n & 31))
    if retain_off is not None:
        for n in range(N):
            if n not in retain_off:
                pl.retain[0, n >> 5] |= np.uint32(1 << (n & 31))
    return pl


def simple_problem(preds, D, lat, peak=None, model=None, session=None, arrival=(0,), weight=(10,),
                   load=None, cap=None, grant=0):
    """A window from explicit lists; by default peak = weight + 1 on every
    device, free loads and ample capacity."""
    N = len(preds)
    M = len(weight)
    model = list(model) if model is not None else [0] * N
    off = np.zeros(N + 1, np.int32)
    off[1:] = np.cumsum([len(p) for p in preds])
    lat = np.asarray(lat, np.int64).reshape(N, D)
    if peak is None:
        peak = [[weight[model[n]] + 1] * D for n in range(N)]
    return wfgen.Problem(
        N=N, D=D, M=M, W=len(arrival), pred_off=off,
        pred_idx=np.array([u for p in preds for u in p], np.int32),
        model=np.array(model, np.uint8),
        session=np.array(session if session is not None else [0] * N, np.int32),
        arrival_us=np.array(arrival, np.int64), lat_us=lat.astype(np.int32).reshape(-1),
        peak_mib=np.array(peak, np.int32).reshape(-1),
        weight_mib=np.array(weight, np.int32),
        load_us=np.array(load if load is not None else [[0] * D] * M, np.int32).reshape(-1),
        cap_mib=np.array(cap if cap is not None else [10**6] * D, np.int32), grant_us=grant)


def random_dag(rng, N, p_edge=0.3):
    perm = rng.permutation(N)
    preds = [[] for _ in range(N)]
    for j in range(N):
        for i in range(j):
            if rng.random() < p_edge:
                preds[perm[j]].append(int(perm[i]))
    return preds


def topo_order(preds):
    g = nx.DiGraph()
    g.add_nodes_from(range(len(preds)))
    g.add_edges_from((u, v) for v, ps in enumerate(preds) for u in ps)
    return list(nx.topological_sort(g))


def longest_path_to_each(preds, w_node, w_source):
    """Longest weighted path ending at each node, via networkx on a graph with
    a super source; node weights become in-edge weights."""
    N = len(preds)
    g = nx.DiGraph()
    for v in range(N):
        g.add_edge("src", v, w=int(w_source[v]) + int(w_node[v]))
        for u in preds[v]:
            g.add_edge(u, v, w=int(w_node[v]))
    out = np.zeros(N, np.int64)
    for v in range(N):
        sub = g.subgraph(nx.ancestors(g, v) | {v})
        out[v] = nx.dag_longest_path_length(sub, weight="w")
    return out


# --------------------------------------------------------------------------
# textbook routines
# --------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_private_devices_give_longest_path(seed):
    """Each node alone on its own device, free loads, no grant: every finish
    time is the longest path to that node (Eq. 2 + Eq. 7 with no contention)."""
    rng = np.random.default_rng(seed)
    N = int(rng.integers(5, 14))
    preds = random_dag(rng, N)
    sess = [0] * N
    lat = rng.integers(1, 1000, size=(N, N))
    arr = (int(rng.integers(0, 50)),)
    prob = simple_problem(preds, N, lat, session=sess, arrival=arr)
    res = oracle.eval_plan(prob, one_plan(N, list(range(N)), topo_order(preds)), 0, trace=True)
    lp = longest_path_to_each(preds, [lat[n, n] for n in range(N)], [arr[0]] * N)
    assert res["trace"]["finish"].tolist() == lp.tolist()
    assert res["makespan"] == int(lp.max()) - arr[0]
    # with every node prefetched and a uniform load cost C the source edge becomes max(arr + C, ...)
    C = int(rng.integers(1, 300))
    prob2 = prob.with_(load_us=np.full(N, C, np.int32))
    res2 = oracle.eval_plan(prob2, one_plan(N, list(range(N)), topo_order(preds),
                                            prefetch=range(N)), 0, trace=True)
    lp2 = longest_path_to_each(preds, [lat[n, n] for n in range(N)], [arr[0] + C] * N)
    assert res2["trace"]["finish"].tolist() == lp2.tolist()


@pytest.mark.parametrize("seed", range(6))
def test_forecast_is_longest_path(seed):
    """Eq. 2 over the window: comp[n] = longest path with the fastest feasible
    run time per node, from the session arrival."""
    rng = np.random.default_rng(100 + seed)
    prob = random_problem(rng, n_sessions=3)
    rel, comp = oracle.forecast(prob)
    N, D = prob.N, prob.D
    lat = prob.lat_us.reshape(N, D)
    fits = prob.peak_mib.reshape(N, D) <= prob.cap_mib[None, :]
    lmin = np.where(fits, lat, np.iinfo(np.int32).max).min(axis=1)
    preds = [preds_of(prob, v) for v in range(N)]
    lp = longest_path_to_each(preds, lmin, prob.arrival_us[prob.session])
    assert comp.tolist() == lp.tolist()
    assert (comp - rel == lmin).all()


@pytest.mark.parametrize("k,seed", [(1, 0), (2, 1), (3, 2), (4, 3), (3, 4)])
def test_single_device_loads_are_lru_cache_misses(k, seed):
    """One device, equal model sizes, no KV, capacity k models, no
    dependencies: the reclamation rule is a k-slot LRU cache, so the number of
    loads equals functools.lru_cache's miss count and makespan = sum L + C * misses."""
    rng = np.random.default_rng(seed)
    M, N, C, w = 6, 40, 7, 10
    seq = [int(x) for x in rng.integers(0, M, size=N)]
    lat = rng.integers(1, 50, size=(N, 1))
    prob = simple_problem([[] for _ in range(N)], 1, lat, model=seq,
                          peak=[[w]] * N, weight=[w] * M, load=[[C]] * M, cap=[k * w])

    @functools.lru_cache(maxsize=k)
    def fetch(m):
        return m

    for m in seq:
        fetch(m)
    misses = fetch.cache_info().misses
    res = oracle.eval_plan(prob, one_plan(N, [0] * N, list(range(N))), 0, trace=True)
    assert int((res["trace"]["load_start"] >= 0).sum()) == misses
    assert res["makespan"] == int(lat.sum()) + C * misses


@pytest.mark.parametrize("seed", range(4))
def test_p95_is_nearest_rank_percentile(seed):
    rng = np.random.default_rng(200 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(2, 25)), sizes=(4, 6), D=4)
    plans = wfgen.make_plans(prob, 8, seed)
    for p in range(8):
        res = oracle.eval_plan(prob, plans, p, trace=True)
        fin = res["trace"]["finish"]
        comp = [fin[prob.session == w].max() - prob.arrival_us[w] for w in range(prob.W)]
        assert res["p95"] == int(np.percentile(comp, 95, method="inverted_cdf"))


# --------------------------------------------------------------------------
# closed forms
# --------------------------------------------------------------------------

@pytest.mark.parametrize("fused", [False, True])
def test_single_model_chain_closed_form(fused):
    """D=1, one model, a chain: makespan = C + sum L + grant * (number of units)."""
    N, C, g = 7, 13, 4
    lat = np.arange(1, N + 1).reshape(N, 1) * 10
    prob = simple_problem([[]] + [[i] for i in range(N - 1)], 1, lat, load=[[C]], grant=g)
    res = oracle.eval_plan(prob, one_plan(N, [0] * N, list(range(N)),
                                          fuse=range(1, N) if fused else ()), 0)
    units = 1 if fused else N
    assert res["makespan"] == C + int(lat.sum()) + g * units == res["gpu"]


@pytest.mark.parametrize("seed", range(3))
def test_independent_work_partition_closed_form(seed):
    """Brute force over all 2^6 placements of 6 independent activations on 2
    devices (free loads, ample memory): makespan = max over devices of the
    summed run times, GPU time = makespan * devices used."""
    rng = np.random.default_rng(300 + seed)
    N, D = 6, 2
    lat = rng.integers(1, 100, size=(N, D))
    prob = simple_problem([[] for _ in range(N)], D, lat)
    places = list(itertools.product(range(D), repeat=N))
    pl = wfgen.Plans.empty(len(places), N)
    for r, pc in enumerate(places):
        pl.place[r, :N] = pc
        pl.order[r, :N] = rng.permutation(N)
    mk, p95, gpu, st = oracle.eval_plans(prob, pl)
    for r, pc in enumerate(places):
        loads = [sum(int(lat[n, d]) for n in range(N) if pc[n] == d) for d in range(D)]
        assert mk[r] == max(loads)
        assert gpu[r] == mk[r] * sum(1 for d in range(D) if loads[d] > 0 or d in pc)
    best = min(max(sum(int(lat[n, d]) for n in range(N) if pc[n] == d) for d in range(D))
               for pc in places)
    assert mk.min() == best


def test_brute_force_same_model_chain_optimum():
    """Exhaustive N=6, D=2: a same-model 6-chain with dev0 strictly faster.
    The unique best makespan is every activation on dev0, fully fused:
    C + grant + sum L0 (one load, one grant)."""
    N, D, C, g = 6, 2, 50, 3
    lat = np.array([[10 * (n + 1), 10 * (n + 1) + 7] for n in range(N)])
    prob = simple_problem([[]] + [[i] for i in range(N - 1)], D, lat, load=[[C, C]], grant=g)
    rows = []
    for pc in itertools.product(range(D), repeat=N):
        for fz in range(1 << (N - 1)):
            rows.append((pc, [n for n in range(1, N) if (fz >> (n - 1)) & 1]))
    pl = wfgen.Plans.empty(len(rows), N)
    for r, (pc, fu) in enumerate(rows):
        pl.place[r, :N] = pc
        pl.order[r, :N] = range(N)
        for n in fu:
            pl.fuse[r, 0] |= np.uint32(1 << n)
    mk, p95, gpu, st = oracle.eval_plans(prob, pl)
    assert (st == 0).all()
    best = C + g + int(lat[:, 0].sum())
    assert mk.min() == best
    winners = [rows[r] for r in np.nonzero(mk == best)[0]]
    assert winners == [((0,) * N, list(range(1, N)))]
    ids, keys = oracle.topk(mk, p95, gpu, st, 3)
    order = np.lexsort((np.arange(len(rows)), gpu, p95, mk))
    assert ids.tolist() == order[:3].tolist()


def test_brute_force_all_plans_satisfy_invariants():
    """Exhaustive N=6, D=2 window: every placement (infeasible ones flagged),
    every topological order, and every fuse x prefetch pattern of one plan."""
    preds = [[], [0], [0], [1, 2], [3], [3]]
    N, D = 6, 2
    rng = np.random.default_rng(7)
    lat = rng.integers(5, 60, size=(N, D))
    model = [0, 1, 1, 0, 0, 1]
    peak = [[30, 30], [25, 25], [25, 25], [30, 30], [30, 30], [45, 25]]  # node 5 does not fit dev0
    prob = simple_problem(preds, D, lat, peak=peak, model=model, weight=(20, 15),
                          load=[[9, 12], [8, 5]], cap=[40, 60], grant=1)
    g = nx.DiGraph([(u, v) for v, ps in enumerate(preds) for u in ps])
    orders = list(nx.all_topological_sorts(g))
    fnext = oracle.fusible_next(prob)
    frc = oracle.forecast(prob)
    rows = [(pc, od, 0, 0) for pc in itertools.product(range(D), repeat=N) for od in orders]
    base_pc, base_od = (0, 1, 0, 1, 1, 1), orders[0]
    rows += [(base_pc, base_od, fz, pf) for fz in range(64) for pf in range(64)]
    pl = wfgen.Plans.empty(len(rows), N)
    for r, (pc, od, fz, pf) in enumerate(rows):
        pl.place[r, :N] = pc
        pl.order[r, :N] = od
        pl.fuse[r, 0] = fz
        pl.prefetch[r, 0] = pf
    n_valid = 0
    op = oracle.OracleProblem(prob)
    for r, (pc, od, fz, pf) in enumerate(rows):
        res = oracle.eval_plan(prob, pl, r, trace=True, op=op)
        assert res["status"] == (2 if pc[5] == 0 else 0)
        if res["status"] == 0:
            n_valid += 1
            check_trace(prob, pl, r, res, fnext, forecast=frc)
    assert n_valid == len(rows) - len(orders) * 2 ** (N - 1)


# --------------------------------------------------------------------------
# invariants on random windows
# --------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(12))
def test_random_windows_satisfy_invariants(seed):
    rng = np.random.default_rng(1000 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 6)), D=int(rng.integers(1, 5)),
                          M=int(rng.integers(1, 6)))
    with_retain = seed % 2 == 1
    plans = wfgen.make_plans(prob, 24, seed, p_fuse=float(rng.uniform(0, 1)),
                             p_prefetch=float(rng.uniform(0, 1)),
                             p_retain=0.6 if with_retain else None)
    fnext = oracle.fusible_next(prob)
    frc = oracle.forecast(prob)
    op = oracle.OracleProblem(prob)
    for p in range(plans.P):
        res = oracle.eval_plan(prob, plans, p, trace=True, op=op)
        assert res["status"] == 0
        check_trace(prob, plans, p, res, fnext, forecast=frc)


def test_fusible_edges_match_definition():
    """Eq. 3 on a random window: compared with networkx degree queries."""
    rng = np.random.default_rng(5)
    prob = random_problem(rng, n_sessions=6)
    fnext = oracle.fusible_next(prob)
    g = nx.DiGraph()
    g.add_nodes_from(range(prob.N))
    g.add_edges_from((u, v) for v in range(prob.N) for u in preds_of(prob, v))
    for u in range(prob.N):
        succ = list(g.successors(u))
        ok = len(succ) == 1 and g.in_degree(succ[0]) == 1 and prob.model[u] == prob.model[succ[0]]
        assert fnext[u] == (succ[0] if ok else -1)
    assert (fnext >= 0).sum() > 0


# --------------------------------------------------------------------------
# monotonicity
# --------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_prefetch_never_delays(seed):
    """Residency decisions do not depend on times, and every time is a max / +
    of earlier times, so setting a prefetch bit can only move finishes earlier."""
    rng = np.random.default_rng(2000 + seed)
    prob = random_problem(rng, n_sessions=4, D=3)
    plans = wfgen.make_plans(prob, 6, seed, p_prefetch=0.0)
    op = oracle.OracleProblem(prob)
    for p in range(plans.P):
        base = oracle.eval_plan(prob, plans, p, trace=True, op=op)
        for n in rng.choice(prob.N, size=min(6, prob.N), replace=False):
            pl = plans.slice(p, p + 1)
            pl.prefetch = pl.prefetch.copy()
            pl.prefetch[0, n >> 5] |= np.uint32(1 << (n & 31))
            pl.plan_base = plans.plan_base + p
            res = oracle.eval_plan(prob, pl, 0, trace=True, op=op)
            assert (res["trace"]["finish"] <= base["trace"]["finish"]).all()
            assert res["makespan"] <= base["makespan"] and res["p95"] <= base["p95"]


@pytest.mark.parametrize("seed", range(3))
def test_grant_and_load_costs_never_speed_up(seed):
    rng = np.random.default_rng(3000 + seed)
    prob = random_problem(rng, n_sessions=4, D=3, grant=0)
    plans = wfgen.make_plans(prob, 8, seed)
    a = oracle.eval_plans(prob, plans)
    b = oracle.eval_plans(prob.with_(grant_us=5), plans)
    c = oracle.eval_plans(prob.with_(load_us=prob.load_us * 2), plans)
    assert (b[0] >= a[0]).all() and (c[0] >= a[0]).all()


@pytest.mark.parametrize("seed", range(6))
def test_phi_terms_closed_form_without_reclamation(seed):
    """Eq. 12's window terms with room for every model and no prefetch bits:
    each model loads once per device, at its first use there, and each load
    delays its unit by exactly the load time, so H_life is the sum of C[m,d]
    over the (device, model) pairs a plan uses, and P_N is 0.  Setting every
    prefetch bit can only make loads timely, never more than there are units."""
    rng = np.random.default_rng(7100 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 5)), D=int(rng.integers(1, 5)),
                          M=int(rng.integers(1, 6)), tight=False)
    prob = prob.with_(cap_mib=np.full(prob.D, 10**8, np.int32))
    plans = wfgen.make_plans(prob, 40, seed, p_prefetch=0.0)
    mk, p95, gpu, st = oracle.eval_plans(prob, plans)
    timely, life = oracle.eval_phi(prob, plans)
    load = np.asarray(prob.load_us).reshape(prob.M, prob.D)
    model = np.asarray(prob.model)
    for p in range(plans.P):
        assert st[p] == 0
        pairs = {(int(plans.place[p, n]), int(model[n])) for n in range(prob.N)}
        assert timely[p] == 0
        assert life[p] == sum(int(load[m, d]) for d, m in pairs)
    allpf = wfgen.make_plans(prob, 40, seed, p_prefetch=1.0)
    timely2, life2 = oracle.eval_phi(prob, allpf)
    assert (timely2 <= prob.N).all() and (life2 <= life).all()
