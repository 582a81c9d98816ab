"""Pins of the oracle's plan constructor (Algorithm 1 read as a whole-window
list scheduler).

The constructor plays each decision forward with the evaluation rules, so its
own end time must equal what the evaluator reports for the plan it builds:
two separate code paths over the same arithmetic.  The other pins check the
decisions against what the reading fixes: validity (Eq. 8-10), the ranking by
release (aging), binding by predicted finish with resident models free of
loads, fused chains (Eq. 3), the prefetch rule, the jitter, Graham's bound for
list schedules, and a hand-worked window.
"""
import numpy as np
import pytest

import oracle
import wfgen
from randprob import random_problem


def consistent(prob, rows, ends):
    mk, p95, gpu, st = oracle.eval_plans(prob, rows)
    assert (st == 0).all()
    assert np.array_equal(mk, ends - int(np.min(prob.arrival_us)))


@pytest.mark.parametrize("jitter", [0, 1, 50000, 10 ** 9])
def test_plans_are_valid_and_play_as_constructed(jitter):
    for t in range(8):
        rng = np.random.default_rng(900 + t)
        prob = random_problem(rng, n_sessions=int(rng.integers(1, 7)), D=int(rng.integers(1, 6)),
                              M=int(rng.integers(1, 6)))
        if t % 2:
            prob = prob.with_(grant_us=int(rng.integers(1, 1000)))
        rows, ends = oracle.construct(prob, 6, seed=t, jitter=jitter, plan_base=100 * t)
        consistent(prob, rows, ends)


@pytest.mark.parametrize("name", ["tiny", "mix", "burst"])
def test_named_workloads_play_as_constructed(name):
    prob = wfgen.config(name).problem
    rows, ends = oracle.construct(prob, 4, seed=3, jitter=100000)
    consistent(prob, rows, ends)


def test_jitter_zero_gives_one_plan_and_jitter_gives_many():
    prob = wfgen.config("mix").problem
    rows, _ = oracle.construct(prob, 5, seed=1, jitter=0, plan_base=7)
    for p in range(1, 5):
        assert np.array_equal(rows.order[p], rows.order[0]) and np.array_equal(rows.place[p], rows.place[0])
    rows, _ = oracle.construct(prob, 8, seed=1, jitter=2_000_000)
    assert len({(rows.order[p].tobytes(), rows.place[p].tobytes()) for p in range(8)}) >= 6


def test_single_device_runs_in_arrival_order():
    """No edges, one device, no loads: the ready set is every node at once,
    ranked by its session's arrival, ties by node id."""
    N = 7
    arr = np.array([50, 10, 10, 0, 70, 20, 0], np.int64)
    prob = wfgen.Problem(N=N, D=1, M=1, W=N, pred_off=np.zeros(N + 1, np.int32), pred_idx=np.zeros(0, np.int32),
                         model=np.zeros(N, np.uint8), session=np.arange(N, dtype=np.int32), arrival_us=arr,
                         lat_us=np.full(N, 5, np.int32), peak_mib=np.full(N, 3, np.int32),
                         weight_mib=np.array([2], np.int32), load_us=np.zeros(1, np.int32),
                         cap_mib=np.array([8], np.int32))
    rows, ends = oracle.construct(prob, 1, seed=0, jitter=0)
    assert rows.order[0].tolist() == sorted(range(N), key=lambda v: (arr[v], v))
    consistent(prob, rows, ends)


def test_graham_bound_for_independent_units():
    """Identical devices, no loads or memory pressure, independent units all
    released at 0: a list schedule ends by sum(L) / D + max(L) (Graham 1966)."""
    rng = np.random.default_rng(31)
    for t in range(20):
        N, D = int(rng.integers(1, 40)), int(rng.integers(1, 6))
        L = rng.integers(1, 1000, N).astype(np.int32)
        prob = wfgen.Problem(N=N, D=D, M=1, W=1, pred_off=np.zeros(N + 1, np.int32), pred_idx=np.zeros(0, np.int32),
                             model=np.zeros(N, np.uint8), session=np.zeros(N, np.int32),
                             arrival_us=np.zeros(1, np.int64), lat_us=np.repeat(L, D).astype(np.int32),
                             peak_mib=np.full(N * D, 3, np.int32), weight_mib=np.array([1], np.int32),
                             load_us=np.zeros(D, np.int32), cap_mib=np.full(D, 1 << 20, np.int32))
        rows, ends = oracle.construct(prob, 3, seed=t, jitter=0)  # device jitter would break the greedy
        assert (ends * D <= int(L.sum()) + D * int(L.max())).all()
        consistent(prob, rows, ends)


def test_hand_worked_reuse_and_prefetch():
    """Two identical devices, one model (load 40 us), three independent nodes
    of one session at t=0 with L = 100, 10, 10, and the model fits once per
    device.  Ranks tie at 0, so nodes go in id order:
      n0 -> device 0 (both empty: finish 40 + 100 = 140 on either; tie -> 0);
      n1 -> device 1: finish 40 + 10 = 50, against 140 + 10 = 150 on device 0;
      n2 -> device 1, now resident: 50 + 10 = 60 (no load), against 150.
    No prefetch bit: every load starts when its device is free, at or after
    the release."""
    prob = wfgen.Problem(N=3, D=2, M=1, W=1, pred_off=np.zeros(4, np.int32), pred_idx=np.zeros(0, np.int32),
                         model=np.zeros(3, np.uint8), session=np.zeros(3, np.int32),
                         arrival_us=np.zeros(1, np.int64), lat_us=np.array([100, 100, 10, 10, 10, 10], np.int32),
                         peak_mib=np.full(6, 5, np.int32), weight_mib=np.array([4], np.int32),
                         load_us=np.array([40, 40], np.int32), cap_mib=np.array([6, 6], np.int32))
    rows, ends = oracle.construct(prob, 1, seed=0, jitter=0)
    assert rows.order[0].tolist() == [0, 1, 2]
    assert rows.place[0].tolist() == [0, 1, 1]
    assert rows.prefetch[0, 0] == 0 and rows.fuse[0, 0] == 0
    assert ends[0] == 140
    consistent(prob, rows, ends)


def test_resident_model_wins_a_tie_breaker():
    """n0 fits only device 1 (load 200, run 40: free at 240).  n1 (same model,
    another session arriving at 400) fits both: device 0 would prefetch and
    finish at 400 + 200 + 10 = 610, device 1 reuses the resident model and
    finishes at 410.  Without the residency credit the two would tie at 610
    and the lower device would win."""
    prob = wfgen.Problem(N=2, D=2, M=1, W=2, pred_off=np.zeros(3, np.int32), pred_idx=np.zeros(0, np.int32),
                         model=np.zeros(2, np.uint8), session=np.array([0, 1], np.int32),
                         arrival_us=np.array([0, 400], np.int64), lat_us=np.array([40, 40, 10, 10], np.int32),
                         peak_mib=np.array([9, 5, 5, 5], np.int32), weight_mib=np.array([4], np.int32),
                         load_us=np.array([200, 200], np.int32), cap_mib=np.array([6, 9], np.int32))
    rows, ends = oracle.construct(prob, 1, seed=0, jitter=0)
    assert rows.place[0].tolist() == [1, 1] and ends[0] == 410
    consistent(prob, rows, ends)


def test_prefetch_when_the_device_would_idle():
    """Chain a -> b of different models on a single device: b is released at
    a's finish, and its load could start earlier -- but the device is busy
    with a until then, so no prefetch.  On two devices b goes to the idle
    one and its load is prefetched (it starts at the arrival)."""
    def prob_of(D):
        return wfgen.Problem(N=2, D=D, M=2, W=1, pred_off=np.array([0, 0, 1], np.int32),
                             pred_idx=np.array([0], np.int32), model=np.array([0, 1], np.uint8),
                             session=np.zeros(2, np.int32), arrival_us=np.zeros(1, np.int64),
                             lat_us=np.full(2 * D, 100, np.int32), peak_mib=np.full(2 * D, 3, np.int32),
                             weight_mib=np.array([2, 2], np.int32), load_us=np.full(2 * D, 30, np.int32),
                             cap_mib=np.full(D, 8, np.int32))
    rows, ends = oracle.construct(prob_of(1), 1, seed=0, jitter=0)
    assert rows.prefetch[0, 0] == 0 and ends[0] == 30 + 100 + 30 + 100
    consistent(prob_of(1), rows, ends)
    rows, ends = oracle.construct(prob_of(2), 1, seed=0, jitter=0)
    assert rows.place[0].tolist() == [0, 1] and rows.prefetch[0, 0] == 0b10 and ends[0] == 30 + 100 + 100
    consistent(prob_of(2), rows, ends)


def test_decisions_follow_the_rules():
    """On random windows (no jitter): every fusible chain member that fits its
    head's device is fused onto it; fuse bits appear nowhere else; a head's
    prefetch bit is set exactly when its model was not resident and its
    device was free before its release."""
    for t in range(10):
        rng = np.random.default_rng(1200 + t)
        prob = random_problem(rng, n_sessions=int(rng.integers(1, 6)), D=int(rng.integers(1, 5)))
        rows, ends = oracle.construct(prob, 1, seed=t, jitter=0)
        N, D = prob.N, prob.D
        fn = oracle.fusible_next(prob)
        place, order = rows.place[0], rows.order[0]
        fbit = lambda n: (int(rows.fuse[0, n >> 5]) >> (n & 31)) & 1
        pbit = lambda n: (int(rows.prefetch[0, n >> 5]) >> (n & 31)) & 1
        pos = np.empty(N, int)
        pos[order] = np.arange(N)
        peak = prob.peak_mib.reshape(N, D)
        heads = set(range(N))
        for u in range(N):
            if fbit(u):
                heads.discard(u)
        fprev = {int(fn[u]): u for u in range(N) if fn[u] >= 0}
        for s in range(N):
            if fbit(s):
                u = fprev[s]
                assert place[s] == place[u] and pos[s] == pos[u] + 1
            elif s in fprev:
                u = fprev[s]
                assert peak[s, place[u]] > prob.cap_mib[place[u]]
        tr = oracle.eval_plan(prob, rows, 0, trace=True)["trace"]
        t_free = {}
        for i in range(len(tr["unit_head"])):
            h = int(tr["unit_head"][i])
            d = int(place[h])
            miss = int(tr["load_start"][h]) >= 0
            before = t_free.get(d, 0)
            assert pbit(h) == int(miss and before < int(tr["rel"][h]))
            t_free[d] = int(tr["finish"][tr["head_of"] == h].max())
        for n in range(N):
            if n not in heads:
                assert pbit(n) == 0
        # RankReady: each head is the smallest (release, id) among the nodes
        # whose predecessors were all dispatched before it
        done = np.zeros(N, bool)
        fin = tr["finish"]
        preds = [prob.pred_idx[prob.pred_off[v]:prob.pred_off[v + 1]] for v in range(N)]
        release = lambda v: max([int(prob.arrival_us[prob.session[v]])] + [int(fin[x]) for x in preds[v]])
        for h in tr["unit_head"]:
            ready = [v for v in range(N) if not done[v] and all(done[x] for x in preds[v])]
            assert min(ready, key=lambda v: (release(v), v)) == h
            done[tr["head_of"] == h] = True


def test_better_than_random_plans():
    """Not a definition pin: the constructed plan beats the best of 256 random
    plans on the tiny and mix windows (the evaluator scores both)."""
    for name in ("tiny", "mix"):
        prob = wfgen.config(name).problem
        rows, ends = oracle.construct(prob, 1, seed=0, jitter=0)
        rnd = oracle.eval_plans(prob, wfgen.make_plans(prob, 256, 5), threads=8)
        assert ends[0] - int(np.min(prob.arrival_us)) <= rnd[0][rnd[3] == 0].min()
