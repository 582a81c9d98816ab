"""Pins for the oracle's replica batch limit B_q (simulate_batched).

Eq. 11 sums the request memory of every unit active at a transition
boundary, and concurrent units of one replica respect its batch limit B_q
(Section 3.5).  Read here: units of a device's current replica share it, up
to B_q at once, admitted in dispatch order to the slot that frees earliest
once resident weights + the KV needs of running units + their own fit; a unit
of another model waits for the device to drain.  Pinned by the hand-worked
windows t10-t12 (tests/golden), and here by the classic play at B_q = 1, an
invariant replay of every admission, and closed forms.
"""
import numpy as np
import pytest

import oracle
import wfgen
from randprob import preds_of, random_problem


def _plans(prob, P, seed, retain=None):
    return wfgen.make_plans(prob, P, seed, p_retain=retain)


@pytest.mark.parametrize("seed", range(6))
def test_batch_one_is_the_classic_play(seed):
    """B_q = 1 gives exactly the one-unit-at-a-time play (an independently
    pinned function), with retain bits, grants and prefetch bits."""
    rng = np.random.default_rng(900 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(2, 6)), D=int(rng.integers(1, 4)),
                          M=int(rng.integers(1, 5)), tight=bool(seed % 2))
    plans = _plans(prob, 40, seed, retain=0.6 if seed % 3 == 0 else None)
    a = oracle.eval_plans(prob, plans)
    b = oracle.eval_plans(prob.with_(batch=1), plans)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)


def _replay(prob, plans, p, B):
    """Every admission of plan p against Eq. 11 and the batch limit."""
    res = oracle.eval_plan(prob, plans, p, trace=True)
    if res["status"]:
        return res
    tr = res["trace"]
    N, D = prob.N, prob.D
    fin, start = tr["finish"], tr["start"]
    place, order = plans.place[p, :N], plans.order[p, :N]
    heads = [int(h) for h in tr["unit_head"]]
    members = {h: [n for n in range(N) if tr["head_of"][n] == h] for h in heads}
    end = {h: int(max(fin[n] for n in members[h])) for h in heads}
    adm = {h: int(tr["adm"][h]) for h in heads}
    pos = {int(order[i]): i for i in range(N)}
    for h in heads:
        d, m = int(place[h]), int(prob.model[h])
        # release (Eq. 2, 7) and execution back to back (Eq. 4)
        rel = max([int(prob.arrival_us[prob.session[h]])] + [int(fin[u]) for u in preds_of(prob, h)])
        assert start[h] >= rel + prob.grant_us
        assert adm[h] <= start[h] - prob.grant_us
        earlier = [g for g in heads if int(place[g]) == d and pos[g] < pos[h]]
        # admissions in dispatch order on each device
        assert all(adm[g] <= adm[h] for g in earlier)
        running = [g for g in earlier if end[g] > adm[h]]
        # units of another model never overlap this one
        assert all(int(prob.model[g]) == m for g in running if end[g] > adm[h])
        # the batch limit, counting this unit
        assert len(running) + 1 <= B
        # Eq. 11 at the admission: resident weights after it + running KV + own KV
        kv = sum(int(tr["kv_adm"][g]) for g in running)
        assert int(tr["used_after"][h]) + kv + int(tr["kv_adm"][h]) <= int(prob.cap_mib[d])
    return res


@pytest.mark.parametrize("seed", range(8))
def test_every_admission_respects_eq11_and_the_batch_limit(seed):
    rng = np.random.default_rng(950 + seed)
    B = int(rng.integers(2, 6))
    prob = random_problem(rng, n_sessions=int(rng.integers(2, 6)), D=int(rng.integers(1, 4)),
                          M=int(rng.integers(1, 5)), tight=bool(seed % 2)).with_(batch=B)
    plans = _plans(prob, 24, seed)
    for p in range(plans.P):
        _replay(prob, plans, p, B)


def _independent(n, lat, C, grant, cap=10**6, kv=5, weight=10):
    """n independent nodes of one model on one device, all arriving at 0."""
    return wfgen.Problem(
        N=n, D=1, M=1, W=1, pred_off=np.zeros(n + 1, np.int32), pred_idx=np.zeros(0, np.int32),
        model=np.zeros(n, np.uint8), session=np.zeros(n, np.int32), arrival_us=np.zeros(1, np.int64),
        lat_us=np.array(lat, np.int32), peak_mib=np.full(n, weight + kv, np.int32),
        weight_mib=np.array([weight], np.int32), load_us=np.array([C], np.int32),
        cap_mib=np.array([cap], np.int32), grant_us=grant)


def _one_plan(prob):
    pl = wfgen.Plans.empty(1, prob.N)
    pl.order[0, :prob.N] = range(prob.N)
    return pl


@pytest.mark.parametrize("n,B", [(1, 1), (3, 3), (5, 8), (6, 2), (7, 3)])
def test_closed_form_independent_units(n, B):
    """n independent units of one model, equal run time L: they run in waves
    of B after one load, so makespan = C + ceil(n / B) (grant + L)."""
    L, C, grant = 37, 11, 3
    prob = _independent(n, [L] * n, C, grant).with_(batch=B)
    res = oracle.eval_plan(prob, _one_plan(prob), 0)
    assert res["makespan"] == C + -(-n // B) * (grant + L) == res["gpu"]


@pytest.mark.parametrize("B", [2, 4])
def test_closed_form_capacity_for_k_units(B):
    """Capacity for the weights and k KV needs (k < B): at most k units run at
    once, so the units run in waves of k."""
    n, L, C, k = 6, 50, 7, 2
    prob = _independent(n, [L] * n, C, 0, cap=10 + k * 5).with_(batch=B)
    res = oracle.eval_plan(prob, _one_plan(prob), 0)
    assert res["makespan"] == C + -(-n // min(k, B)) * L
