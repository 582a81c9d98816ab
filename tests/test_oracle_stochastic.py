"""Pins for the stochastic-latency evaluation (S > 0).

The multiplier of (plan, sample, node) comes from a SplitMix64 hash through
integer Box-Muller tables; results are floor means of makespan and GPU time
over samples and a nearest-rank p95 over the pooled S x W completions.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import wfgen
from randprob import random_problem

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
GAMMA = 0x9E3779B97F4A7C15


def test_splitmix64_published_vector():
    with open(os.path.join(GOLDEN, "splitmix64_rosetta.json")) as f:
        fx = json.load(f)
    state = fx["seed"]
    for k, want in enumerate(fx["outputs"]):
        # output k is the finaliser of state + (k+1) * gamma; orc_splitmix64(x)
        # adds one gamma itself
        assert oracle.splitmix64((state + k * GAMMA) % (1 << 64)) == int(want)


def test_multiplier_hand_derived():
    """The multiplier of three (seed, plan, sample, node) tuples worked by hand
    in tests/golden/multiplier_hand_derived.json: each nested mix input is a
    Rosetta state, so every hash value is a published SplitMix64 output; the
    table entries, the floored product and the multiplier follow from the
    table formulas.  A wrong nesting order, wrong index bits, a truncating
    zq or a wrong table entry changes the result."""
    with open(os.path.join(GOLDEN, "multiplier_hand_derived.json")) as f:
        fx = json.load(f)
    with open(os.path.join(GOLDEN, "splitmix64_rosetta.json")) as f:
        out = [int(x) for x in json.load(f)["outputs"]]
    state = {int(k): int(v) for k, v in fx["states"].items()}
    for k, v in state.items():
        assert v == (1234567 + k * GAMMA) % (1 << 64)
    r, c, e = wfgen.box_muller_tables()
    rng = np.random.default_rng(0)
    for case in fx["cases"]:
        seed, plan, sample, node = (int(case[x]) for x in ("seed", "plan", "sample", "node"))
        a, b, cc = case["a"], case["b"], case["c"]
        # the chosen inputs land each nested step on a published state
        assert seed ^ plan == state[a]
        assert out[a] ^ sample == state[b]
        assert out[b] ^ node == state[cc]
        steps = list(case["steps"].values())
        assert int(steps[2]) == out[cc]
        prob = _stoch_problem(rng, S=1, tables=(r, c, e)).with_(seed=seed)
        assert oracle.multiplier(prob, plan, sample, node) == case["multiplier"]


def _stoch_problem(rng, S, tables=None, **kw):
    prob = random_problem(rng, **kw)
    r, c, e = tables or wfgen.box_muller_tables()
    return prob.with_(S=S, seed=int(rng.integers(0, 2**63)), bm_r=r, bm_c=c, bm_e=e)


def test_tables_shape():
    r, c, e = wfgen.box_muller_tables()
    assert len(r) == len(c) == 4096 and len(e) % 2 == 1
    zoff = (len(e) - 1) // 2
    assert e[zoff] == 65536
    assert (np.diff(r) <= 0).all() and r.min() >= 0
    # the largest |floor(R*C / 2^18)| fits the multiplier table
    prod = int(r.max()) * int(np.abs(c).max())
    assert -((-prod) >> 18) <= zoff


def test_multiplier_statistics():
    """log(multiplier) ~ N(0, 0.3^2): mean, spread, tails, and independence
    between samples and between nodes."""
    rng = np.random.default_rng(11)
    prob = _stoch_problem(rng, S=4)
    op = oracle.OracleProblem(prob)
    import ctypes
    f = op.lib.orc_multiplier
    vals = np.array([[f(ctypes.byref(op.c), p, s, n) for s in range(8) for n in range(40)]
                     for p in range(300)], np.float64)
    lz = np.log(vals / 65536.0).reshape(300, 8, 40)
    z = lz / 0.3
    assert abs(z.mean()) < 0.02
    assert abs(z.std() - 1.0) < 0.02
    assert abs((np.abs(z) > 1.959964).mean() - 0.05) < 0.006
    assert abs(np.corrcoef(z[:, 0, :].ravel(), z[:, 1, :].ravel())[0, 1]) < 0.05
    assert abs(np.corrcoef(z[:, :, 0].ravel(), z[:, :, 1].ravel())[0, 1]) < 0.05
    assert abs(np.corrcoef(z[:-1].ravel(), z[1:].ravel())[0, 1]) < 0.05


@pytest.mark.parametrize("seed", range(4))
def test_unit_multiplier_reproduces_deterministic(seed):
    """With every table entry 65536 (multiplier 1) each sample is the
    deterministic play, so the floor means and the pooled p95 equal it."""
    rng = np.random.default_rng(500 + seed)
    r, c, e = wfgen.box_muller_tables()
    prob = _stoch_problem(rng, S=3, tables=(r, c, np.full_like(e, 65536)), n_sessions=5)
    plans = wfgen.make_plans(prob, 16, seed, p_retain=0.7 if seed % 2 else None)
    a = oracle.eval_plans(prob, plans)
    b = oracle.eval_plans(prob.with_(S=0), plans)
    for x, y in zip(a, b):
        assert (x == y).all()


def test_scaled_multiplier_rounds_half_up():
    """Multiplier 1.5 everywhere: L' = floor(1.5 L + 1/2); on one device with
    free loads the makespan of a chain is the sum of the rounded run times."""
    rng = np.random.default_rng(3)
    N = 9
    lat = np.array([1, 2, 3, 5, 7, 11, 101, 1001, 99999], np.int64)
    r, c, e = wfgen.box_muller_tables()
    prob = wfgen.Problem(
        N=N, D=1, M=1, W=1, pred_off=np.arange(N + 1, dtype=np.int32) - 1,
        pred_idx=np.arange(N - 1, dtype=np.int32), model=np.zeros(N, np.uint8),
        session=np.zeros(N, np.int32), arrival_us=np.zeros(1, np.int64),
        lat_us=lat.astype(np.int32), peak_mib=np.full(N, 11, np.int32),
        weight_mib=np.array([10], np.int32), load_us=np.zeros(1, np.int32),
        cap_mib=np.array([100], np.int32), S=2, seed=int(rng.integers(0, 2**62)),
        bm_r=r, bm_c=c, bm_e=np.full_like(e, 98304))
    prob.pred_off[0] = 0
    pl = wfgen.Plans.empty(1, N)
    pl.order[0, :N] = range(N)
    res = oracle.eval_plan(prob, pl, 0)
    want = sum(math.floor(Fraction(3, 2) * int(x) + Fraction(1, 2)) for x in lat)
    assert res["makespan"] == want == res["p95"] == res["gpu"]


@pytest.mark.parametrize("seed", range(3))
def test_stochastic_aggregation(seed):
    """The stochastic result equals S deterministic plays with the per-sample
    run times, combined as floor means and a pooled nearest-rank p95."""
    rng = np.random.default_rng(700 + seed)
    prob = _stoch_problem(rng, S=5, n_sessions=4)
    plans = wfgen.make_plans(prob, 5, seed, plan_base=1000 * seed)
    op = oracle.OracleProblem(prob)
    import ctypes
    N, D = prob.N, prob.D
    for p in range(plans.P):
        got = oracle.eval_plan(prob, plans, p, op=op)
        mks, gpus, pool = [], [], []
        for s in range(prob.S):
            mult = np.array([op.lib.orc_multiplier(ctypes.byref(op.c), plans.plan_base + p, s, n)
                             for n in range(N)], np.int64)
            lat = (prob.lat_us.reshape(N, D).astype(np.int64) * mult[:, None] + 32768) >> 16
            det = prob.with_(S=0, lat_us=lat.astype(np.int32).reshape(-1))
            res = oracle.eval_plan(det, plans, p, trace=True)
            fin = res["trace"]["finish"]
            pool += [int(fin[det.session == w].max() - det.arrival_us[w]) for w in range(det.W)]
            mks.append(res["makespan"])
            gpus.append(res["gpu"])
        assert got["makespan"] == sum(mks) // prob.S
        assert got["gpu"] == sum(gpus) // prob.S
        assert got["p95"] == int(np.percentile(pool, 95, method="inverted_cdf"))


def test_samples_differ_and_plans_differ():
    rng = np.random.default_rng(9)
    prob = _stoch_problem(rng, S=1, n_sessions=3)
    plans = wfgen.make_plans(prob, 2, 0)
    same = plans.slice(0, 1)
    other = plans.slice(0, 1)
    other.plan_base = 12345
    a = oracle.eval_plan(prob, same, 0)
    b = oracle.eval_plan(prob, other, 0)
    assert a["makespan"] != b["makespan"]  # the hash depends on the plan index


@pytest.mark.parametrize("r,c,mult", [(1, -1, 2), (262144, -1, 2), (1, 1, 1), (262144, 1, 3), (0, -5, 1)])
def test_z_is_floor_of_product(r, c, mult):
    """zq = floor(R * Cc / 2^18) exactly: with one-valued tables the product
    is known, and E = [2, 1, 3] * 65536 maps zq = -1, 0, 1 to multipliers 2, 1, 3.
    R*Cc = -1 floors to -1 (truncation would give 0)."""
    N = 4
    lat = np.array([3, 10, 100, 7], np.int64)
    prob = wfgen.Problem(
        N=N, D=1, M=1, W=1, pred_off=np.array([0, 0, 1, 2, 3], np.int32),
        pred_idx=np.array([0, 1, 2], np.int32), model=np.zeros(N, np.uint8),
        session=np.zeros(N, np.int32), arrival_us=np.zeros(1, np.int64),
        lat_us=lat.astype(np.int32), peak_mib=np.full(N, 11, np.int32),
        weight_mib=np.array([10], np.int32), load_us=np.zeros(1, np.int32),
        cap_mib=np.array([100], np.int32), S=3, seed=77,
        bm_r=np.full(16, r, np.int32), bm_c=np.full(16, c, np.int32),
        bm_e=np.array([2, 1, 3], np.int32) * 65536)
    pl = wfgen.Plans.empty(1, N)
    pl.order[0, :N] = range(N)
    res = oracle.eval_plan(prob, pl, 0)
    assert res["makespan"] == mult * int(lat.sum())
