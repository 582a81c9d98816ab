"""Bit-exact parity of reclamation by next use with the oracle."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import assert_same, gpu_eval, lib, oracle_eval
from randprob import random_problem

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,P", [("tiny", 1024), ("mix", 4096), ("burst", 2048)])
def test_named_workloads(name, P):
    w = wfgen.config(name)
    prob = w.problem.with_(reclaim=1)
    plans = wfgen.make_plans(prob, P, w.plan_seed)
    got = gpu_eval(prob, plans, k=16)
    want = oracle_eval(prob, plans)
    assert_same(got, want)
    lru = oracle_eval(w.problem, plans)
    assert not np.array_equal(want["makespan"], lru["makespan"]) or name == "tiny"


@pytest.mark.parametrize("seed", range(6))
def test_random_windows(seed):
    rng = np.random.default_rng(3100 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 7)), D=int(rng.integers(1, 6)),
                          M=int(rng.integers(2, 16 if seed == 5 else 8))).with_(reclaim=1)
    if seed % 2:
        prob = prob.with_(grant_us=int(rng.integers(1, 300)))
    plans = wfgen.make_plans(prob, int(rng.integers(1, 400)), seed, p_retain=0.5 if seed % 3 else None)
    from test_gpu_parity import inject_invalid
    if plans.P >= 8:
        inject_invalid(plans, prob, rng)
    assert_same(gpu_eval(prob, plans), oracle_eval(prob, plans))


def test_overflowing_times_keep_the_policy():
    """Times beyond 2^32 us move plans to the 64-bit sweep, which applies the
    same reclamation order."""
    rng = np.random.default_rng(53)
    prob = random_problem(rng, n_sessions=5, sizes=(6, 10), D=2, M=4)
    lat = prob.lat_us.astype(np.int64).reshape(prob.N, prob.D)
    lat[:2, 1] = (1 << 31) - 1
    prob = prob.with_(lat_us=lat.astype(np.int32).reshape(-1), reclaim=1)
    plans = wfgen.make_plans(prob, 300, 7)
    want = oracle_eval(prob, plans)
    mk = want["makespan"][want["status"] == 0]
    assert (mk >= (1 << 32)).any() and (mk < (1 << 31)).any()
    assert_same(gpu_eval(prob, plans), want)


def test_policy_switch_on_one_context():
    import torch
    wf = lib()
    w = wfgen.config("mix")
    plans = wfgen.make_plans(w.problem, 512, 3)
    ctx = wf.Ctx(w.problem, max_P=512)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    outs = []
    for pol in (0, 1, 0, 1):
        wf.wf_ctx_set_reclaim(ctx, pol)
        res = wf.Results(512)
        wf.wf_eval_plans(ctx, dp, res)
        torch.cuda.synchronize()
        outs.append(res.numpy())
    for a, b in zip(outs[0], outs[2]):
        assert np.array_equal(a, b)
    for a, b in zip(outs[1], outs[3]):
        assert np.array_equal(a, b)
    want = oracle.eval_plans(w.problem.with_(reclaim=1), plans, threads=8)
    assert np.array_equal(outs[1][0], want[0]) and np.array_equal(outs[1][2], want[2])


def test_stochastic_problems_refuse_the_policy():
    wf = lib()
    w = wfgen.config("stochastic")
    ctx = wf.Ctx(w.problem, max_P=8)
    with pytest.raises(wf.WfError):
        wf.wf_ctx_set_reclaim(ctx, 1)
