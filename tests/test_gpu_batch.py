"""GPU parity for the replica batch limit B_q (wf_ctx_set_batch): the int64
path's batched play against the oracle's, element by element."""
import numpy as np
import pytest

import oracle
import wfgen
from golden_util import fixture_names, load, plans_of, problem_of
from gpu_util import THREADS, assert_same, gpu_eval, lib, oracle_eval
from randprob import random_problem
from test_gpu_parity import inject_invalid

pytestmark = pytest.mark.gpu


def _gpu(prob, plans, k=None):
    wf = lib()
    ctx = wf.Ctx(prob, max_P=plans.P)  # the context takes prob.batch (wf_ctx_set_batch)
    out = gpu_eval(prob, plans, k=k, ctx=ctx)
    ctx.close()
    return out


@pytest.mark.parametrize("seed", range(8))
def test_random_windows(seed):
    rng = np.random.default_rng(3100 + seed)
    B = [1, 2, 3, 5][seed % 4]
    prob = random_problem(rng, n_sessions=int(rng.integers(2, 7)), D=int(rng.integers(1, 5)),
                          M=int(rng.integers(1, 6)), tight=bool(seed % 2)).with_(batch=B)
    plans = wfgen.make_plans(prob, int(rng.integers(50, 400)), seed, p_retain=0.6 if B == 1 else None)
    inject_invalid(plans, prob, rng)
    got = _gpu(prob, plans, k=8)
    want = oracle_eval(prob, plans)
    assert_same(got, want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], 8)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)


@pytest.mark.parametrize("name", [n for n in fixture_names() if n.startswith(("t10", "t11", "t12"))])
def test_hand_worked_windows(name):
    fx = load(name)
    for case in fx["cases"]:
        prob = problem_of(fx, case)
        plans = plans_of(fx, [case])
        got = _gpu(prob, plans)
        exp = case["expect"]
        assert (int(got["makespan"][0]), int(got["p95"][0]), int(got["gpu"][0])) == \
            (exp["makespan"], exp["p95"], exp["gpu"]), case["label"]


@pytest.mark.parametrize("B", [1, 2, 4])
def test_burst_window_in_full(B):
    w = wfgen.config("burst")
    prob = w.problem.with_(batch=B)
    plans = wfgen.make_plans(prob, w.P, w.plan_seed)
    got = _gpu(prob, plans, k=w.k)
    want = oracle_eval(prob, plans)
    assert_same(got, want)


def test_batch_one_equals_the_sweep():
    """B_q = 1 on the int64 path gives the shared-memory sweep's results."""
    w = wfgen.config("mix")
    plans = wfgen.make_plans(w.problem, 8192, 4)
    a = gpu_eval(w.problem, plans)
    b = _gpu(w.problem.with_(batch=1), plans)
    assert_same(b, a)


def test_refusals():
    wf = lib()
    import torch
    s = wfgen.config("stochastic").problem
    ctx = wf.Ctx(s, max_P=8)
    with pytest.raises(wf.WfError) as e:
        wf.wf_ctx_set_batch(ctx, 2)
    assert e.value.code == wf.WF_EINVAL
    ctx.close()
    w = wfgen.config("tiny")
    ctx = wf.Ctx(w.problem, max_P=16)
    with pytest.raises(wf.WfError):
        wf.wf_ctx_set_batch(ctx, 65)
    wf.wf_ctx_set_batch(ctx, 2)
    with pytest.raises(wf.WfError):
        wf.wf_ctx_set_reclaim(ctx, 1)
    plans = wfgen.make_plans(w.problem, 16, 1, p_retain=0.5)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    res = wf.Results(16)
    with pytest.raises(wf.WfError) as e:
        wf.wf_eval_plans(ctx, dp, res)
    assert "retain" in str(e.value)
    nr = wf.DevicePlans.from_host(wfgen.make_plans(w.problem, 16, 1), "cuda")
    t = torch.empty(16, dtype=torch.int64, device="cuda")
    with pytest.raises(wf.WfError):
        wf.wf_eval_plans_phi(ctx, nr, res, t, torch.empty_like(t))
    wf.wf_eval_plans(ctx, nr, res)  # the context still works
    wf.wf_ctx_status(ctx)
    ctx.close()
