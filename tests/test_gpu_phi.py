"""Eq. 12's window terms (timely prefetches, lifecycle overhead) and the top-k
by that key: bit-exact against the oracle on every evaluation path."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import THREADS, lib
from randprob import random_problem
from test_gpu_parity import inject_invalid

pytestmark = pytest.mark.gpu


def gpu_phi(prob, plans, k, reclaim=0, int64_path=False):
    import torch
    wf = lib()
    ctx = wf.Ctx(prob, max_P=plans.P)
    if reclaim:
        wf.wf_ctx_set_reclaim(ctx, 1)
    if int64_path:
        wf.wf_ctx_set_eval_path(ctx, wf.PATH_INT64)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    res = wf.Results(plans.P)
    timely = torch.empty(plans.P, dtype=torch.int64, device="cuda")
    life = torch.empty_like(timely)
    wf.wf_eval_plans_phi(ctx, dp, res, timely, life)
    ids = torch.empty(k, dtype=torch.int32, device="cuda")
    keys = torch.empty((k, 3), dtype=torch.int64, device="cuda")
    wf.wf_topk_phi(ctx, res, timely, life, plans.P, k, ids, keys)
    torch.cuda.synchronize()
    wf.wf_ctx_status(ctx)
    mk, p95, gpu, st = res.numpy()
    out = dict(makespan=mk, p95=p95, gpu=gpu, status=st, timely=timely.cpu().numpy(), life=life.cpu().numpy(),
               ids=ids.cpu().numpy(), keys=keys.cpu().numpy())
    ctx.close()
    return out


def check(prob, plans, k, reclaim=0, int64_path=False):
    got = gpu_phi(prob, plans, k, reclaim, int64_path)
    p = prob.with_(reclaim=reclaim)
    mk, p95, gpu, st = oracle.eval_plans(p, plans, threads=THREADS)
    timely, life = oracle.eval_phi(p, plans, threads=THREADS)
    for name, want in (("makespan", mk), ("p95", p95), ("gpu", gpu), ("status", st), ("timely", timely),
                       ("life", life)):
        assert np.array_equal(got[name], want), name
    ids, keys = oracle.topk_phi(mk, timely, life, st, k)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)
    return got


@pytest.mark.parametrize("name", ["tiny", "mix", "burst"])
def test_named_workloads(name):
    w = wfgen.config(name)
    P = min(w.P, 4096)
    plans = wfgen.make_plans(w.problem, P, w.plan_seed)
    got = check(w.problem, plans, k=32)
    assert (got["timely"] > 0).any() and (got["life"] > 0).any()


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("reclaim", [0, 1])
def test_random_windows(seed, reclaim):
    """Invalid plans, retain bits, grants, tight capacities, both
    reclamation orders."""
    rng = np.random.default_rng(8100 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 7)), sizes=(4, 12), D=int(rng.integers(1, 9)),
                          M=int(rng.integers(1, 9)))
    P = int(rng.integers(8, 600))
    plans = wfgen.make_plans(prob, P, seed, p_prefetch=float(rng.uniform(0.2, 1)),
                             p_retain=float(rng.uniform(0.3, 1)) if seed % 2 else None)
    inject_invalid(plans, prob, rng)
    check(prob, plans, k=int(rng.integers(1, min(P, 64) + 1)), reclaim=reclaim)


def test_int64_path():
    w = wfgen.config("mix")
    plans = wfgen.make_plans(w.problem, 1024, 5, p_retain=0.5)
    inject_invalid(plans, w.problem, np.random.default_rng(2))
    check(w.problem, plans, k=16, int64_path=True)


def test_times_beyond_u32():
    """Every makespan beyond 2^32 us: the plans go on from the 32-bit sweep
    to the 64-bit one and the int64 path, which must carry the terms too."""
    rng = np.random.default_rng(31)
    prob = random_problem(rng, n_sessions=5, sizes=(6, 10), D=3, M=3)
    lat = (prob.lat_us.astype(np.int64) % 1000 + (1 << 30) - 5000).astype(np.int32)
    prob = prob.with_(lat_us=lat)
    plans = wfgen.make_plans(prob, 300, 3, p_retain=0.5)
    check(prob, plans, k=10)


def test_large_topk_and_stochastic_refusal():
    """More than 16,384 plans (the multi-CTA top-k); a stochastic window is
    refused."""
    import torch
    w = wfgen.config("mix")
    plans = wfgen.make_plans(w.problem, 20000, 9)
    check(w.problem, plans, k=64)
    wf = lib()
    s = wfgen.config("stochastic")
    ctx = wf.Ctx(s.problem, max_P=8)
    dp = wf.DevicePlans.from_host(wfgen.make_plans(s.problem, 8, 1), "cuda")
    t = torch.empty(8, dtype=torch.int64, device="cuda")
    with pytest.raises(wf.WfError):
        wf.wf_eval_plans_phi(ctx, dp, wf.Results(8), t, torch.empty_like(t))
