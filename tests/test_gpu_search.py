"""Bit-exact parity of the local search (mutate, merge, rounds) with the oracle."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import lib
from randprob import random_problem

pytestmark = pytest.mark.gpu


def host_rows(dp, N):
    return dp.numpy(N)


def assert_rows(dp, want, N):
    got = dp.numpy(N)
    for a, (g, w) in enumerate(zip(got, (want.place, want.order, want.fuse, want.prefetch, want.retain))):
        if w is None:
            assert g is None
        else:
            assert np.array_equal(g, w), ("row field", a)


def stochastic(prob, S, seed):
    r, c, e = wfgen.box_muller_tables()
    return prob.with_(S=S, seed=seed, bm_r=r, bm_c=c, bm_e=e)


@pytest.mark.parametrize("case", range(5))
def test_mutate_matches_oracle(case):
    import torch
    wf = lib()
    rng = np.random.default_rng(600 + case)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 6)), D=int(rng.integers(1, 6)))
    P = int(rng.integers(1, 40))
    par = wfgen.make_plans(prob, P, case, p_retain=0.5 if case % 2 else None)
    if case == 3:  # invalid parents mutate the same way
        par.order[0, 0] = par.order[0, 1]
        par.place[min(1, P - 1), 0] = 200
    C = int(rng.integers(1, 500))
    n_ops = [0, 1, 3, 9, 40][case]
    ctx = wf.Ctx(prob, max_P=max(P, C))
    dpar = wf.DevicePlans.from_host(par, "cuda")
    dch = wf.DevicePlans.empty(C, prob.N, par.retain is not None)
    wf.wf_mutate_plans(ctx, dpar, dch, seed=12345 + case, round_=case, n_ops=n_ops)
    torch.cuda.synchronize()
    assert_rows(dch, oracle.mutate(prob, par, C, 12345 + case, case, n_ops), prob.N)


def eval_dev(wf, ctx, dp, P):
    import torch
    res = wf.Results(P)
    wf.wf_eval_plans(ctx, dp, res)
    torch.cuda.synchronize()
    return res


def test_merge_matches_oracle():
    import torch
    wf = lib()
    w = wfgen.config("mix")
    prob = w.problem
    for k, C, seed in ((1, 1, 0), (7, 30, 1), (32, 900, 2), (64, 64, 3)):
        elite = wfgen.make_plans(prob, k, 50 + seed)
        ctx = wf.Ctx(prob, max_P=k + C)
        de = wf.DevicePlans.from_host(elite, "cuda")
        er = eval_dev(wf, ctx, de, k)
        dch = wf.DevicePlans.empty(C, prob.N)
        wf.wf_mutate_plans(ctx, de, dch, seed=seed, round_=0, n_ops=2)
        cr = eval_dev(wf, ctx, dch, C)
        want_met = [m.copy() for m in er.numpy()]
        ch_host = oracle.mutate(prob, elite, C, seed, 0, 2)
        pairs, new = oracle.merge_elite(want_met, cr.numpy(), k)
        rows = oracle.PlanRows.copy_of(elite, prob.N)
        for s, c in pairs:
            for a in ("place", "order", "fuse", "prefetch"):
                getattr(rows, a)[s] = getattr(ch_host, a)[c]
        wf.wf_merge_elite(ctx, de, er, dch, cr)
        torch.cuda.synchronize()
        assert_rows(de, rows, prob.N)
        for a, b in zip(er.numpy(), new):
            assert np.array_equal(a, b)


@pytest.mark.parametrize("name,k,C,rounds,n_ops,S", [
    ("tiny", 8, 64, 6, 3, 0),
    ("mix", 16, 512, 3, 2, 0),
    ("burst", 32, 1024, 2, 4, 0),
    ("random", 5, 200, 4, 5, 0),
    ("random_stochastic", 6, 96, 3, 3, 8),
])
def test_local_search_matches_oracle(name, k, C, rounds, n_ops, S):
    import torch
    wf = lib()
    if name.startswith("random"):
        rng = np.random.default_rng(77)
        prob = random_problem(rng, n_sessions=5, D=4)
        if S:
            prob = stochastic(prob, S, 4242)
        elite = wfgen.make_plans(prob, k, 3, p_retain=0.6, plan_base=1000)
    else:
        prob = wfgen.config(name).problem
        elite = wfgen.make_plans(prob, k, 3)
    ctx = wf.Ctx(prob, max_P=k + C)
    de = wf.DevicePlans.from_host(elite, "cuda")
    er = eval_dev(wf, ctx, de, k)
    met0 = [m.copy() for m in er.numpy()]
    dch = wf.DevicePlans.empty(C, prob.N, elite.retain is not None, plan_base=5000)
    cr = wf.Results(C)
    wf.wf_local_search(ctx, de, er, dch, cr, seed=99, round0=10, rounds=rounds, n_ops=n_ops)
    torch.cuda.synchronize()
    rows, met = oracle.local_search(prob, elite, met0, C, 99, 10, rounds, n_ops, children_plan_base=5000,
                                    threads=8)
    assert_rows(de, rows, prob.N)
    for a, b in zip(er.numpy(), met):
        assert np.array_equal(a, b)
    best0 = min(zip(met0[3].tolist(), met0[0].tolist()))
    best1 = min(zip(met[3].tolist(), met[0].tolist()))
    assert best1 <= best0


@pytest.mark.parametrize("N", [3600, 3700, 5000])
@pytest.mark.parametrize("retain", [False, True])
def test_mutate_long_rows(N, retain):
    """Rows on both sides of the staged kernel's limit (eight warps' row sets
    in 96 KB of shared memory; the retain row counts): 3,600 activations are
    staged with and without retain rows, 3,700 only without, 5,000 never."""
    import torch
    from test_gpu_edges import chains_window
    wf = lib()
    prob = chains_window([N // 4] * 4, D=3, M=3, seed=N)
    par = wfgen.make_plans(prob, 7, N, p_retain=0.5 if retain else None)
    C = 300
    ctx = wf.Ctx(prob, max_P=C)
    dpar = wf.DevicePlans.from_host(par, "cuda")
    dch = wf.DevicePlans.empty(C, prob.N, retain)
    wf.wf_mutate_plans(ctx, dpar, dch, seed=99, round_=2, n_ops=5)
    torch.cuda.synchronize()
    assert_rows(dch, oracle.mutate(prob, par, C, 99, 2, 5), prob.N)
