"""A forecast -> eval -> top-k step captured into a CUDA graph and replayed
gives the same results as direct calls (the library only launches on the
caller's stream while capturing, and skips its path-choice read-back)."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import lib

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["mix", "burst", "stochastic"])
def test_captured_step_replays(name):
    import torch
    wf = lib()
    w = wfgen.config(name)
    P = min(w.P, 4096)
    plans = wfgen.make_plans(w.problem, P, w.plan_seed)
    ctx = wf.Ctx(w.problem, max_P=P)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    res = wf.Results(P)
    rel = torch.empty(w.problem.N, dtype=torch.int64, device="cuda")
    comp = torch.empty_like(rel)
    ids = torch.empty(w.k, dtype=torch.int32, device="cuda")
    keys = torch.empty((w.k, 3), dtype=torch.int64, device="cuda")
    s = torch.cuda.Stream()

    def step():
        wf.wf_forecast_readiness(ctx, rel, comp, s)
        wf.wf_eval_plans(ctx, dp, res, s)
        wf.wf_topk(ctx, res, P, w.k, ids, keys, s)

    with torch.cuda.stream(s):
        step()  # warm-up outside the capture (attributes, first launches)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        step()
    for t in (res.makespan, res.p95, res.gpu, res.status, ids, keys, rel, comp):
        t.fill_(-1)
    g.replay()
    torch.cuda.synchronize()
    wf.wf_ctx_status(ctx)
    mk, p95, gpu, st = oracle.eval_plans(w.problem, plans, threads=8)
    got = res.numpy()
    assert np.array_equal(got[0], mk) and np.array_equal(got[1], p95)
    assert np.array_equal(got[2], gpu) and np.array_equal(got[3], st)
    want_ids, want_keys = oracle.topk(mk, p95, gpu, st, w.k)
    assert np.array_equal(ids.cpu().numpy(), want_ids) and np.array_equal(keys.cpu().numpy(), want_keys)
    r, c = oracle.forecast(w.problem)
    assert np.array_equal(rel.cpu().numpy(), r) and np.array_equal(comp.cpu().numpy(), c)
    # replay again on new plans copied into the same buffers
    plans2 = wfgen.make_plans(w.problem, P, w.plan_seed + 1)
    d2 = wf.DevicePlans.from_host(plans2, "cuda")
    for a in ("place", "order", "fuse", "prefetch"):
        getattr(dp, a).copy_(getattr(d2, a))
    g.replay()
    torch.cuda.synchronize()
    mk2 = oracle.eval_plans(w.problem, plans2, threads=8)[0]
    assert np.array_equal(res.makespan.cpu().numpy(), mk2)
