"""Helpers for the GPU parity tests: run the CUDA path through the C ABI."""
import os

import numpy as np

import oracle

THREADS = min(32, os.cpu_count() or 1)


def lib():
    from paper_2609_03335_gb300 import build, wf
    build.build()
    wf.load_library()
    return wf


def gpu_eval(prob, plans, k=None, ctx=None, forecast=False, int64_path=False):
    """Evaluate on cuda:0 through the C ABI; returns a dict of numpy arrays.
    int64_path: every plan on the exact int64 path (wf_ctx_set_eval_path)."""
    import torch
    wf = lib()
    dev = torch.device("cuda", 0)
    own = ctx is None
    ctx = ctx or wf.Ctx(prob, max_P=plans.P, device=0)
    if int64_path:
        wf.wf_ctx_set_eval_path(ctx, wf.PATH_INT64)
    dp = wf.DevicePlans.from_host(plans, dev)
    res = wf.Results(plans.P, dev)
    wf.wf_eval_plans(ctx, dp, res)
    out = {}
    if k is not None:
        ids = torch.empty(k, dtype=torch.int32, device=dev)
        keys = torch.empty((k, 3), dtype=torch.int64, device=dev)
        wf.wf_topk(ctx, res, plans.P, k, ids, keys)
        out["ids"], out["keys"] = ids.cpu().numpy(), keys.cpu().numpy()
    if forecast:
        rel = torch.empty(prob.N, dtype=torch.int64, device=dev)
        comp = torch.empty_like(rel)
        wf.wf_forecast_readiness(ctx, rel, comp)
        out["rel"], out["comp"] = rel.cpu().numpy(), comp.cpu().numpy()
    wf.wf_ctx_status(ctx)
    out["makespan"], out["p95"], out["gpu"], out["status"] = res.numpy()
    if own:
        ctx.close()
    return out


def oracle_eval(prob, plans, lo=0, hi=None):
    mk, p95, gpu, st = oracle.eval_plans(prob, plans, lo, hi, threads=THREADS)
    return dict(makespan=mk, p95=p95, gpu=gpu, status=st)


def assert_same(got, want, sl=slice(None)):
    for name in ("status", "makespan", "p95", "gpu"):
        g = np.asarray(got[name])[sl].astype(np.int64)
        w = np.asarray(want[name]).astype(np.int64)
        bad = np.nonzero(g != w)[0]
        assert bad.size == 0, (f"{name}: {bad.size} plans differ, first at {bad[:5]}: "
                               f"gpu {g[bad[:5]]} oracle {w[bad[:5]]}")
