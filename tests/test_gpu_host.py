"""wf_eval_topk_host: one step of the hot path from and to host memory, through
the C ABI, against the device-pointer calls and the oracle."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import assert_same, gpu_eval, lib, oracle_eval
from randprob import random_problem
from test_gpu_parity import inject_invalid

pytestmark = pytest.mark.gpu


def _host_step(wf, ctx, plans, k, pin=True, forecast=True, with_out=True, stream=None):
    """Issue one call; returns the host buffers it fills (read them after a sync)."""
    import torch
    hp = wf.DevicePlans.host(plans, pin=pin)
    mk = (lambda *shape, dt: torch.empty(shape, dtype=dt).pin_memory()) if pin else \
        (lambda *shape, dt: torch.empty(shape, dtype=dt))
    bufs = {"ids": mk(k, dt=torch.int32), "keys": mk(k, 3, dt=torch.int64), "plans": hp}
    bufs["out"] = wf.Results(plans.P, device="cpu", pin=pin) if with_out else None
    if forecast:
        bufs["rel"], bufs["comp"] = mk(plans.N, dt=torch.int64), mk(plans.N, dt=torch.int64)
    wf.wf_eval_topk_host(ctx, hp, k, bufs["ids"], bufs["keys"], bufs["out"], bufs.get("rel"), bufs.get("comp"),
                         stream)
    return bufs


def _check(bufs, prob, plans, k, want=None):
    want = want or oracle_eval(prob, plans)
    if bufs["out"] is not None:
        mk, p95, gpu, st = bufs["out"].numpy()
        assert_same(dict(makespan=mk, p95=p95, gpu=gpu, status=st), want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], k)
    assert np.array_equal(bufs["ids"].numpy(), ids) and np.array_equal(bufs["keys"].numpy(), keys)
    if "rel" in bufs:
        rel, comp = oracle.forecast(prob)
        assert np.array_equal(bufs["rel"].numpy(), rel) and np.array_equal(bufs["comp"].numpy(), comp)


@pytest.mark.parametrize("seed", range(4))
def test_random_windows_match_oracle_and_device_calls(seed):
    import torch
    wf = lib()
    rng = np.random.default_rng(7100 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(2, 8)), D=int(rng.integers(1, 6)),
                          M=int(rng.integers(1, 6)))
    P = int(rng.integers(20, 500))
    plans = wfgen.make_plans(prob, P, seed, p_retain=0.5 if seed % 2 else None)
    inject_invalid(plans, prob, rng)
    k = int(rng.integers(1, min(P, 40) + 1))
    ctx = wf.Ctx(prob, max_P=P + 17)
    bufs = _host_step(wf, ctx, plans, k)
    torch.cuda.synchronize()
    want = oracle_eval(prob, plans)
    _check(bufs, prob, plans, k, want)
    dev = gpu_eval(prob, plans, k=k)
    assert np.array_equal(bufs["ids"].numpy(), dev["ids"])
    ctx.close()


def test_back_to_back_calls_alternate_slots():
    """Four batches issued without a synchronisation between them: each call's
    copy runs while the previous call evaluates, in the other staging slot."""
    import torch
    wf = lib()
    w = wfgen.config("mix")
    batches = [wfgen.make_plans(w.problem, 6000, 40 + i) for i in range(4)]
    ctx = wf.Ctx(w.problem, max_P=6000)
    wf.wf_ctx_reserve_host(ctx)
    stream = torch.cuda.Stream()
    issued = [_host_step(wf, ctx, b, 16, forecast=i == 0, stream=stream) for i, b in enumerate(batches)]
    torch.cuda.synchronize()
    for b, bufs in zip(batches, issued):
        _check(bufs, w.problem, b, 16)
    ctx.close()


def test_pageable_host_memory_and_no_optional_outputs():
    import torch
    wf = lib()
    w = wfgen.config("tiny")
    plans = wfgen.make_plans(w.problem, 700, 3, p_retain=0.6)
    ctx = wf.Ctx(w.problem, max_P=700)
    bufs = _host_step(wf, ctx, plans, 9, pin=False, forecast=False, with_out=False)
    torch.cuda.synchronize()
    _check(bufs, w.problem, plans, 9)
    ctx.close()


def test_wider_host_strides():
    """Host rows padded beyond the staged row size take the row-by-row copy."""
    import torch
    wf = lib()
    rng = np.random.default_rng(77)
    prob = random_problem(rng, n_sessions=5, D=4, M=3)
    plans = wfgen.make_plans(prob, 300, 2, p_retain=0.5)
    hp = wf.DevicePlans.host(plans)

    def widen(t):
        w = torch.zeros((t.shape[0], t.shape[1] + 16 // t.element_size()), dtype=t.dtype).pin_memory()
        w[:, :t.shape[1]] = t
        return w[:, :t.shape[1]]
    wide = wf.DevicePlans(widen(hp.place), widen(hp.order), widen(hp.fuse), widen(hp.prefetch), widen(hp.retain))
    assert wide.place.stride(0) == hp.place.stride(0) + 16
    ctx = wf.Ctx(prob, max_P=300)
    ids = torch.empty(7, dtype=torch.int32).pin_memory()
    keys = torch.empty((7, 3), dtype=torch.int64).pin_memory()
    out = wf.Results(300, device="cpu")
    wf.wf_eval_topk_host(ctx, wide, 7, ids, keys, out)
    torch.cuda.synchronize()
    _check({"ids": ids, "keys": keys, "out": out}, prob, plans, 7)
    ctx.close()


def test_burst_window_in_full():
    """The headline batch (16,384 plans), and a second call on the same context."""
    import torch
    wf = lib()
    w = wfgen.config("burst")
    plans = wfgen.make_plans(w.problem, w.P, w.plan_seed)
    want = oracle_eval(w.problem, plans)
    ctx = wf.Ctx(w.problem, max_P=w.P)
    for _ in range(2):
        bufs = _host_step(wf, ctx, plans, w.k)
        torch.cuda.synchronize()
        _check(bufs, w.problem, plans, w.k, want)
    ctx.close()


def test_stochastic_window():
    import torch
    wf = lib()
    w = wfgen.config("stochastic")
    plans = wfgen.make_plans(w.problem, 512, 5)
    ctx = wf.Ctx(w.problem, max_P=512)
    bufs = _host_step(wf, ctx, plans, 8)
    torch.cuda.synchronize()
    _check(bufs, w.problem, plans, 8)
    ctx.close()


def test_refusals():
    import torch
    wf = lib()
    w = wfgen.config("tiny")
    plans = wfgen.make_plans(w.problem, 32, 1)
    ctx = wf.Ctx(w.problem, max_P=32)
    hp = wf.DevicePlans.host(plans)
    ids = torch.empty(64, dtype=torch.int32).pin_memory()
    rel = torch.empty(w.problem.N, dtype=torch.int64)
    for args in ((hp, 0, ids, None, None, None, None), (hp, 33, ids, None, None, None, None),
                 (hp, 4, ids, None, None, rel, None)):
        with pytest.raises(wf.WfError) as e:
            wf.wf_eval_topk_host(ctx, *args)
        assert e.value.code == wf.WF_EINVAL
    big = wfgen.make_plans(w.problem, 33, 1)
    with pytest.raises(wf.WfError):
        wf.wf_eval_topk_host(ctx, wf.DevicePlans.host(big), 4, ids)
    bufs = _host_step(wf, ctx, plans, 4)  # the context still works
    torch.cuda.synchronize()
    _check(bufs, w.problem, plans, 4)
    ctx.close()
