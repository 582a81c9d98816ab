"""wf_eval_plans_static: the entry point for callers that cannot allocate
device memory (for instance a scheduler inside a serving engine that reserved
almost all GPU memory for weights and KV cache).  Its scratch is the library's
static device array; it must give exactly what the context-based entry point
and the CPU oracle give, call after call, without allocating.  This file is
collected last on purpose."""
import re

import numpy as np
import pytest

import oracle
import wfgen

pytestmark = pytest.mark.gpu


def _both(wf, prob, plans, ctx, dprob):
    import torch
    dp = wf.DevicePlans.from_host(plans, "cuda")
    ref = wf.Results(plans.P)
    wf.wf_eval_plans(ctx, dp, ref)
    got = wf.Results(plans.P)
    wf.wf_eval_plans_static(dprob, dp, got)
    wf.wf_static_status()
    torch.cuda.synchronize()
    return ref.numpy(), got.numpy()


def test_static_entry_matches_context_entry_and_oracle_twice_in_a_row():
    from paper_2609_03335_gb300 import build, wf
    build.build()
    # call 1: the burst window, 1500 plans with some invalid ones
    w1 = wfgen.config("burst")
    p1 = wfgen.make_plans(w1.problem, 1500, 11)
    p1.place[3, 7] = w1.problem.D
    p1.order[9, 0] = p1.order[9, 1]
    ctx1 = wf.Ctx(w1.problem, max_P=p1.P)
    ref1, got1 = _both(wf, w1.problem, p1, ctx1, wf.DeviceProblem(w1.problem))
    # call 2 right after: another window and retain bits
    w2 = wfgen.config("mix")
    p2 = wfgen.make_plans(w2.problem, 5000, 12, p_retain=0.6)
    ctx2 = wf.Ctx(w2.problem, max_P=p2.P)
    ref2, got2 = _both(wf, w2.problem, p2, ctx2, wf.DeviceProblem(w2.problem))
    for ref, got in ((ref1, got1), (ref2, got2)):
        for a, b in zip(ref, got):
            assert np.array_equal(a, b)
    assert got1[3][3] != 0 and got1[3][9] != 0
    # the oracle on a sample of each batch
    for prob, plans, got in ((w1.problem, p1, got1), (w2.problem, p2, got2)):
        sub = plans.slice(0, 300)
        want = oracle.eval_plans(prob, sub)
        for a, b in zip(got, want):
            assert np.array_equal(a[:300], b)
    ctx1.close()
    ctx2.close()


def test_static_entry_allocates_nothing():
    import torch
    from paper_2609_03335_gb300 import build, wf
    build.build()
    w = wfgen.config("mix")
    plans = wfgen.make_plans(w.problem, 2000, 5)
    dprob = wf.DeviceProblem(w.problem)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    out = wf.Results(plans.P)
    wf.wf_eval_plans_static(dprob, dp, out)  # the first call loads the module and looks the array up
    wf.wf_static_status()
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    wf.wf_eval_plans_static(dprob, dp, out)
    wf.wf_static_status()
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_static_entry_accepts_exactly_the_largest_batch_it_names():
    import torch
    from paper_2609_03335_gb300 import build, wf
    build.build()
    w = wfgen.config("burst")
    plans = wfgen.make_plans(w.problem, 4000, 1)
    dprob = wf.DeviceProblem(w.problem)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    out = wf.Results(plans.P)
    with pytest.raises(wf.WfError) as e:
        wf.wf_eval_plans_static(dprob, dp, out)
    assert e.value.code == wf.WF_EINVAL and "at most" in str(e.value)
    fit = int(re.search(r"at most (\d+) plans", str(e.value)).group(1))
    assert 1000 < fit < plans.P
    wf.wf_eval_plans_static(dprob, wf.DevicePlans.from_host(plans.slice(0, fit), "cuda"), wf.Results(fit))
    wf.wf_static_status()
    torch.cuda.synchronize()
    with pytest.raises(wf.WfError) as e:
        wf.wf_eval_plans_static(dprob, wf.DevicePlans.from_host(plans.slice(0, fit + 1), "cuda"),
                                wf.Results(fit + 1))
    assert e.value.code == wf.WF_EINVAL
    s = wfgen.config("stochastic").problem
    sp = wfgen.make_plans(s, 8, 1)
    with pytest.raises(wf.WfError) as e:
        wf.wf_eval_plans_static(wf.DeviceProblem(s), wf.DevicePlans.from_host(sp, "cuda"), wf.Results(8))
    assert e.value.code == wf.WF_EINVAL


def test_static_entry_reports_tables_that_fail_its_device_check():
    """A model id >= M in the device tables: the device check catches it before
    any table is indexed by it; every plan gets WF_ST_TABLES and INT64_MAX, and
    wf_static_status names the failure.  The next good call is clean."""
    import torch
    from paper_2609_03335_gb300 import build, wf
    build.build()
    w = wfgen.config("tiny")
    plans = wfgen.make_plans(w.problem, 64, 3)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    bad = wf.DeviceProblem(w.problem)
    bad.tensors["model"][5] = w.problem.M  # in bounds of the array; out of the model range
    out = wf.Results(plans.P)
    wf.wf_eval_plans_static(bad, dp, out)
    with pytest.raises(wf.WfError) as e:
        wf.wf_static_status()
    assert e.value.code == wf.WF_EINVAL and "model id" in str(e.value)
    mk, p95, gpu, st = out.numpy()
    assert (st == wf.ST_TABLES).all() and (mk == wf.INT64_MAX).all() and (gpu == wf.INT64_MAX).all()
    good = wf.DeviceProblem(w.problem)
    wf.wf_eval_plans_static(good, dp, out)
    wf.wf_static_status()
    torch.cuda.synchronize()
    want = oracle.eval_plans(w.problem, plans)
    for a, b in zip(out.numpy(), want):
        assert np.array_equal(a, b)
