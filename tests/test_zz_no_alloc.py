"""wf_eval_plans_static: the entry point for callers that cannot allocate
device memory (for instance a scheduler inside a serving engine that reserved
almost all GPU memory for weights and KV cache).  Its scratch is the library's
static device array; it must give exactly what the context-based entry point
gives, call after call.  This file is collected last on purpose."""
import numpy as np
import pytest

import wfgen

pytestmark = pytest.mark.gpu


def _both(wf, prob, plans, ctx, dprob):
    import torch
    dp = wf.DevicePlans.from_host(plans, "cuda")
    ref = wf.Results(plans.P)
    wf.wf_eval_plans(ctx, dp, ref)
    got = wf.Results(plans.P)
    wf.wf_eval_plans_static(dprob, dp, got)
    torch.cuda.synchronize()
    return ref.numpy(), got.numpy()


def test_static_entry_matches_context_entry_twice_in_a_row():
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
    ctx1.close()
    ctx2.close()


def test_static_entry_rejects_what_it_cannot_hold():
    from paper_2609_03335_gb300 import build, wf
    build.build()
    w = wfgen.config("burst")
    plans = wfgen.make_plans(w.problem, 4000, 1)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    out = wf.Results(plans.P)
    with pytest.raises(wf.WfError) as e:
        wf.wf_eval_plans_static(wf.DeviceProblem(w.problem), dp, out)
    assert e.value.code == wf.WF_EINVAL and "at most" in str(e.value)
    s = wfgen.config("stochastic").problem
    sp = wfgen.make_plans(s, 8, 1)
    with pytest.raises(wf.WfError) as e:
        wf.wf_eval_plans_static(wf.DeviceProblem(s), wf.DevicePlans.from_host(sp, "cuda"), wf.Results(8))
    assert e.value.code == wf.WF_EINVAL
