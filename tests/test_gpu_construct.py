"""Bit-exact parity of the GPU plan constructor with the oracle's, and the
evaluator reproducing the constructor's timeline."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import lib
from randprob import random_problem

pytestmark = pytest.mark.gpu


def build(prob, P, seed, jitter, plan_base=0, retain=False):
    import torch
    wf = lib()
    ctx = wf.Ctx(prob, max_P=P)
    out = wf.DevicePlans.empty(P, prob.N, with_retain=retain, plan_base=plan_base)
    wf.wf_construct_plans(ctx, out, seed, jitter)
    res = wf.Results(P)
    wf.wf_eval_plans(ctx, out, res)
    torch.cuda.synchronize()
    wf.wf_ctx_status(ctx)
    return out.numpy(prob.N), res.numpy()


def check(prob, got, res, want, ends):
    for a, (g, w) in enumerate(zip(got[:4], (want.place, want.order, want.fuse, want.prefetch))):
        assert np.array_equal(g, w), ("field", a)
    mk, p95, gpu, st = res
    assert (st == 0).all()
    assert np.array_equal(mk, ends - int(np.min(prob.arrival_us)))


@pytest.mark.parametrize("case", range(6))
def test_random_windows(case):
    rng = np.random.default_rng(1500 + case)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 7)), D=int(rng.integers(1, 7)),
                          M=int(rng.integers(1, 7)))
    if case % 2:
        prob = prob.with_(grant_us=int(rng.integers(1, 500)))
    P = int(rng.integers(1, 200))
    jitter = [0, 1, 1000, 10 ** 6, 10 ** 9, 37][case]
    got, res = build(prob, P, seed=case, jitter=jitter, plan_base=17 * case, retain=case == 2)
    want, ends = oracle.construct(prob, P, seed=case, jitter=jitter, plan_base=17 * case)
    check(prob, got, res, want, ends)
    if case == 2:
        N = prob.N
        bits = np.unpackbits(got[4].view(np.uint8), bitorder="little", axis=1)[:, :N]
        assert bits.all() and not np.unpackbits(got[4].view(np.uint8), bitorder="little", axis=1)[:, N:].any()


@pytest.mark.parametrize("jitter", [2, 3, (1 << 40) + 12345, (1 << 46) - 1])
def test_jitter_remainders(jitter):
    """Jitter draws mod (jitter + 1) over the whole 64-bit range of the hash:
    the kernel's reciprocal-multiply remainder against the oracle's %."""
    rng = np.random.default_rng(77)
    prob = random_problem(rng, n_sessions=5, D=4, M=4)
    got, res = build(prob, 64, seed=9, jitter=jitter, plan_base=5)
    want, ends = oracle.construct(prob, 64, seed=9, jitter=jitter, plan_base=5)
    check(prob, got, res, want, ends)


@pytest.mark.parametrize("name,P", [("tiny", 300), ("mix", 200), ("burst", 64), ("large", 8)])
def test_named_workloads(name, P):
    prob = wfgen.config(name).problem
    got, res = build(prob, P, seed=5, jitter=200000, plan_base=3)
    want, ends = oracle.construct(prob, P, seed=5, jitter=200000, plan_base=3)
    check(prob, got, res, want, ends)
