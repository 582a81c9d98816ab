"""Edge cases through the C ABI: the largest window, argument errors, padded
rows, and two contexts working on two streams at once."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import assert_same, gpu_eval, lib, oracle_eval
from randprob import random_problem

pytestmark = pytest.mark.gpu


def chains_window(lengths, D=2, M=2, seed=0):
    """Independent chains of the given lengths, one session each (alternating
    models, so nothing is fusible)."""
    rng = np.random.default_rng(seed)
    N = int(sum(lengths))
    n_sessions = len(lengths)
    session = np.repeat(np.arange(n_sessions), lengths).astype(np.int32)
    first = np.r_[0, np.cumsum(lengths)[:-1]]
    pred_off = np.zeros(N + 1, np.int32)
    pred_idx = []
    for v in range(N):
        if v != first[session[v]]:
            pred_idx.append(v - 1)
        pred_off[v + 1] = len(pred_idx)
    model = (np.arange(N) % M).astype(np.uint8)
    lat = rng.integers(1, 1000, N * D).astype(np.int32)
    weight = np.array([2 + m for m in range(M)], np.int32)
    peak = (weight[model].repeat(D) + rng.integers(0, 3, N * D)).astype(np.int32)
    return wfgen.Problem(N=N, D=D, M=M, W=n_sessions, pred_off=pred_off, pred_idx=np.array(pred_idx, np.int32),
                         model=model, session=session,
                         arrival_us=rng.integers(0, 10000, n_sessions).astype(np.int64), lat_us=lat,
                         peak_mib=peak, weight_mib=weight, load_us=rng.integers(1, 100, M * D).astype(np.int32),
                         cap_mib=np.full(D, 12, np.int32))


def test_largest_window():
    """N = 65535, the ABI's limit (beyond the shared-memory sweep, which
    takes N <= 65534; five sessions of 13,107 activations would also need
    more finish-time slots than the sweep holds: the exact int64 path runs)."""
    prob = chains_window([13107] * 5)
    assert prob.N == 65535
    plans = wfgen.make_plans(prob, 3, 1)
    got = gpu_eval(prob, plans, k=2, forecast=True)
    assert_same(got, oracle_eval(prob, plans))
    rel, comp = oracle.forecast(prob)
    assert np.array_equal(got["rel"], rel) and np.array_equal(got["comp"], comp)


def test_largest_sweep_window_and_constructor():
    """N = 65534 in 33 sessions still fits the sweep's 16-bit positions and
    its slots; the constructor's 16-bit node ids cover it too."""
    import torch
    wf = lib()
    prob = chains_window([2047] * 32 + [30], seed=2)
    assert prob.N == 65534
    plans = wfgen.make_plans(prob, 2, 3)
    assert_same(gpu_eval(prob, plans), oracle_eval(prob, plans))
    ctx = wf.Ctx(prob, max_P=2)
    out = wf.DevicePlans.empty(2, prob.N)
    wf.wf_construct_plans(ctx, out, seed=4, jitter_us=100)
    torch.cuda.synchronize()
    want, _ = oracle.construct(prob, 2, seed=4, jitter=100)
    got = out.numpy(prob.N)
    assert np.array_equal(got[0], want.place) and np.array_equal(got[1], want.order)


def test_argument_errors():
    import torch
    wf = lib()
    w = wfgen.config("tiny")
    ctx = wf.Ctx(w.problem, max_P=16)
    plans = wf.DevicePlans.from_host(wfgen.make_plans(w.problem, 16, 0), "cuda")
    res = wf.Results(16)
    with pytest.raises(wf.WfError):
        wf.wf_eval_plans(ctx, plans, res, P=0)
    big = wf.DevicePlans.from_host(wfgen.make_plans(w.problem, 17, 0), "cuda")
    with pytest.raises(wf.WfError):
        wf.wf_eval_plans(ctx, big, wf.Results(17))
    ids = torch.empty(17, dtype=torch.int32, device="cuda")
    wf.wf_eval_plans(ctx, plans, res)
    with pytest.raises(wf.WfError):
        wf.wf_topk(ctx, res, 16, 17, ids)
    odd = wf.DevicePlans(plans.place[:, :12], plans.order, plans.fuse, plans.prefetch)  # stride 16 ok
    wf.wf_eval_plans(ctx, odd, res)
    bad = wf.DevicePlans(plans.place.reshape(-1)[4:4 + 16 * 12].reshape(16, 12), plans.order, plans.fuse,
                         plans.prefetch)  # 12-byte rows: stride not a multiple of 16
    with pytest.raises(wf.WfError):
        wf.wf_eval_plans(ctx, bad, res)
    torch.cuda.synchronize()
    wf.wf_ctx_status(ctx)


def test_padded_rows():
    """Rows with twice the minimal stride give the same results."""
    import torch
    wf = lib()
    w = wfgen.config("mix")
    host = wfgen.make_plans(w.problem, 300, 8)
    dense = wf.DevicePlans.from_host(host, "cuda")

    def widen(t):
        wide = torch.zeros((t.shape[0], 2 * t.shape[1]), dtype=t.dtype, device=t.device)
        wide[:, :t.shape[1]] = t
        return wide[:, :t.shape[1]]
    wide = wf.DevicePlans(widen(dense.place), widen(dense.order), widen(dense.fuse), widen(dense.prefetch))
    assert wide.place.stride(0) == 2 * dense.place.stride(0)
    got = gpu_eval(w.problem, host)
    ctx = wf.Ctx(w.problem, max_P=300)
    res = wf.Results(300)
    wf.wf_eval_plans(ctx, wide, res)
    torch.cuda.synchronize()
    for a, b in zip(res.numpy(), (got["makespan"], got["p95"], got["gpu"], got["status"])):
        assert np.array_equal(a, b)


def test_two_contexts_on_two_streams():
    import torch
    wf = lib()
    jobs = []
    for name, seed in (("burst", 1), ("mix", 2)):
        w = wfgen.config(name)
        host = wfgen.make_plans(w.problem, 2048, seed)
        ctx = wf.Ctx(w.problem, max_P=2048)
        dp = wf.DevicePlans.from_host(host, "cuda")
        jobs.append((w.problem, host, ctx, dp, wf.Results(2048), torch.cuda.Stream()))
    torch.cuda.synchronize()
    for _ in range(3):
        for prob, host, ctx, dp, res, s in jobs:
            with torch.cuda.stream(s):
                wf.wf_eval_plans(ctx, dp, res, s)
    torch.cuda.synchronize()
    for prob, host, ctx, dp, res, s in jobs:
        want = oracle.eval_plans(prob, host, threads=8)
        for a, b in zip(res.numpy(), want):
            assert np.array_equal(a, b)


def fanout_window(F, sessions=3, D=3, M=4, seed=0):
    """Per session a source A, F helpers B_i and F joins C_i with
    predecessors {A, B_i}: every C_i waits on its own accumulator slot, so
    A's write list holds F codes (F = 4 travels in the unit record; F >= 5
    is read by the timing stage from global memory, F > 7 beyond the
    record's 3-bit count)."""
    rng = np.random.default_rng(seed)
    preds, session = [], []
    for w in range(sessions):
        a = len(preds)
        preds.append([])
        preds += [[] for _ in range(F)]
        preds += [[a, a + 1 + i] for i in range(F)]
        session += [w] * (2 * F + 1)
    N = len(preds)
    off = np.zeros(N + 1, np.int32)
    off[1:] = np.cumsum([len(x) for x in preds])
    idx = np.array([y for x in preds for y in x], np.int32)
    weight = rng.integers(2, 5, M).astype(np.int32)
    return wfgen.Problem(N=N, D=D, M=M, W=sessions, pred_off=off, pred_idx=idx,
                         model=rng.integers(0, M, N).astype(np.uint8), session=np.array(session, np.int32),
                         arrival_us=rng.integers(0, 500, sessions).astype(np.int64),
                         lat_us=rng.integers(10, 400, N * D).astype(np.int32),
                         peak_mib=rng.integers(5, 9, N * D).astype(np.int32), weight_mib=weight,
                         load_us=rng.integers(1, 60, M * D).astype(np.int32), cap_mib=np.full(D, 12, np.int32))


@pytest.mark.parametrize("F", [3, 4, 5, 7, 9])
def test_long_write_lists(F):
    """Units that publish their finish to F slots (the sweep's record paths
    for three, four, five to seven and more than seven codes)."""
    prob = fanout_window(F, seed=F)
    plans = wfgen.make_plans(prob, 300, F)
    assert_same(gpu_eval(prob, plans), oracle_eval(prob, plans))


def test_bounded_wait_expiry_is_reported():
    """A device-side wait that nothing completes gives up on its own (in
    about 4 s), the host reads WF_ETIMEOUT from wf_ctx_status, and the
    context evaluates correctly afterwards."""
    import time
    import torch
    wf = lib()
    w = wfgen.config("tiny")
    ctx = wf.Ctx(w.problem, max_P=64)
    t0 = time.perf_counter()
    wf.wf_ctx_check_wait_expiry(ctx)
    with pytest.raises(wf.WfError) as e:
        wf.wf_ctx_status(ctx)
    assert e.value.code == wf.WF_ETIMEOUT
    assert time.perf_counter() - t0 < 30
    wf.wf_ctx_status(ctx)  # cleared
    host = wfgen.make_plans(w.problem, 64, 3)
    plans = wf.DevicePlans.from_host(host, "cuda")
    res = wf.Results(64)
    wf.wf_eval_plans(ctx, plans, res)
    torch.cuda.synchronize()
    wf.wf_ctx_status(ctx)
    for a, b in zip(res.numpy(), oracle.eval_plans(w.problem, host)):
        assert np.array_equal(a, b)


@pytest.mark.parametrize("reclaim", [0, 1])
def test_placement_errors_found_by_the_sweep(reclaim):
    """Placement and fit errors the sweep's producers find (the status pass
    checks only the order of such plans): a fused chain member that does not
    fit its head's device, a device index beyond D, valid plans beside them.
    Under next-use reclamation the status pass checks placement itself."""
    N, D = 15, 2
    prob = chains_window([5, 5, 5], D=D, M=1, seed=9)  # one model: every chain edge is fusible
    peak = np.full((N, D), 3, np.int32)
    peak[2, 0] = peak[7, 0] = 20  # nodes 2 and 7 fit device 1 only
    prob = prob.with_(peak_mib=peak.reshape(-1), cap_mib=np.array([12, 30], np.int32), reclaim=reclaim)
    P = 96
    plans = wfgen.Plans.empty(P, N)
    rng = np.random.default_rng(3)
    for p in range(P):
        nxt, order = [0, 5, 10], []
        while len(order) < N:  # the three chains interleaved in a random order
            c = int(rng.choice([i for i in range(3) if nxt[i] < 5 * i + 5]))
            order.append(nxt[c])
            nxt[c] += 1
        plans.order[p, :N] = order
        place = rng.integers(0, D, size=N)
        if p % 4 == 0:
            place[:] = 0  # whole chains fused on device 0, with members 2 and 7 that do not fit it
        elif p % 4 == 1:
            place[rng.integers(N)] = D + int(rng.integers(0, 200))
        elif p % 4 == 2:
            place[:] = 1
        plans.place[p, :N] = place
        plans.fuse[p, :] = 0xFFFFFFFF
        plans.prefetch[p, :] = rng.integers(0, 2**32, size=plans.prefetch.shape[1], dtype=np.uint64).astype(np.uint32)
    want = oracle_eval(prob, plans)
    assert (want["status"] & 2).any() and (want["status"] & 1).any() and (want["status"] == 0).any()
    assert_same(gpu_eval(prob, plans, k=8), want)
