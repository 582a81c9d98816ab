"""Bit-exact parity of the CUDA path (through the C ABI) with the CPU oracle.

Every quantity is an integer, so every comparison is exact equality.
"""
import numpy as np
import pytest

import oracle
import wfgen
from golden_util import fixture_names, load, plans_of, problem_of
from gpu_util import assert_same, gpu_eval, lib, oracle_eval
from randprob import random_problem

pytestmark = pytest.mark.gpu


def inject_invalid(plans, prob, rng, frac=0.1):
    """Corrupt a fraction of the plans in every way the status bits name."""
    N, D = prob.N, prob.D
    fits = prob.fits()
    P = plans.P
    idx = rng.choice(P, size=max(4, int(frac * P)), replace=False)
    for j, p in enumerate(idx):
        kind = j % 5
        if kind == 0:
            plans.place[p, rng.integers(N)] = D + rng.integers(0, 255 - D + 1)
        elif kind == 1:
            bad = np.argwhere(~fits)
            if len(bad):
                n, d = bad[rng.integers(len(bad))]
                plans.place[p, n] = d
        elif kind == 2:
            i, j2 = rng.choice(N, size=2, replace=N < 2)
            plans.order[p, i] = plans.order[p, j2]
        elif kind == 3:
            plans.order[p, rng.integers(N)] = N + rng.integers(0, 65535 - N + 1)
        else:
            # swap a node with its predecessor's position (against an edge)
            v = int(rng.choice(np.nonzero(np.diff(prob.pred_off) > 0)[0]))
            u = int(prob.pred_idx[prob.pred_off[v]])
            pos = np.empty(N, int)
            pos[plans.order[p, :N]] = np.arange(N)
            plans.order[p, pos[u]], plans.order[p, pos[v]] = v, u
    return idx


@pytest.mark.parametrize("name", ["tiny", "mix", "burst"])
def test_named_workload_full_parity(name):
    w = wfgen.config(name)
    plans = wfgen.make_plans(w.problem, w.P, w.plan_seed)
    got = gpu_eval(w.problem, plans, k=w.k, forecast=True)
    want = oracle_eval(w.problem, plans)
    assert_same(got, want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], w.k)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)
    rel, comp = oracle.forecast(w.problem)
    assert np.array_equal(got["rel"], rel) and np.array_equal(got["comp"], comp)


def test_stochastic_workload_full_parity():
    w = wfgen.config("stochastic")
    plans = wfgen.make_plans(w.problem, w.P, w.plan_seed)
    got = gpu_eval(w.problem, plans, k=w.k)
    want = oracle_eval(w.problem, plans)
    assert_same(got, want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], w.k)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)


def test_large_window_parity():
    """Full size (P=131072, N=8192, D=16); the oracle checks every plan.  Two
    calls on one context: the first plays the 32-bit sweep and hands every
    plan to the 64-bit one; once that count has arrived, later calls start
    with the 64-bit sweep over the whole batch, the launch the bench times."""
    w = wfgen.config("large")
    plans = wfgen.make_plans(w.problem, w.P, w.plan_seed)
    want = oracle_eval(w.problem, plans)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], w.k)
    ctx = lib().Ctx(w.problem, max_P=plans.P, device=0)
    for call in range(2):
        got = gpu_eval(w.problem, plans, k=w.k, ctx=ctx, forecast=call == 0)
        assert_same(got, want)
        assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)
        if call == 0:
            rel, comp = oracle.forecast(w.problem)
            assert np.array_equal(got["rel"], rel) and np.array_equal(got["comp"], comp)
    ctx.close()


@pytest.mark.parametrize("name", fixture_names())
def test_golden_windows_on_gpu(name):
    fx = load(name)
    for case in fx["cases"]:
        prob = problem_of(fx, case)
        plans = plans_of(fx, [case])
        got = gpu_eval(prob, plans)
        exp = case["expect"]
        assert got["status"][0] == exp["status"], case["label"]
        if exp["status"] == 0:
            assert (got["makespan"][0], got["p95"][0], got["gpu"][0]) == \
                (exp["makespan"], exp["p95"], exp["gpu"]), case["label"]


@pytest.mark.parametrize("seed", range(8))
def test_random_windows_with_invalid_plans_retain_and_grant(seed):
    rng = np.random.default_rng(4000 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 9)), sizes=(4, 12),
                          D=int(rng.integers(1, 9)), M=int(rng.integers(1, 9)))
    P = int(rng.integers(1, 700))
    plans = wfgen.make_plans(prob, P, seed, p_fuse=float(rng.uniform(0, 1)),
                             p_prefetch=float(rng.uniform(0, 1)),
                             p_retain=float(rng.uniform(0.3, 1)) if seed % 2 else None)
    if P >= 8:
        inject_invalid(plans, prob, rng)
    k = int(rng.integers(1, min(P, 64) + 1))
    got = gpu_eval(prob, plans, k=k, forecast=True)
    want = oracle_eval(prob, plans)
    assert_same(got, want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], k)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)
    rel, comp = oracle.forecast(prob)
    assert np.array_equal(got["rel"], rel) and np.array_equal(got["comp"], comp)


@pytest.mark.parametrize("seed", range(10))
def test_random_device_and_model_counts(seed):
    """Device counts 1-32 and model counts 1-16 (so residency lanes own one to
    eight devices, queues of 32 or 64 bits), with retain bits, grant and
    admission margin, and both reclamation policies."""
    rng = np.random.default_rng(5200 + seed)
    D, M = int(rng.integers(1, 33)), int(rng.integers(1, 17))
    prob = random_problem(rng, n_sessions=int(rng.integers(2, 10)), sizes=(4, 12), D=D, M=M)
    prob = prob.with_(grant_us=int(rng.integers(0, 300)), margin_mib=int(rng.integers(0, 3)),
                      reclaim=int(seed % 3 == 2))
    if not prob.fits().any(axis=1).all():  # every activation must fit somewhere
        prob = prob.with_(margin_mib=0)
    P = int(rng.integers(50, 600))
    plans = wfgen.make_plans(prob, P, seed, p_fuse=float(rng.uniform(0, 1)),
                             p_prefetch=float(rng.uniform(0, 1)),
                             p_retain=float(rng.uniform(0.3, 1)) if seed % 2 else None)
    assert_same(gpu_eval(prob, plans, k=min(P, 8)), oracle_eval(prob, plans))


@pytest.mark.parametrize("seed", range(3))
def test_random_stochastic_windows(seed):
    rng = np.random.default_rng(4100 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 6)), D=int(rng.integers(1, 6)))
    r, c, e = wfgen.box_muller_tables()
    prob = prob.with_(S=int(rng.integers(1, 100)), seed=int(rng.integers(0, 2**63)), bm_r=r, bm_c=c, bm_e=e)
    plans = wfgen.make_plans(prob, int(rng.integers(1, 300)), seed, plan_base=int(rng.integers(0, 10**6)),
                             p_retain=0.7 if seed % 2 else None)
    if plans.P >= 8:
        inject_invalid(plans, prob, rng)
    got = gpu_eval(prob, plans)
    assert_same(got, oracle_eval(prob, plans))


@pytest.mark.parametrize("S", [1, 2, 31, 63, 64, 65])
def test_stochastic_sample_counts(S):
    """Sample counts around the width of the per-plan sample block (64 lanes)
    and beyond it (the int64 path evaluates S > 64)."""
    rng = np.random.default_rng(4200 + S)
    prob = random_problem(rng, n_sessions=4, D=3)
    r, c, e = wfgen.box_muller_tables()
    prob = prob.with_(S=S, seed=int(rng.integers(0, 2**63)), bm_r=r, bm_c=c, bm_e=e)
    plans = wfgen.make_plans(prob, 200, S, plan_base=int(rng.integers(0, 10**6)), p_retain=0.6)
    inject_invalid(plans, prob, rng)
    got = gpu_eval(prob, plans, k=7)
    want = oracle_eval(prob, plans)
    assert_same(got, want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], 7)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)


def test_stochastic_int64_path_matches_oracle():
    """The per-sample int64 path on its own, forced for every plan."""
    w = wfgen.config("stochastic")
    plans = wfgen.make_plans(w.problem, 512, 91, p_retain=0.5)
    inject_invalid(plans, w.problem, np.random.default_rng(2))
    got = gpu_eval(w.problem, plans, k=8, int64_path=True)
    assert_same(got, oracle_eval(w.problem, plans))


def test_stochastic_mixed_overflow_batch():
    """Sampled times beyond 2^32 us for some plans (two activations are very
    slow on device 1), within it for the others: the plans that overflow go to
    the int64 path."""
    rng = np.random.default_rng(41)
    prob = random_problem(rng, n_sessions=4, sizes=(5, 9), D=2, M=3)
    lat = prob.lat_us.astype(np.int64).reshape(prob.N, prob.D)
    lat[:2, 1] = (1 << 31) - 1
    r, c, e = wfgen.box_muller_tables()
    prob = prob.with_(lat_us=lat.astype(np.int32).reshape(-1),
                      peak_mib=np.minimum(prob.peak_mib, prob.cap_mib.min()).astype(np.int32)
                      .clip(min=prob.weight_mib[prob.model].repeat(prob.D)),
                      S=16, seed=99, bm_r=r, bm_c=c, bm_e=e)
    plans = wfgen.make_plans(prob, 400, 6)
    got = gpu_eval(prob, plans, k=5)
    want = oracle_eval(prob, plans)
    mk = want["makespan"][want["status"] == 0]
    assert (mk >= (1 << 32)).any() and (mk < (1 << 31)).any()
    assert_same(got, want)


def test_ties_break_by_plan_index():
    w = wfgen.config("tiny")
    base = wfgen.make_plans(w.problem, 64, 3)
    plans = wfgen.Plans.empty(256, w.problem.N)
    for a in ("place", "order", "fuse", "prefetch"):
        getattr(plans, a)[:] = np.tile(getattr(base, a), (4, 1))
    got = gpu_eval(w.problem, plans, k=40)
    want = oracle_eval(w.problem, plans)
    assert_same(got, want)
    ids, _ = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], 40)
    assert np.array_equal(got["ids"], ids)


def test_sub_batches_reproduce_the_batch():
    """Evaluating row ranges with an offset equals evaluating the whole batch."""
    import torch
    from gpu_util import lib
    wf = lib()
    w = wfgen.config("mix")
    plans = wfgen.make_plans(w.problem, 3000, 5, p_retain=0.5)
    ctx = wf.Ctx(w.problem, max_P=3000)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    whole = wf.Results(3000)
    wf.wf_eval_plans(ctx, dp, whole)
    parts = wf.Results(3000)
    for lo, hi in ((0, 1), (1, 1000), (1000, 2999), (2999, 3000)):
        wf.wf_eval_plans(ctx, dp, parts, P=hi - lo, offset=lo)
    torch.cuda.synchronize()
    for a, b in zip(whole.numpy(), parts.numpy()):
        assert np.array_equal(a, b)


def test_single_node_and_extreme_shapes():
    rng = np.random.default_rng(17)
    one = wfgen.Problem(N=1, D=1, M=1, W=1, pred_off=np.zeros(2, np.int32),
                        pred_idx=np.zeros(0, np.int32), model=np.zeros(1, np.uint8),
                        session=np.zeros(1, np.int32), arrival_us=np.array([5], np.int64),
                        lat_us=np.array([7], np.int32), peak_mib=np.array([3], np.int32),
                        weight_mib=np.array([2], np.int32), load_us=np.array([11], np.int32),
                        cap_mib=np.array([4], np.int32), grant_us=1)
    plans = wfgen.make_plans(one, 3, 0)
    got = gpu_eval(one, plans, k=3)
    assert got["makespan"].tolist() == [19, 19, 19]  # load 11 + grant 1 + run 7
    assert got["ids"].tolist() == [0, 1, 2]
    # 32 devices, 16 models, tight memory
    prob = random_problem(rng, n_sessions=12, sizes=(6, 14), D=32, M=16)
    plans = wfgen.make_plans(prob, 777, 1, p_retain=0.5)
    got = gpu_eval(prob, plans, k=1)
    assert_same(got, oracle_eval(prob, plans))


def test_long_chain_window():
    """A 20000-activation window (chains of one model, heavy fusion)."""
    N = 20000
    n_sess = 40
    sizes = wfgen.split_sizes(N, n_sess)
    sess = [wfgen.fam_softdev(s) for s in sizes]
    rng = np.random.default_rng(23)
    prob = wfgen.assemble("long", sess, np.zeros(n_sess, np.int64), wfgen.DEV_BURST,
                          [3, 6, 8, 14], rng)
    plans = wfgen.make_plans(prob, 512, 2, p_fuse=0.9)
    got = gpu_eval(prob, plans, k=16, forecast=True)  # beyond the shared-memory forecast
    want = oracle_eval(prob, plans)
    assert_same(got, want)
    ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], 16)
    assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)
    rel, comp = oracle.forecast(prob)
    assert np.array_equal(got["rel"], rel) and np.array_equal(got["comp"], comp)


@pytest.mark.parametrize("name", ["mix", "burst"])
def test_int64_path_matches_oracle(name):
    """The exact int64 path (taken for plans whose times overflow the
    shared-memory sweep's u32 slots) on its own, forced for every plan."""
    w = wfgen.config(name)
    plans = wfgen.make_plans(w.problem, 2048, 77, p_retain=0.5)
    inject_invalid(plans, w.problem, np.random.default_rng(1))
    got = gpu_eval(w.problem, plans, k=8, int64_path=True)
    assert_same(got, oracle_eval(w.problem, plans))


def _eval_on_path(prob, plans, k, path):
    wf = lib()
    ctx = wf.Ctx(prob, max_P=plans.P)
    if path != "auto":
        wf.wf_ctx_set_eval_path(ctx, wf.PATH_RELATIVE if path == "relative" else wf.PATH_WIDE)
    got = gpu_eval(prob, plans, k=k, ctx=ctx)
    ctx.close()
    return got


@pytest.mark.parametrize("path", ["auto", "wide", "relative"])
def test_times_beyond_u32_take_the_int64_path(path):
    """Run times near 2^30 us make every makespan exceed 2^32 us; those plans
    must still match the oracle exactly, started in any sweep."""
    rng = np.random.default_rng(31)
    prob = random_problem(rng, n_sessions=5, sizes=(6, 10), D=3, M=3)
    lat = (prob.lat_us.astype(np.int64) % 1000 + (1 << 30) - 5000).astype(np.int32)
    prob = prob.with_(lat_us=lat)
    plans = wfgen.make_plans(prob, 300, 3, p_retain=0.5)
    got = _eval_on_path(prob, plans, 10, path)
    want = oracle_eval(prob, plans)
    assert (want["makespan"][want["status"] == 0] >= (1 << 32)).all()
    assert_same(got, want)


@pytest.mark.parametrize("path", ["auto", "wide", "relative"])
def test_fused_run_time_beyond_u32(path):
    """Fused chains of near-2^31 us members: a unit's summed run time alone
    leaves 32 bits, with a start of 0 on some plans; started in any sweep."""
    rng = np.random.default_rng(43)
    prob = random_problem(rng, n_sessions=3, sizes=(6, 9), D=2, M=2)
    lat = np.full(prob.N * prob.D, (1 << 31) - 1, np.int32)
    prob = prob.with_(lat_us=lat, arrival_us=np.zeros(prob.W, np.int64),
                      load_us=np.zeros_like(prob.load_us), grant_us=0)
    plans = wfgen.make_plans(prob, 300, 8, p_fuse=0.95)
    got = _eval_on_path(prob, plans, 4, path)
    want = oracle_eval(prob, plans)
    assert (want["makespan"][want["status"] == 0] >= (1 << 32)).all()
    assert_same(got, want)


def test_relative_sweep_with_an_idle_device():
    """Plans that leave a device unused keep their base at zero in the
    relative sweep (the smallest free time is that device's 0), so their times
    leave 32 bits and go on to the 64-bit sweep; the others rebase."""
    wf = lib()
    rng = np.random.default_rng(59)
    prob = random_problem(rng, n_sessions=8, sizes=(8, 14), D=3, M=3, tight=False)
    lat = (prob.lat_us.astype(np.int64) % 1000 + (1 << 27)).astype(np.int32)
    prob = prob.with_(lat_us=lat, peak_mib=np.minimum(prob.peak_mib, np.repeat(prob.cap_mib[None, :], prob.N, 0)
                                                      .reshape(-1)).astype(np.int32))
    plans = wfgen.make_plans(prob, 400, 21, p_retain=0.5)
    plans.place[::2, :prob.N] %= 2  # every other plan on devices 0 and 1 only
    want = oracle_eval(prob, plans)
    ok = want["status"] == 0
    assert ok[::2].sum() > 100 and (want["makespan"][ok] >= 1 << 32).mean() > 0.9
    ctx = wf.Ctx(prob, max_P=plans.P)
    wf.wf_ctx_set_eval_path(ctx, wf.PATH_RELATIVE)
    for _ in range(2):
        assert_same(gpu_eval(prob, plans, k=8, ctx=ctx), want)
    ctx.close()


def test_horizon_beyond_2_40_uses_8_byte_slots():
    """The 64-bit sweep keeps its finish slots in 40 bits only while the
    context's horizon (latest arrival plus every node's worst run and load)
    stays below 2^40 us.  About 600 nodes of near 2^31 us each push it past;
    two calls check both launch shapes of the 8-byte-slot sweep."""
    wf = lib()
    rng = np.random.default_rng(53)
    prob = random_problem(rng, n_sessions=20, sizes=(26, 34), D=4, M=3)
    lat = ((1 << 31) - 1 - prob.lat_us.astype(np.int64) % 1000).astype(np.int32)
    prob = prob.with_(lat_us=lat)
    worst = (lat.reshape(prob.N, prob.D).astype(np.int64)
             + prob.load_us.reshape(prob.M, prob.D)[prob.model].astype(np.int64)).max(axis=1)
    horizon = int(prob.arrival_us.max()) + int((worst + prob.grant_us).sum())
    assert horizon >= 1 << 40
    plans = wfgen.make_plans(prob, 400, 11)
    inject_invalid(plans, prob, rng)
    want = oracle_eval(prob, plans)
    assert (want["makespan"][want["status"] == 0] >= (1 << 32)).all()
    ctx = wf.Ctx(prob, max_P=plans.P, device=0)
    for _ in range(2):
        assert_same(gpu_eval(prob, plans, k=8, ctx=ctx), want)
    ctx.close()


def test_repeated_calls_after_overflow():
    """A context whose batches leave 32 bits starts later calls with the u64
    sweep; every call gives the oracle's results."""
    import torch
    from gpu_util import lib
    wf = lib()
    rng = np.random.default_rng(47)
    prob = random_problem(rng, n_sessions=6, sizes=(6, 12), D=3, M=3)
    lat = (prob.lat_us.astype(np.int64) % 1000 + (1 << 30) - 5000).astype(np.int32)
    prob = prob.with_(lat_us=lat)
    plans = wfgen.make_plans(prob, 700, 9, p_retain=0.4)
    want = oracle_eval(prob, plans)
    assert (want["makespan"][want["status"] == 0] >= (1 << 32)).all()
    ctx = wf.Ctx(prob, max_P=plans.P)
    dp = wf.DevicePlans.from_host(plans, "cuda")
    for _ in range(3):
        res = wf.Results(plans.P)
        wf.wf_eval_plans(ctx, dp, res)
        torch.cuda.synchronize()
        mk, p95, gpu, st = res.numpy()
        assert np.array_equal(mk, want["makespan"]) and np.array_equal(p95, want["p95"])
        assert np.array_equal(gpu, want["gpu"]) and np.array_equal(st, want["status"])


def test_mixed_overflow_batch():
    """Some plans overflow u32, some do not, in one batch."""
    rng = np.random.default_rng(37)
    prob = random_problem(rng, n_sessions=4, sizes=(5, 9), D=2, M=3)
    lat = prob.lat_us.astype(np.int64).reshape(prob.N, prob.D)
    lat[:, 1] = (1 << 29)  # device 1 is very slow
    prob = prob.with_(lat_us=lat.astype(np.int32).reshape(-1),
                      peak_mib=np.minimum(prob.peak_mib, prob.cap_mib.min()).astype(np.int32)
                      .clip(min=prob.weight_mib[prob.model].repeat(prob.D)))
    plans = wfgen.make_plans(prob, 500, 4)
    got = gpu_eval(prob, plans, k=5)
    want = oracle_eval(prob, plans)
    big = want["makespan"][want["status"] == 0] >= (1 << 32)
    assert big.any() and (~big).any()
    assert_same(got, want)


def test_wide_fanout_write_lists():
    """A node whose finish feeds many multi-predecessor successors (long
    write lists) and a session with many sinks."""
    N, D, M = 80, 3, 2
    preds = [[] for _ in range(N)]
    # hubs 0 and 1 each feed nodes 2..41, which also depend on both hubs
    for v in range(2, 42):
        preds[v] = [0, 1]
    for v in range(42, N):
        preds[v] = [v - 40]
    rng = np.random.default_rng(5)
    off = np.zeros(N + 1, np.int32)
    off[1:] = np.cumsum([len(p) for p in preds])
    prob = wfgen.Problem(N=N, D=D, M=M, W=1, pred_off=off,
                         pred_idx=np.array([u for p in preds for u in p], np.int32),
                         model=rng.integers(0, M, N).astype(np.uint8), session=np.zeros(N, np.int32),
                         arrival_us=np.zeros(1, np.int64),
                         lat_us=rng.integers(1, 1000, N * D).astype(np.int32),
                         peak_mib=np.full(N * D, 30, np.int32), weight_mib=np.array([20, 25], np.int32),
                         load_us=rng.integers(0, 100, M * D).astype(np.int32),
                         cap_mib=np.array([60, 60, 200], np.int32))
    plans = wfgen.make_plans(prob, 200, 9, p_retain=0.7)
    got = gpu_eval(prob, plans, k=3)
    assert_same(got, oracle_eval(prob, plans))


def test_topk_with_massive_ties():
    """More tied candidates than one sorting tile: 3000 copies of one plan
    plus distinct plans; the tie-break by plan index must hold."""
    w = wfgen.config("mix")
    base = wfgen.make_plans(w.problem, 200, 8)
    P = 3200
    plans = wfgen.Plans.empty(P, w.problem.N)
    best = 0
    for a in ("place", "order", "fuse", "prefetch"):
        arr = getattr(plans, a)
        arr[:3000] = getattr(base, a)[best]
        arr[3000:] = getattr(base, a)[:200]
    for k in (1, 37, 1024):
        got = gpu_eval(w.problem, plans, k=k)
        want = oracle_eval(w.problem, plans)
        ids, keys = oracle.topk(want["makespan"], want["p95"], want["gpu"], want["status"], k)
        assert np.array_equal(got["ids"], ids) and np.array_equal(got["keys"], keys)


@pytest.mark.parametrize("seed", range(3))
def test_admission_margin(seed):
    """The admission margin (peak + margin in every capacity check) on random
    windows and the burst window."""
    rng = np.random.default_rng(5100 + seed)
    prob = random_problem(rng, n_sessions=int(rng.integers(1, 6)), D=int(rng.integers(1, 5)))
    margin = int(rng.integers(1, 400))
    fits = prob.with_(margin_mib=margin).fits().any(axis=1).all()
    prob = prob.with_(margin_mib=margin if fits else 0)
    plans = wfgen.make_plans(prob, int(rng.integers(1, 300)), seed, p_retain=0.5 if seed % 2 else None)
    if plans.P >= 8:
        inject_invalid(plans, prob, rng)
    assert_same(gpu_eval(prob, plans, forecast=True), oracle_eval(prob, plans))
    w = wfgen.config("burst")
    prob = w.problem.with_(margin_mib=512)
    plans = wfgen.make_plans(prob, 1024, seed)
    got = gpu_eval(prob, plans, k=8, forecast=True)
    want = oracle_eval(prob, plans)
    assert_same(got, want)
    rel, comp = oracle.forecast(prob)
    assert np.array_equal(got["rel"], rel) and np.array_equal(got["comp"], comp)


@pytest.mark.parametrize("n_sessions,path", [(33, "auto"), (70, "auto"), (256, "auto"), (300, "auto"),
                                             (70, "wide"), (300, "wide"), (70, "relative"), (300, "relative")])
def test_many_sessions_p95(n_sessions, path):
    """More than 32 sessions: a warp per plan selects the p95 after the sweep
    (up to 256 latencies held in registers, more read from shared memory for
    every bit), on each sweep; equal latencies from sessions with equal
    shapes and arrivals."""
    wf = lib()
    rng = np.random.default_rng(6100 + n_sessions)
    prob = random_problem(rng, n_sessions=n_sessions, sizes=(4, 6), D=4, M=3, arrivals=n_sessions % 2 == 0)
    if path == "relative":
        lat = (prob.lat_us.astype(np.int64) % 1000 + (1 << 26)).astype(np.int32)
        prob = prob.with_(lat_us=lat)
    plans = wfgen.make_plans(prob, 400, n_sessions, p_retain=0.5)
    inject_invalid(plans, prob, rng)
    want = oracle_eval(prob, plans)
    ctx = wf.Ctx(prob, max_P=plans.P)
    if path != "auto":
        wf.wf_ctx_set_eval_path(ctx, wf.PATH_RELATIVE if path == "relative" else wf.PATH_WIDE)
    for _ in range(2):
        assert_same(gpu_eval(prob, plans, k=8, ctx=ctx), want)
    ctx.close()
