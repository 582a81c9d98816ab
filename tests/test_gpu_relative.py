"""Windows whose times run far past 2^32 us, started in the sweep with 32-bit
times relative to a per-plan base (PATH_RELATIVE) and in the 64-bit sweep
(PATH_WIDE), against the oracle.  The cases cover bases raised while
sessions still arrive (arrivals up to 4e9 us), sessions that finish long
before their plan ends, devices that empty and fill again (retain rows),
invalid plans, and the plans that leave 32 bits even so (a device left idle
keeps a plan's base at zero; a fused chain's summed run time of 2^32 or more
sends its plan to the int64 path), whichever of those the random windows
produce."""
import numpy as np
import pytest

import wfgen
from gpu_util import assert_same, gpu_eval, lib, oracle_eval
from randprob import random_problem
from test_gpu_parity import inject_invalid

pytestmark = pytest.mark.gpu

# seed, log2 of the node run times, latest arrival, devices
CASES = [
    (0, 30, 500, 3),
    (1, 27, 4_000_000_000, 3),
    (2, 28, 2_000_000_000, 2),
    (3, 29, 3_500_000_000, 4),
    (4, 26, 1_000_000_000, 2),
    (5, 25, 3_000_000_000, 5),
]


def wide_window(seed, lat_bits, arr_max, D):
    """A random window with node run times near 2^lat_bits us and session
    arrivals spread over [0, arr_max]."""
    rng = np.random.default_rng(9100 + seed)
    prob = random_problem(rng, n_sessions=12, sizes=(8, 16), D=D, M=3)
    lat = (prob.lat_us.astype(np.int64) % 1000 + (1 << lat_bits)).astype(np.int32)
    arr = np.sort(rng.integers(0, arr_max + 1, prob.W)).astype(np.int64)
    arr[0] = 0
    return prob.with_(lat_us=lat, arrival_us=arr), rng


@pytest.mark.parametrize("seed,lat_bits,arr_max,D", CASES)
@pytest.mark.parametrize("path", ["relative", "wide"])
def test_windows_past_32_bits(seed, lat_bits, arr_max, D, path):
    wf = lib()
    prob, rng = wide_window(seed, lat_bits, arr_max, D)
    plans = wfgen.make_plans(prob, 600, seed, p_retain=0.4 if seed % 2 else None)
    inject_invalid(plans, prob, rng)
    want = oracle_eval(prob, plans)
    ok = want["status"] == 0
    assert ok.sum() > 300 and (want["makespan"][ok] >= 1 << 32).mean() > 0.9
    ctx = wf.Ctx(prob, max_P=plans.P)
    wf.wf_ctx_set_eval_path(ctx, wf.PATH_RELATIVE if path == "relative" else wf.PATH_WIDE)
    for _ in range(2):
        assert_same(gpu_eval(prob, plans, k=8, ctx=ctx), want)
    ctx.close()


def test_automatic_switch_to_the_relative_sweep():
    """Under PATH_AUTO the first call plays the 32-bit sweep, which hands
    every plan on; later calls start in the relative sweep."""
    wf = lib()
    prob, rng = wide_window(1, 27, 4_000_000_000, 3)
    plans = wfgen.make_plans(prob, 900, 77, p_retain=0.3)
    want = oracle_eval(prob, plans)
    ctx = wf.Ctx(prob, max_P=plans.P)
    for _ in range(3):
        assert_same(gpu_eval(prob, plans, k=8, ctx=ctx), want)
    ctx.close()


def test_relative_path_refused_where_it_does_not_apply():
    """A window with more sessions than half its finish slots has no room for
    the sessions' 64-bit latencies in slot pairs: PATH_RELATIVE is refused,
    PATH_WIDE accepted, and the context still evaluates."""
    wf = lib()
    rng = np.random.default_rng(5)
    dev = wfgen.DeviceSpec(cap_gib=[40.0, 40.0], speed=[1.0, 1.5], bw_gbps=[10, 10])
    prob = wfgen.assemble("solo", [[("solo", [])] for _ in range(40)], np.zeros(40, np.int64), dev,
                          [4.0, 8.0], rng, lat_median_us=100, kv_lo=1, kv_hi=20)
    plans = wfgen.make_plans(prob, 64, 1)
    ctx = wf.Ctx(prob, max_P=plans.P)
    with pytest.raises(wf.WfError) as e:
        wf.wf_ctx_set_eval_path(ctx, wf.PATH_RELATIVE)
    assert e.value.code == wf.WF_EINVAL
    wf.wf_ctx_set_eval_path(ctx, wf.PATH_WIDE)
    assert_same(gpu_eval(prob, plans, ctx=ctx), oracle_eval(prob, plans))
    with pytest.raises(wf.WfError):
        wf.wf_ctx_set_eval_path(ctx, 4)
    ctx.close()
