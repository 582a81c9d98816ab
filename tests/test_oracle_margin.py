"""Pins of the admission margin (Section 3.3: the memory reserved for
admission is the predicted peak plus a margin epsilon_M)."""
import numpy as np

import oracle
import wfgen


def t1(kv, margin):
    """The hand-worked forced eviction: one device of 100 MiB; models A (60
    MiB, load 20 us) and B (30 MiB, load 10 us); chain n0 (A, 100 us) -> n1 (B,
    50 us) -> n2 (A, 70 us), each needing `kv` MiB beyond its weights."""
    weight = np.array([60, 30], np.int32)
    model = np.array([0, 1, 0], np.uint8)
    return wfgen.Problem(N=3, D=1, M=2, W=1, pred_off=np.array([0, 0, 1, 2], np.int32),
                         pred_idx=np.array([0, 1], np.int32), model=model, session=np.zeros(3, np.int32),
                         arrival_us=np.zeros(1, np.int64), lat_us=np.array([100, 50, 70], np.int32),
                         peak_mib=(weight[model] + kv).astype(np.int32), weight_mib=weight,
                         load_us=np.array([20, 10], np.int32), cap_mib=np.array([100], np.int32),
                         margin_mib=margin)


def one_plan(prob):
    P = wfgen.Plans.empty(1, prob.N)
    P.place[0, :prob.N] = 0
    P.order[0, :prob.N] = np.arange(prob.N)
    return P


def test_margin_adds_to_the_admission_memory():
    """kv = 20: A + B + 20 > 100 forces both evictions (makespan 270); kv = 10
    fits exactly (60 + 30 + 10 = 100) without any (n2 ends at 250).  kv = 10
    with a 10 MiB margin admits like kv = 20, and one MiB of margin already
    tips it over the capacity."""
    assert oracle.eval_plan(t1(20, 0), one_plan(t1(20, 0)), 0)["makespan"] == 270
    assert oracle.eval_plan(t1(10, 0), one_plan(t1(10, 0)), 0)["makespan"] == 250
    assert oracle.eval_plan(t1(10, 10), one_plan(t1(10, 10)), 0)["makespan"] == 270
    assert oracle.eval_plan(t1(10, 1), one_plan(t1(10, 1)), 0)["makespan"] == 270


def test_margin_decides_where_a_node_fits():
    """Peak exactly at capacity on device 0 fits without a margin and not with
    one (status bit 2); the forecast then takes the other device's run time."""
    prob = wfgen.Problem(N=1, D=2, M=1, W=1, pred_off=np.zeros(2, np.int32), pred_idx=np.zeros(0, np.int32),
                         model=np.zeros(1, np.uint8), session=np.zeros(1, np.int32),
                         arrival_us=np.zeros(1, np.int64), lat_us=np.array([10, 30], np.int32),
                         peak_mib=np.array([8, 8], np.int32), weight_mib=np.array([4], np.int32),
                         load_us=np.zeros(2, np.int32), cap_mib=np.array([8, 20], np.int32))
    place0 = np.zeros(1, np.uint8)
    order = np.zeros(1, np.uint16)
    assert oracle.status(prob, place0, order) == 0
    assert oracle.status(prob.with_(margin_mib=1), place0, order) == 2
    assert oracle.forecast(prob)[1][0] == 10
    assert oracle.forecast(prob.with_(margin_mib=1))[1][0] == 30
    assert not prob.with_(margin_mib=1).fits()[0, 0] and prob.with_(margin_mib=1).fits()[0, 1]
