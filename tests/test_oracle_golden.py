"""Oracle against hand-worked windows (tests/golden/*.json).

Every expected number in those files is derived by hand in the file itself
from the paper's rules (each fixture cites its equations); none comes from a
program.
"""
import numpy as np
import pytest

import oracle
from golden_util import fixture_names, load, plans_of, problem_of

CASES = [(n, i) for n in fixture_names() for i in range(len(load(n)["cases"]))]


@pytest.mark.parametrize("name,idx", CASES, ids=[f"{n}[{i}]" for n, i in CASES])
def test_golden_case(name, idx):
    fx = load(name)
    case = fx["cases"][idx]
    prob = problem_of(fx, case)
    plans = plans_of(fx, [case])
    res = oracle.eval_plan(prob, plans, 0, trace=True)
    exp = case["expect"]
    assert res["status"] == exp["status"]
    if exp["status"] != 0:
        assert res["makespan"] == res["p95"] == res["gpu"] == oracle.INT64_MAX
        return
    assert (res["makespan"], res["p95"], res["gpu"]) == (exp["makespan"], exp["p95"], exp["gpu"])
    tr = res["trace"]
    if "finish" in exp:
        assert tr["finish"].tolist() == exp["finish"]
    if "loads" in exp:
        assert int((tr["load_start"] >= 0).sum()) == exp["loads"]
    if "units" in exp:
        assert len(tr["unit_head"]) == exp["units"]
    if "timely" in exp:  # the window terms of Eq. 12's ranking key
        timely, life = oracle.eval_phi(prob, plans)
        assert (int(timely[0]), int(life[0])) == (exp["timely"], exp["life"])
    if "evicted" in exp:
        got = {str(h): [m for m in range(32) if (int(tr["evicted"][h]) >> m) & 1]
               for h in tr["unit_head"] if tr["evicted"][h]}
        assert got == exp["evicted"]


def test_status_via_batch_matches_single():
    fx = load("t7_status_bits")
    prob = problem_of(fx)
    plans = plans_of(fx, fx["cases"])
    mk, p95, gpu, st = oracle.eval_plans(prob, plans)
    assert st.tolist() == [c["expect"]["status"] for c in fx["cases"]]
    assert all(mk[i] == oracle.INT64_MAX for i in range(len(st)) if st[i])
