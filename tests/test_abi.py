"""The C-ABI library loads and exports every entry point include/*.h declares;
host-side validation rejects malformed problems (no GPU needed)."""
import ctypes
import glob
import os
import re

import numpy as np
import pytest

import wfgen
from randprob import random_problem

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def wf():
    from paper_2609_03335_gb300 import build, wf
    build.build()
    wf.load_library()
    return wf


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"\b(wf_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


def test_every_declared_symbol_is_exported(wf):
    names = declared_functions()
    assert "wf_eval_plans" in names and "wf_topk" in names
    lib = ctypes.CDLL(wf.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) <= set(wf.EXPORTS)


def test_strerror(wf):
    for code in range(5):
        assert wf.wf_strerror(code)
    assert wf.wf_strerror(99) == "unknown error"


@pytest.mark.parametrize("name", wfgen.CONFIG_NAMES)
def test_named_workloads_are_valid(wf, name):
    assert wf.wf_problem_check(wfgen.config(name).problem) == wf.WF_OK


def _mutate(prob, **kw):
    return prob.with_(**{k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in kw.items()})


def test_validation_rejects(wf):
    rng = np.random.default_rng(0)
    p = random_problem(rng, n_sessions=3, permute=False)
    assert wf.wf_problem_check(p) == wf.WF_OK
    bad = []
    # cycle: make node 0 depend on the last node of its session
    w0 = np.nonzero(p.session == 0)[0]
    off = p.pred_off.copy()
    idx = list(p.pred_idx)
    preds = [idx[off[v]:off[v + 1]] for v in range(p.N)]
    preds[int(w0[0])] = [int(w0[-1])]
    noff = np.zeros(p.N + 1, np.int32)
    noff[1:] = np.cumsum([len(x) for x in preds])
    bad.append(("cycle", p.with_(pred_off=noff, pred_idx=np.array([u for x in preds for u in x], np.int32))))
    # cross-session edge
    preds2 = [list(x) for x in [idx[off[v]:off[v + 1]] for v in range(p.N)]]
    w1 = np.nonzero(p.session == 1)[0]
    preds2[int(w1[-1])].append(int(w0[0]))
    noff2 = np.zeros(p.N + 1, np.int32)
    noff2[1:] = np.cumsum([len(x) for x in preds2])
    bad.append(("cross", p.with_(pred_off=noff2, pred_idx=np.array([u for x in preds2 for u in x], np.int32))))
    # infeasible node
    pk = p.peak_mib.copy().reshape(p.N, p.D)
    pk[3, :] = p.cap_mib.max() + 1
    bad.append(("nofit", p.with_(peak_mib=pk.reshape(-1))))
    # peak below weight
    pk2 = p.peak_mib.copy().reshape(p.N, p.D)
    pk2[2, 0] = p.weight_mib[p.model[2]] - 1
    bad.append(("peak<W", p.with_(peak_mib=pk2.reshape(-1))))
    bad.append(("model>=M", p.with_(model=np.full(p.N, p.M, np.uint8))))
    bad.append(("D=0", p.with_(D=0)))
    bad.append(("D=33", p.with_(D=33)))
    bad.append(("M=17", p.with_(M=17)))
    s = p.session.copy()
    s[s == 2] = 1
    bad.append(("empty session", p.with_(session=s)))
    arr = p.arrival_us.copy()
    arr[1] = -1
    bad.append(("negative arrival", p.with_(arrival_us=arr)))
    bad.append(("negative grant", p.with_(grant_us=-1)))
    r, c, e = wfgen.box_muller_tables()
    bad.append(("short E", p.with_(S=2, bm_r=r, bm_c=c, bm_e=e[100:-100])))
    bad.append(("non-pow2 R", p.with_(S=2, bm_r=r[:4000], bm_c=c, bm_e=e)))
    for label, q in bad:
        assert wf.wf_problem_check(q) == wf.WF_EINVAL, label
        assert wf.wf_last_error(), label
    assert wf.wf_problem_check(p.with_(S=2, bm_r=r, bm_c=c, bm_e=e)) == wf.WF_OK
