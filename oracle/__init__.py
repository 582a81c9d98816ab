"""CPU oracle for batched plan evaluation -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg (and its ``--impl reference`` arm) may import this package.  The product
library never does, and this package imports nothing from it.

The arithmetic lives in ``wf_oracle.c`` (plain single-threaded C, built here
with the host compiler); this module marshals arrays to it and adds the top-k
selection, which is a plain sort of the (status, makespan, p95, gpu, plan id)
key (the analog of the lexicographic ranking key of Eq. 12).

Inputs are duck-typed: any object with the attributes of a problem (N, D, M,
W, pred_off, pred_idx, model, session, arrival_us, lat_us, peak_mib,
weight_mib, load_us, cap_mib, grant_us, S, seed, bm_r, bm_c, bm_e) and of a
plan batch (P, place, order, fuse, prefetch, retain, plan_base and strides).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wf_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None
_lock = threading.Lock()
INT64_MAX = np.iinfo(np.int64).max


def build(force: bool = False, extra_flags: tuple = (), out: str | None = None) -> str:
    """Compile the oracle into an in-tree shared library (gcc -O2)."""
    target = out or _LIB
    if force or out or not os.path.exists(target) or os.path.getmtime(target) < os.path.getmtime(_SRC):
        tmp = target + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", *extra_flags,
                               "-o", tmp, _SRC])
        os.replace(tmp, target)
    return target


class _Problem(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int32), ("D", ctypes.c_int32), ("M", ctypes.c_int32),
                ("W", ctypes.c_int32),
                ("pred_off", ctypes.c_void_p), ("pred_idx", ctypes.c_void_p),
                ("model", ctypes.c_void_p), ("session", ctypes.c_void_p),
                ("arrival", ctypes.c_void_p), ("lat", ctypes.c_void_p), ("peak", ctypes.c_void_p),
                ("weight", ctypes.c_void_p), ("load", ctypes.c_void_p), ("cap", ctypes.c_void_p),
                ("grant", ctypes.c_int32), ("S", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("bm_r", ctypes.c_void_p), ("bm_c", ctypes.c_void_p), ("bm_e", ctypes.c_void_p),
                ("bm_rn", ctypes.c_int32), ("bm_cn", ctypes.c_int32), ("bm_en", ctypes.c_int32),
                ("reclaim", ctypes.c_int32), ("batch", ctypes.c_int32)]


class _Trace(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "unit_head", "n_units", "head_of", "start", "finish", "rel", "load_start", "load_end",
        "kv_adm", "used_after", "evicted", "reclaimed", "occ_start", "occ_end", "occ_dev", "n_occ", "adm")]


def _setup(lib):
    p = ctypes.c_void_p
    i64 = ctypes.c_int64
    lib.orc_fusible_next.argtypes = [p, p]
    lib.orc_forecast.argtypes = [p, p, p]
    lib.orc_status.argtypes = [p, p, p, p]
    lib.orc_eval_plan.argtypes = [p, p, p, p, p, p, p, i64, p, p, p]
    lib.orc_eval_batch.argtypes = [p, p, p, i64, p, i64, p, p, p, i64, i64, i64, i64, p, p, p, p]
    lib.orc_eval_phi_batch.argtypes = [p, p, p, i64, p, i64, p, p, p, i64, i64, i64, p, p]
    lib.orc_splitmix64.argtypes = [ctypes.c_uint64]
    lib.orc_splitmix64.restype = ctypes.c_uint64
    lib.orc_multiplier.argtypes = [p, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64]
    lib.orc_multiplier.restype = ctypes.c_int64
    lib.orc_mutate.argtypes = [p, p, i64, p, i64, p, p, p, i64, i64, p, i64, p, i64, p, p, p, i64, i64,
                               ctypes.c_uint64, i64, ctypes.c_int32]
    lib.orc_construct.argtypes = [p, p, ctypes.c_uint64, ctypes.c_uint64, i64, p, p, p, p, p]
    for f in ("orc_fusible_next", "orc_forecast", "orc_status", "orc_eval_plan", "orc_eval_batch", "orc_mutate",
              "orc_construct", "orc_eval_phi_batch"):
        getattr(lib, f).restype = ctypes.c_int
    return lib


def load(path: str | None = None):
    """The oracle library (built on first use).  ``path``, or the environment
    variable WF_ORACLE_LIB, loads another build instead: the mutation test
    points it at copies of this source with a planted mistake."""
    global _lib
    if path is not None:
        return _setup(ctypes.CDLL(path))
    with _lock:
        if _lib is None:
            alt = os.environ.get("WF_ORACLE_LIB")
            _lib = _setup(ctypes.CDLL(alt if alt else build()))
    return _lib


def _a(x, dt):
    return np.ascontiguousarray(np.asarray(x, dtype=dt))


class OracleProblem:
    """Holds contiguous copies of a problem's arrays and the C view of them."""

    def __init__(self, prob, lib=None):
        self.lib = lib or load()
        self.N, self.D, self.M, self.W = int(prob.N), int(prob.D), int(prob.M), int(prob.W)
        self.arrays = dict(
            pred_off=_a(prob.pred_off, np.int32), pred_idx=_a(prob.pred_idx, np.int32),
            model=_a(prob.model, np.uint8), session=_a(prob.session, np.int32),
            arrival=_a(prob.arrival_us, np.int64), lat=_a(prob.lat_us, np.int32),
            # admission memory (Section 3.3): predicted peak + margin, in every capacity check
            peak=_a(np.asarray(prob.peak_mib, np.int64) + int(getattr(prob, "margin_mib", 0)), np.int32),
            weight=_a(prob.weight_mib, np.int32),
            load=_a(prob.load_us, np.int32), cap=_a(prob.cap_mib, np.int32),
            bm_r=_a(prob.bm_r, np.int32), bm_c=_a(prob.bm_c, np.int32), bm_e=_a(prob.bm_e, np.int32))
        if self.arrays["pred_idx"].size == 0:
            self.arrays["pred_idx"] = np.zeros(1, np.int32)
        ar = self.arrays
        self.S = int(prob.S)
        self.c = _Problem(self.N, self.D, self.M, self.W,
                          *[ar[k].ctypes.data for k in ("pred_off", "pred_idx", "model", "session",
                                                        "arrival", "lat", "peak", "weight", "load", "cap")],
                          int(prob.grant_us), self.S, int(prob.seed) & ((1 << 64) - 1),
                          ar["bm_r"].ctypes.data, ar["bm_c"].ctypes.data, ar["bm_e"].ctypes.data,
                          int(np.asarray(prob.bm_r).size), int(np.asarray(prob.bm_c).size),
                          int(np.asarray(prob.bm_e).size), int(getattr(prob, "reclaim", 0)),
                          int(getattr(prob, "batch", 0)))
        self.fnext = np.empty(self.N, np.int32)
        if self.lib.orc_fusible_next(ctypes.byref(self.c), self.fnext.ctypes.data) != 0:
            raise MemoryError("oracle allocation failed")


def fusible_next(prob) -> np.ndarray:
    """fnext[u] = v when edge (u, v) satisfies Eq. 3, else -1."""
    return OracleProblem(prob).fnext.copy()


def forecast(prob):
    """Release forecast (Eq. 2): (rel, comp) int64 [N] each."""
    op = OracleProblem(prob)
    rel = np.empty(op.N, np.int64)
    comp = np.empty(op.N, np.int64)
    rc = op.lib.orc_forecast(ctypes.byref(op.c), rel.ctypes.data, comp.ctypes.data)
    if rc != 0:
        raise ValueError(f"oracle forecast failed ({rc})")
    return rel, comp


def status(prob, place_row, order_row) -> int:
    op = OracleProblem(prob)
    st = np.zeros(1, np.uint32)
    pl = _a(place_row, np.uint8)
    od = _a(order_row, np.uint16)
    if op.lib.orc_status(ctypes.byref(op.c), pl.ctypes.data, od.ctypes.data, st.ctypes.data):
        raise MemoryError
    return int(st[0])


def _row(arr, p, dt):
    return None if arr is None else _a(arr[p], dt)


def eval_plan(prob, plans, p: int, trace: bool = False, op: OracleProblem | None = None):
    """Evaluate plan p.  Returns dict(makespan, p95, gpu, status[, trace])."""
    op = op or OracleProblem(prob)
    N, D = op.N, op.D
    pl, od = _row(plans.place, p, np.uint8), _row(plans.order, p, np.uint16)
    fu, pf = _row(plans.fuse, p, np.uint32), _row(plans.prefetch, p, np.uint32)
    rt = _row(plans.retain, p, np.uint32)
    out = np.zeros(3, np.int64)
    st = np.zeros(1, np.uint32)
    tr = None
    tra = None
    if trace:
        tra = dict(unit_head=np.full(N, -1, np.int32), n_units=np.zeros(1, np.int32),
                   head_of=np.full(N, -1, np.int32), start=np.full(N, -1, np.int64),
                   finish=np.full(N, -1, np.int64), rel=np.full(N, -1, np.int64),
                   load_start=np.full(N, -1, np.int64), load_end=np.full(N, -1, np.int64),
                   kv_adm=np.zeros(N, np.int32), used_after=np.zeros(N, np.int32),
                   evicted=np.zeros(N, np.uint32), reclaimed=np.zeros(N, np.uint8),
                   occ_start=np.zeros(N + D, np.int64), occ_end=np.zeros(N + D, np.int64),
                   occ_dev=np.zeros(N + D, np.int32), n_occ=np.zeros(1, np.int32),
                   adm=np.full(N, -1, np.int64))
        tr = _Trace(*[tra[f].ctypes.data for f, _ in _Trace._fields_])
    rc = op.lib.orc_eval_plan(ctypes.byref(op.c), op.fnext.ctypes.data, pl.ctypes.data, od.ctypes.data,
                              fu.ctypes.data, pf.ctypes.data, None if rt is None else rt.ctypes.data,
                              int(getattr(plans, "plan_base", 0)) + p, out.ctypes.data, st.ctypes.data,
                              None if tr is None else ctypes.byref(tr))
    if rc != 0:
        raise RuntimeError(f"oracle eval failed ({rc})")
    res = dict(makespan=int(out[0]), p95=int(out[1]), gpu=int(out[2]), status=int(st[0]))
    if trace:
        nu, no = int(tra["n_units"][0]), int(tra["n_occ"][0])
        tra["unit_head"] = tra["unit_head"][:nu]
        for k in ("occ_start", "occ_end", "occ_dev"):
            tra[k] = tra[k][:no]
        res["trace"] = tra
    return res


def eval_plans(prob, plans, lo: int = 0, hi: int | None = None, threads: int = 1):
    """Evaluate plans [lo, hi).  Returns (makespan, p95, gpu, status) arrays of
    length hi - lo.  ``threads`` > 1 maps the single-threaded oracle over
    contiguous plan ranges in parallel (the harness is the only parallel part)."""
    op = OracleProblem(prob)
    hi = plans.P if hi is None else hi
    n = hi - lo
    mk = np.zeros(n, np.int64)
    p95 = np.zeros(n, np.int64)
    gpu = np.zeros(n, np.int64)
    st = np.zeros(n, np.uint32)
    place = np.ascontiguousarray(plans.place[lo:hi])
    order = np.ascontiguousarray(plans.order[lo:hi])
    fuse = np.ascontiguousarray(plans.fuse[lo:hi])
    pref = np.ascontiguousarray(plans.prefetch[lo:hi])
    ret = None if plans.retain is None else np.ascontiguousarray(plans.retain[lo:hi])
    base = int(getattr(plans, "plan_base", 0)) + lo

    def run(rng):
        a, b = rng
        rc = op.lib.orc_eval_batch(ctypes.byref(op.c), op.fnext.ctypes.data,
                                   place.ctypes.data, place.shape[1], order.ctypes.data,
                                   order.shape[1] * 2, fuse.ctypes.data, pref.ctypes.data,
                                   None if ret is None else ret.ctypes.data, fuse.shape[1] * 4,
                                   base, a, b, mk.ctypes.data, p95.ctypes.data, gpu.ctypes.data,
                                   st.ctypes.data)
        if rc != 0:
            raise RuntimeError(f"oracle eval failed ({rc})")

    if threads <= 1 or n < 2:
        run((0, n))
    else:
        step = max(1, (n + threads * 4 - 1) // (threads * 4))
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(run, [(a, min(n, a + step)) for a in range(0, n, step)]))
    return mk, p95, gpu, st


def eval_phi(prob, plans, lo: int = 0, hi: int | None = None, threads: int = 1):
    """The window terms of Eq. 12's ranking key for plans [lo, hi) of a
    deterministic batch: (timely prefetches P_N, lifecycle overhead H_life in
    us), INT64_MAX for invalid plans.  See orc_eval_phi_batch."""
    op = OracleProblem(prob)
    hi = plans.P if hi is None else hi
    n = hi - lo
    timely = np.zeros(n, np.int64)
    life = np.zeros(n, np.int64)
    place = np.ascontiguousarray(plans.place[lo:hi])
    order = np.ascontiguousarray(plans.order[lo:hi])
    fuse = np.ascontiguousarray(plans.fuse[lo:hi])
    pref = np.ascontiguousarray(plans.prefetch[lo:hi])
    ret = None if plans.retain is None else np.ascontiguousarray(plans.retain[lo:hi])

    def run(rng):
        a, b = rng
        rc = op.lib.orc_eval_phi_batch(ctypes.byref(op.c), op.fnext.ctypes.data,
                                       place.ctypes.data, place.shape[1], order.ctypes.data,
                                       order.shape[1] * 2, fuse.ctypes.data, pref.ctypes.data,
                                       None if ret is None else ret.ctypes.data, fuse.shape[1] * 4,
                                       a, b, timely.ctypes.data, life.ctypes.data)
        if rc != 0:
            raise RuntimeError(f"oracle phi failed ({rc})")

    if threads <= 1 or n < 2:
        run((0, n))
    else:
        step = max(1, (n + threads * 4 - 1) // (threads * 4))
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(run, [(a, min(n, a + step)) for a in range(0, n, step)]))
    return timely, life


def topk_phi(makespan, timely, life, status, k: int, plan_base: int = 0):
    """The k best plans by Eq. 12's window key (invalid last, latest
    completion, most timely prefetches, least lifecycle overhead, plan id).
    Returns (ids int32 [k], keys int64 [k][3] = makespan, timely, life)."""
    P = len(makespan)
    key = sorted(range(P), key=lambda p: (int(status[p]) != 0, int(makespan[p]), -int(timely[p]),
                                          int(life[p]), p))
    ids = np.array(key[:k], np.int32)
    keys = np.stack([np.asarray(makespan)[ids], np.asarray(timely)[ids], np.asarray(life)[ids]], axis=1)
    return ids + plan_base, keys.astype(np.int64)


def topk(makespan, p95, gpu, status, k: int, plan_base: int = 0):
    """The k best plans by (invalid last, makespan, p95, gpu, plan id).
    Returns (ids int32 [k], keys int64 [k][3])."""
    P = len(makespan)
    key = sorted(range(P), key=lambda p: (int(status[p]) != 0, int(makespan[p]), int(p95[p]),
                                          int(gpu[p]), p))
    ids = np.array(key[:k], np.int32)
    keys = np.stack([np.asarray(makespan)[ids], np.asarray(p95)[ids], np.asarray(gpu)[ids]], axis=1)
    return ids + plan_base, keys.astype(np.int64)


def splitmix64(x: int) -> int:
    return int(load().orc_splitmix64(x & ((1 << 64) - 1)))


def multiplier(prob, plan: int, sample: int, node: int) -> int:
    op = OracleProblem(prob)
    return int(op.lib.orc_multiplier(ctypes.byref(op.c), plan, sample, node))


class PlanRows:
    """A batch of plan rows (the layout of the evaluator's inputs)."""

    def __init__(self, P: int, N: int, with_retain: bool, plan_base: int = 0):
        words = (N + 31) // 32
        self.P, self.N, self.plan_base = P, N, plan_base
        self.place = np.zeros((P, N), np.uint8)
        self.order = np.zeros((P, N), np.uint16)
        self.fuse = np.zeros((P, words), np.uint32)
        self.prefetch = np.zeros((P, words), np.uint32)
        self.retain = np.zeros((P, words), np.uint32) if with_retain else None

    @staticmethod
    def copy_of(plans, N: int):
        """Rows 0..P-1 of any batch with the same fields (padding dropped)."""
        words = (N + 31) // 32
        retain = getattr(plans, "retain", None)
        out = PlanRows(plans.P, N, retain is not None, int(getattr(plans, "plan_base", 0)))
        out.place[:] = plans.place[:, :N]
        out.order[:] = plans.order[:, :N]
        out.fuse[:] = plans.fuse[:, :words]
        out.prefetch[:] = plans.prefetch[:, :words]
        if retain is not None:
            out.retain[:] = retain[:, :words]
        return out


def mutate(prob, parents, n_children: int, seed: int, round_: int, n_ops: int, plan_base: int = 0):
    """Children of a parent batch: child c copies parent c mod P and takes
    n_ops point changes (move / fuse flip / prefetch flip / adjacent swap)
    decoded from SplitMix64 of (seed, round, c, step)."""
    op = OracleProblem(prob)
    N = op.N
    par = {a: np.ascontiguousarray(getattr(parents, a)) for a in ("place", "order", "fuse", "prefetch")}
    ret = None if parents.retain is None else np.ascontiguousarray(parents.retain)
    ch = PlanRows(n_children, N, ret is not None, plan_base)
    rc = op.lib.orc_mutate(ctypes.byref(op.c), par["place"].ctypes.data, par["place"].shape[1],
                           par["order"].ctypes.data, par["order"].shape[1] * 2,
                           par["fuse"].ctypes.data, par["prefetch"].ctypes.data,
                           None if ret is None else ret.ctypes.data, par["fuse"].shape[1] * 4, parents.P,
                           ch.place.ctypes.data, N, ch.order.ctypes.data, 2 * N,
                           ch.fuse.ctypes.data, ch.prefetch.ctypes.data,
                           None if ch.retain is None else ch.retain.ctypes.data, ch.fuse.shape[1] * 4,
                           n_children, seed & ((1 << 64) - 1), round_, n_ops)
    if rc != 0:
        raise RuntimeError(f"oracle mutate failed ({rc})")
    return ch


def merge_elite(elite_metrics, child_metrics, k: int):
    """The k best of elite (indices 0..k-1) and children (k, k+1, ...) by the
    top-k key, kept in place: elite slots whose plan stays keep it; the
    leaving slots, in ascending order, take the entering children in key
    order.  Returns [(slot, child)] and the elite's new metrics."""
    union = [np.concatenate([np.asarray(e), np.asarray(c)]) for e, c in zip(elite_metrics, child_metrics)]
    ids, _ = topk(union[0], union[1], union[2], union[3], k)
    ids = [int(i) for i in ids]
    entering = [i - k for i in ids if i >= k]
    kept = set(i for i in ids if i < k)
    leaving = [s for s in range(k) if s not in kept]
    pairs = list(zip(leaving, entering))
    new = [np.asarray(e).copy() for e in elite_metrics]
    for s, c in pairs:
        for a in range(4):
            new[a][s] = np.asarray(child_metrics[a])[c]
    return pairs, new


def local_search(prob, elite, elite_metrics, n_children: int, seed: int, round0: int, rounds: int,
                 n_ops: int, children_plan_base: int = 0, threads: int = 1):
    """rounds x (children of the elite -> evaluate -> keep the k best in
    place).  Returns the final elite rows and metrics."""
    k = elite.P
    cur = PlanRows.copy_of(elite, int(prob.N))
    met = [np.asarray(m).copy() for m in elite_metrics]
    for r in range(rounds):
        ch = mutate(prob, cur, n_children, seed, round0 + r, n_ops, children_plan_base)
        cm = eval_plans(prob, ch, threads=threads)
        pairs, met = merge_elite(met, cm, k)
        for s, c in pairs:
            for a in ("place", "order", "fuse", "prefetch", "retain"):
                if getattr(cur, a) is not None:
                    getattr(cur, a)[s] = getattr(ch, a)[c]
    return cur, met


def construct(prob, P: int, seed: int, jitter: int, plan_base: int = 0):
    """P plans from the list-scheduling constructor (plan index plan_base + p
    seeds the jitter).  Returns (PlanRows, end times int64 [P])."""
    op = OracleProblem(prob)
    N = op.N
    out = PlanRows(P, N, False, plan_base)
    ends = np.zeros(P, np.int64)
    end = ctypes.c_int64(0)
    for p in range(P):
        rc = op.lib.orc_construct(ctypes.byref(op.c), op.fnext.ctypes.data, seed & ((1 << 64) - 1),
                                  (plan_base + p) & ((1 << 64) - 1), int(jitter),
                                  out.place[p].ctypes.data, out.order[p].ctypes.data,
                                  out.fuse[p].ctypes.data, out.prefetch[p].ctypes.data, ctypes.byref(end))
        if rc != 0:
            raise RuntimeError(f"oracle construct failed ({rc})")
        ends[p] = end.value
    return out, ends
