"""Seeded synthetic workloads for batched plan evaluation (input data only).

This package builds the inputs that both the CPU oracle and the GPU library
consume, and nothing else: it holds none of the evaluation arithmetic (no
release times, no residency, no metrics).

* ``Problem``: one cross-workflow window of the activation DAG (Section 3.2)
  with Predictor-style cost tables (Eq. 1): per activation and device a run
  time in integer microseconds and a peak memory in MiB, per model and device
  a load time, and per device a memory capacity.
* ``Plans``: candidate physical plans (Eq. 6-10): per activation a device, a
  dispatch sequence, and fusion / prefetch / retain bits.
* ``config(name)``: the five named workloads (tiny window, three-scenario mix,
  burst arrivals, stochastic latencies, large window).

The DAG families stand in for the workflow shapes of the paper's three
scenarios (Section 4.1): a software-development chain with unrolled repair
loops, a parallel-research fan-out / fan-in, and a random layered DAG.  No
dataset content is used.  Problem tables come from numpy's PCG64; plans come
from a counter-based SplitMix64 draw per (plan, element) in ``plangen.c``.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "plangen.c")
_LIB = os.path.join(_HERE, "libwfgen.so")
_lib = None
_lib_lock = threading.Lock()

GIB = 1024  # MiB per GiB


def build(force: bool = False) -> str:
    """Compile the plan generator with the host C compiler (in-tree .so)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lib_lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            p = ctypes.c_void_p
            i32, i64, u64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
            lib.wfg_make_plans.restype = ctypes.c_int
            lib.wfg_make_plans.argtypes = [i32, p, p, p, p, p, u64, i64, i64, i64,
                                           u64, u64, u64, p, i64, p, i64, p, p, p, i64]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _round16(x: int) -> int:
    return (x + 15) // 16 * 16


@dataclass
class Problem:
    """One planning window: DAG (pred CSR), sessions, and integer cost tables.

    Layouts: ``lat_us`` and ``peak_mib`` are row-major [N][D]; ``load_us`` is
    [M][D].  Times are microseconds, memory MiB.
    """
    N: int
    D: int
    M: int
    W: int
    pred_off: np.ndarray      # int32 [N+1]
    pred_idx: np.ndarray      # int32 [E]
    model: np.ndarray         # uint8 [N]
    session: np.ndarray       # int32 [N]
    arrival_us: np.ndarray    # int64 [W]
    lat_us: np.ndarray        # int32 [N*D]
    peak_mib: np.ndarray      # int32 [N*D]
    weight_mib: np.ndarray    # int32 [M]
    load_us: np.ndarray       # int32 [M*D]
    cap_mib: np.ndarray       # int32 [D]
    grant_us: int = 0
    S: int = 0
    seed: int = 0
    bm_r: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int32))
    bm_c: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int32))
    bm_e: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int32))
    name: str = ""
    reclaim: int = 0          # reclamation order: 0 least recently used, 1 by next use
    margin_mib: int = 0       # admission margin: capacity checks use peak + margin
    batch: int = 0            # replica batch limit B_q (0: one unit at a time per device)

    @property
    def E(self) -> int:
        return int(self.pred_idx.shape[0])

    def succ_csr(self):
        """Successor lists (CSR) derived from the pred lists."""
        cnt = np.zeros(self.N + 1, np.int64)
        np.add.at(cnt, self.pred_idx.astype(np.int64) + 1, 1)
        off = np.cumsum(cnt).astype(np.int32)
        idx = np.empty(self.E, np.int32)
        fill = off[:-1].astype(np.int64).copy()
        for v in range(self.N):
            for e in range(self.pred_off[v], self.pred_off[v + 1]):
                u = self.pred_idx[e]
                idx[fill[u]] = v
                fill[u] += 1
        return off, idx

    def fits(self) -> np.ndarray:
        """bool [N][D]: peak memory within device capacity (placement sampling)."""
        return self.peak_mib.reshape(self.N, self.D) + int(self.margin_mib) <= self.cap_mib[None, :]

    def with_(self, **kw) -> "Problem":
        d = dict(self.__dict__)
        d.update(kw)
        return Problem(**d)


@dataclass
class Plans:
    """A batch of P plans; each array row is padded to a 16-byte stride."""
    P: int
    N: int
    place: np.ndarray         # uint8  [P][place_stride]
    order: np.ndarray         # uint16 [P][order_stride/2]; order[p][i] = node at position i
    fuse: np.ndarray          # uint32 [P][bits_stride/4]
    prefetch: np.ndarray      # uint32 [P][bits_stride/4]
    retain: np.ndarray | None  # uint32 [P][bits_stride/4] or None (= all retained)
    plan_base: int = 0

    @property
    def place_stride(self) -> int:
        return int(self.place.shape[1])

    @property
    def order_stride(self) -> int:
        return int(self.order.shape[1]) * 2

    @property
    def bits_stride(self) -> int:
        return int(self.fuse.shape[1]) * 4

    @staticmethod
    def empty(P: int, N: int, with_retain: bool = False) -> "Plans":
        words = (N + 31) // 32
        bs = _round16(4 * words)
        return Plans(P=P, N=N,
                     place=np.zeros((P, _round16(N)), np.uint8),
                     order=np.zeros((P, _round16(2 * N) // 2), np.uint16),
                     fuse=np.zeros((P, bs // 4), np.uint32),
                     prefetch=np.zeros((P, bs // 4), np.uint32),
                     retain=np.zeros((P, bs // 4), np.uint32) if with_retain else None)

    def slice(self, lo: int, hi: int) -> "Plans":
        return Plans(P=hi - lo, N=self.N, place=self.place[lo:hi], order=self.order[lo:hi],
                     fuse=self.fuse[lo:hi], prefetch=self.prefetch[lo:hi],
                     retain=None if self.retain is None else self.retain[lo:hi],
                     plan_base=self.plan_base + lo)

    def nbytes(self) -> int:
        n = self.place.nbytes + self.order.nbytes + self.fuse.nbytes + self.prefetch.nbytes
        return n + (0 if self.retain is None else self.retain.nbytes)


def _thresh(p: float) -> int:
    return int(round(min(max(p, 0.0), 1.0) * (1 << 32)))


def make_plans(prob: Problem, P: int, seed: int, plan_base: int = 0,
               p_fuse: float = 0.5, p_prefetch: float = 0.5,
               p_retain: float | None = None, threads: int | None = None) -> Plans:
    """Draw P plans: feasible uniform placements, random topological dispatch
    sequences, Bernoulli fusion / prefetch (/ retain) bits."""
    lib = _load()
    N = prob.N
    plans = Plans.empty(P, N, with_retain=p_retain is not None)
    plans.plan_base = plan_base
    succ_off, succ_idx = prob.succ_csr()
    indeg = np.diff(prob.pred_off).astype(np.int32)
    fits = prob.fits()
    feas_off = np.zeros(N + 1, np.int32)
    feas_off[1:] = np.cumsum(fits.sum(axis=1))
    if np.any(np.diff(feas_off) == 0):
        raise ValueError("a node fits on no device")
    feas_dev = np.nonzero(fits)[1].astype(np.uint8)
    if succ_idx.size == 0:
        succ_idx = np.zeros(1, np.int32)
    keep = (succ_off, succ_idx, indeg, feas_off, feas_dev)
    nthreads = threads or min(32, os.cpu_count() or 1)
    chunk = max(1, (P + nthreads * 4 - 1) // (nthreads * 4))

    def run(lo):
        hi = min(P, lo + chunk)
        rc = lib.wfg_make_plans(
            N, _ptr(succ_off), _ptr(succ_idx), _ptr(indeg), _ptr(feas_off), _ptr(feas_dev),
            seed, plan_base, lo, hi,
            _thresh(p_fuse), _thresh(p_prefetch), _thresh(p_retain or 0.0),
            _ptr(plans.place[lo:]), plans.place_stride,
            _ptr(plans.order[lo:]), plans.order_stride,
            _ptr(plans.fuse[lo:]), _ptr(plans.prefetch[lo:]),
            None if plans.retain is None else _ptr(plans.retain[lo:]),
            plans.bits_stride)
        if rc != 0:
            raise MemoryError("plan generator out of memory")

    starts = list(range(0, P, chunk))
    if len(starts) <= 1:
        for s in starts:
            run(s)
    else:
        with ThreadPoolExecutor(nthreads) as ex:
            list(ex.map(run, starts))
    del keep
    return plans


# ---------------------------------------------------------------------------
# DAG families (node lists of (role, local preds))
# ---------------------------------------------------------------------------

def fam_softdev(n: int):
    """planner -> coder -> tester -> (coder -> tester) x r -> reviewer chain."""
    if n < 4:
        raise ValueError("softdev needs >= 4 nodes")
    r = (n - 4) // 2
    roles = ["planner", "coder", "tester"] + ["coder", "tester"] * r
    roles += ["reviewer"] * (n - len(roles))
    return [(ro, [] if i == 0 else [i - 1]) for i, ro in enumerate(roles)]


def fam_research(n: int, width: int = 8):
    """planner -> k parallel researchers -> synthesizer -> reviewer chain."""
    if n < 4:
        raise ValueError("research needs >= 4 nodes")
    k = min(width, n - 3) if n <= width + 3 else width + (n - width - 3) // 2
    nodes = [("planner", [])]
    nodes += [("researcher", [0]) for _ in range(k)]
    nodes.append(("synthesizer", list(range(1, k + 1))))
    for _ in range(n - 2 - k):
        nodes.append(("reviewer", [len(nodes) - 1]))
    return nodes


def fam_layered(n: int, rng: np.random.Generator, width: int = 4):
    """Random layered DAG: layer widths in [1, width], 1-2 preds each from the
    previous layer.  Roles name the layer; models are tied per node below."""
    nodes = [("layer0", [])]
    prev = [0]
    layer = 1
    while len(nodes) < n:
        w = int(min(rng.integers(1, width + 1), n - len(nodes)))
        cur = []
        for _ in range(w):
            k = int(min(len(prev), rng.integers(1, 3)))
            preds = sorted(int(x) for x in rng.choice(prev, size=k, replace=False))
            cur.append(len(nodes))
            nodes.append((f"layer{layer}", preds))
        prev = cur
        layer += 1
    return nodes


# ---------------------------------------------------------------------------
# Problem assembly
# ---------------------------------------------------------------------------

@dataclass
class DeviceSpec:
    cap_gib: list
    speed: list          # run-time multiplier (smaller = faster)
    bw_gbps: list        # load bandwidth GB/s


def assemble(name: str, sessions: list, arrivals_us: np.ndarray, dev: DeviceSpec,
             weights_gib: list, rng: np.random.Generator, grant_us: int = 0,
             lat_median_us: float = 2e6, lat_sigma: float = 0.8,
             kv_lo: int = 256, kv_hi: int = 4096, tie_models: float = 0.5) -> Problem:
    """Build a Problem from per-session node lists.

    Run time L[n,d] = rint(base[n] * speed[d]) with base ~ lognormal(ln 2e6, 0.8)
    microseconds; peak[n,d] = weight[model[n]] + kv[n] MiB with kv ~ U{256..4096};
    load C[m,d] = floor(weight_MiB * 2^20 B / bw[d]) microseconds.  Models are
    drawn per (session, role); in layered DAGs a node keeps its first pred's
    model with probability ``tie_models`` (same-model edges make fusion possible).
    """
    D = len(dev.cap_gib)
    M = len(weights_gib)
    weight = np.array([int(round(g * GIB)) for g in weights_gib], np.int32)
    cap = np.array([int(round(g * GIB)) for g in dev.cap_gib], np.int32)
    max_kv = kv_hi
    fit_models = [m for m in range(M) if weight[m] + max_kv <= cap.max()]
    pred_lists, model, session = [], [], []
    base = 0
    for w, nodes in enumerate(sessions):
        role_model = {}
        local_model = []
        for i, (role, preds) in enumerate(nodes):
            if role.startswith("layer") and preds and rng.random() < tie_models:
                m = local_model[preds[0]]
            else:
                key = role if not role.startswith("layer") else (role, i)
                if key not in role_model:
                    role_model[key] = int(rng.choice(fit_models))
                m = role_model[key]
            local_model.append(m)
            pred_lists.append([base + p for p in preds])
            model.append(m)
            session.append(w)
        base += len(nodes)
    N = base
    pred_off = np.zeros(N + 1, np.int32)
    pred_off[1:] = np.cumsum([len(p) for p in pred_lists])
    pred_idx = np.array([u for p in pred_lists for u in p], np.int32)
    model = np.array(model, np.uint8)
    session = np.array(session, np.int32)
    lb = rng.lognormal(mean=math.log(lat_median_us), sigma=lat_sigma, size=N)
    speed = np.array(dev.speed, np.float64)
    lat = np.clip(np.rint(lb[:, None] * speed[None, :]), 1, 2**31 - 1).astype(np.int32)
    kv = rng.integers(kv_lo, kv_hi + 1, size=N).astype(np.int64)
    peak = (weight[model].astype(np.int64) + kv)[:, None] + np.zeros((1, D), np.int64)
    bw = np.array(dev.bw_gbps, np.int64)
    load = (weight.astype(np.int64)[:, None] * (1 << 20)) // (bw[None, :] * 1000)
    return Problem(N=N, D=D, M=M, W=len(sessions), pred_off=pred_off, pred_idx=pred_idx,
                   model=model, session=session, arrival_us=arrivals_us.astype(np.int64),
                   lat_us=lat.reshape(-1), peak_mib=peak.astype(np.int32).reshape(-1),
                   weight_mib=weight, load_us=load.astype(np.int32).reshape(-1),
                   cap_mib=cap, grant_us=grant_us, name=name)


def poisson_arrivals(W: int, mean_gap_s: float, rng: np.random.Generator) -> np.ndarray:
    """Session arrival offsets in microseconds; the first session arrives at 0."""
    gaps = rng.exponential(mean_gap_s, size=W)
    gaps[0] = 0.0
    return np.rint(np.cumsum(gaps) * 1e6).astype(np.int64)


def split_sizes(total: int, parts: int) -> list:
    q, r = divmod(total, parts)
    return [q + 1 if i < r else q for i in range(parts)]


def three_family_sessions(sizes: list, rng: np.random.Generator) -> list:
    fams = []
    for w, n in enumerate(sizes):
        f = w % 3
        if f == 0:
            fams.append(fam_softdev(n))
        elif f == 1:
            fams.append(fam_research(n))
        else:
            fams.append(fam_layered(n, rng))
    return fams


# ---------------------------------------------------------------------------
# Integer Box-Muller tables for the stochastic-latency workload
# ---------------------------------------------------------------------------

BM_N = 4096      # table length for the radius and the cosine tables
BM_RS = 4096     # radius scale
BM_CS = 16384    # cosine scale
BM_SHIFT = 18    # zq = floor(R*Cc / 2^18) ~ 256 * N(0,1)
BM_ZS = 256      # zq units per standard deviation
BM_SIGMA = 0.3   # log-latency standard deviation
BM_ES = 65536    # multiplier scale (16 fractional bits)


def box_muller_tables(sigma: float = BM_SIGMA):
    """Tables that turn a 64-bit hash into a lognormal latency multiplier.

    R[i] = rint(4096 sqrt(-2 ln((i+0.5)/4096))), Cc[j] = rint(16384 cos(2 pi j/4096)),
    so zq = floor(R[i] Cc[j] / 2^18) ~ 256 z with z ~ N(0,1) (Box and Muller 1958);
    E[k] = rint(65536 exp(sigma (k - ZOFF) / 256)) for k in [0, 2 ZOFF], with ZOFF
    the largest |zq| the two tables can produce.  The tables are data: both
    evaluators receive the same arrays.
    """
    i = np.arange(BM_N, dtype=np.float64)
    r = np.rint(BM_RS * np.sqrt(-2.0 * np.log((i + 0.5) / BM_N))).astype(np.int64)
    c = np.rint(BM_CS * np.cos(2.0 * np.pi * i / BM_N)).astype(np.int64)
    prod = int(np.abs(r).max()) * int(np.abs(c).max())
    zoff = -((-prod) >> BM_SHIFT)  # ceil(prod / 2^18)
    k = np.arange(2 * zoff + 1, dtype=np.float64)
    e = np.rint(BM_ES * np.exp(sigma * (k - zoff) / BM_ZS)).astype(np.int64)
    return r.astype(np.int32), c.astype(np.int32), e.astype(np.int32)


# ---------------------------------------------------------------------------
# The five named workloads
# ---------------------------------------------------------------------------

DEV_TINY = DeviceSpec([24, 48, 80], [1.0, 0.6, 0.4], [3, 6, 10])
DEV_MIX = DeviceSpec([24, 24, 32, 32, 48, 48, 80, 141],
                     [1.0, 1.0, 0.8, 0.8, 0.6, 0.6, 0.4, 0.3],
                     [3, 3, 3, 3, 6, 6, 10, 10])
DEV_BURST = DeviceSpec([24, 24, 48, 48, 80, 80, 141, 141],
                       [1.0, 1.0, 0.6, 0.6, 0.4, 0.4, 0.3, 0.3],
                       [3, 3, 6, 6, 10, 10, 10, 10])
DEV_LARGE = DeviceSpec([24] * 4 + [48] * 4 + [80] * 4 + [141] * 4,
                       [1.0] * 4 + [0.6] * 4 + [0.4] * 4 + [0.3] * 4,
                       [3] * 4 + [6] * 4 + [10] * 4 + [10] * 4)


@dataclass
class Workload:
    name: str
    problem: Problem
    P: int
    k: int
    plan_seed: int
    description: str


def config(name: str) -> Workload:
    """Build one of: tiny, mix, burst, stochastic, large."""
    if name == "tiny":
        rng = np.random.default_rng(0)
        nodes = [("planner", [])] + [("researcher", [0]) for _ in range(4)]
        nodes.append(("synthesizer", [1, 2, 3, 4]))
        nodes.append(("reviewer", [5]))
        for _ in range(5):
            nodes.append(("reviewer", [len(nodes) - 1]))
        prob = assemble("tiny", [nodes], np.zeros(1, np.int64), DEV_TINY, [6, 16, 28, 64], rng)
        return Workload("tiny", prob, 1024, 8, 1000,
                        "1 workflow, N=12 (planner -> 4 researchers -> synthesizer -> "
                        "6-reviewer chain), D=3, M=4, P=1024")
    if name == "mix":
        rng = np.random.default_rng(1)
        sess = []
        for w in range(16):
            f = w % 3
            sess.append(fam_softdev(8) if f == 0 else fam_research(11) if f == 1
                        else fam_layered(int(rng.integers(10, 15)), rng))
        prob = assemble("mix", sess, np.zeros(16, np.int64), DEV_MIX, [6, 8, 16, 28, 40, 64], rng)
        return Workload("mix", prob, 65536, 32, 1001,
                        f"16 workflows (softdev 8 / research 11 / layered), N={prob.N}, D=8, "
                        "M=6, burst arrivals, P=65536, k=32")
    if name == "burst":
        rng = np.random.default_rng(2)
        sess = three_family_sessions(split_sizes(2000, 64), rng)
        arr = poisson_arrivals(64, 0.5, rng)
        prob = assemble("burst", sess, arr, DEV_BURST, [3, 6, 8, 14, 16, 28, 40, 70], rng)
        return Workload("burst", prob, 16384, 32, 1002,
                        "64 sessions, Poisson arrivals (mean gap 0.5 s), N=2000, D=8, M=8, P=16384")
    if name == "stochastic":
        rng = np.random.default_rng(3)
        sess = three_family_sessions(split_sizes(500, 16), rng)
        arr = poisson_arrivals(16, 0.5, rng)
        prob = assemble("stochastic", sess, arr, DEV_BURST, [3, 6, 8, 14, 16, 28, 40, 70], rng)
        r, c, e = box_muller_tables()
        prob = prob.with_(S=64, seed=0x5EED0003, bm_r=r, bm_c=c, bm_e=e)
        return Workload("stochastic", prob, 8192, 32, 1003,
                        "16 sessions, N=500, D=8, M=8, P=8192 plans x S=64 latency samples")
    if name == "large":
        rng = np.random.default_rng(4)
        sess = three_family_sessions(split_sizes(8192, 256), rng)
        arr = poisson_arrivals(256, 0.5, rng)
        prob = assemble("large", sess, arr, DEV_LARGE,
                        [3, 4, 6, 8, 14, 16, 20, 28, 32, 40, 64, 70], rng)
        return Workload("large", prob, 131072, 64, 1004,
                        "256 sessions, N=8192, D=16, M=12, P=131072, k=64")
    raise KeyError(name)


CONFIG_NAMES = ("tiny", "mix", "burst", "stochastic", "large")
