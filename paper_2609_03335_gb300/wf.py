"""ctypes binding of libwf.so (include/wf.h): argument marshalling only.

The functions carry the C ABI's names.  Problem arrays are host numpy arrays;
plan, result and output arrays are device tensors (torch supplies device
memory and streams).  Every step of the evaluation runs in the library's CUDA
kernels; if the library is missing this module raises instead of falling
back to anything else.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libwf.so")

WF_OK, WF_EINVAL, WF_ENOMEM, WF_ECUDA, WF_ETIMEOUT = 0, 1, 2, 3, 4
ST_DEVICE, ST_CAPACITY, ST_PERMUTATION, ST_TOPOLOGY, ST_TABLES = 1, 2, 4, 8, 16
INT64_MAX = np.iinfo(np.int64).max

# Every entry point declared in include/wf.h.
EXPORTS = ("wf_problem_check", "wf_ctx_create", "wf_forecast_readiness", "wf_eval_plans",
           "wf_topk", "wf_ctx_status", "wf_ctx_destroy", "wf_strerror", "wf_last_error",
           "wf_eval_plans_static", "wf_mutate_plans", "wf_merge_elite", "wf_local_search",
           "wf_construct_plans", "wf_ctx_set_reclaim", "wf_ctx_check_wait_expiry", "wf_eval_plans_phi",
           "wf_topk_phi", "wf_static_status", "wf_ctx_set_eval_path",
           "wf_ctx_set_batch", "wf_eval_topk_host", "wf_ctx_reserve_host")


class WfError(RuntimeError):
    def __init__(self, code: int, where: str, detail: str = ""):
        super().__init__(f"{where}: {_strerror(code)} ({code}) {detail}".strip())
        self.code = code


class wf_problem(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int32), ("D", ctypes.c_int32), ("M", ctypes.c_int32),
                ("W", ctypes.c_int32),
                ("pred_off", ctypes.c_void_p), ("pred_idx", ctypes.c_void_p),
                ("model", ctypes.c_void_p), ("session", ctypes.c_void_p),
                ("arrival_us", ctypes.c_void_p), ("lat_us", ctypes.c_void_p),
                ("peak_mib", ctypes.c_void_p), ("weight_mib", ctypes.c_void_p),
                ("load_us", ctypes.c_void_p), ("cap_mib", ctypes.c_void_p),
                ("grant_us", ctypes.c_int32), ("S", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("bm_r", ctypes.c_void_p), ("bm_c", ctypes.c_void_p), ("bm_e", ctypes.c_void_p),
                ("bm_rn", ctypes.c_int32), ("bm_cn", ctypes.c_int32), ("bm_en", ctypes.c_int32),
                ("margin_mib", ctypes.c_int32)]


class wf_plans(ctypes.Structure):
    _fields_ = [("P", ctypes.c_int64), ("plan_base", ctypes.c_int64),
                ("place", ctypes.c_void_p), ("place_stride", ctypes.c_int64),
                ("order", ctypes.c_void_p), ("order_stride", ctypes.c_int64),
                ("fuse", ctypes.c_void_p), ("prefetch", ctypes.c_void_p),
                ("retain", ctypes.c_void_p), ("bits_stride", ctypes.c_int64)]


class wf_eval_out(ctypes.Structure):
    _fields_ = [("makespan_us", ctypes.c_void_p), ("p95_us", ctypes.c_void_p),
                ("gpu_us", ctypes.c_void_p), ("status", ctypes.c_void_p)]


_lib = None


def load_library():
    """Load libwf.so (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libwf.so not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    p, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    sig = {
        "wf_problem_check": ([p], ctypes.c_int),
        "wf_ctx_create": ([p, ctypes.c_int, i64, p], ctypes.c_int),
        "wf_forecast_readiness": ([p, p, p, p], ctypes.c_int),
        "wf_eval_plans": ([p, p, p, p], ctypes.c_int),
        "wf_topk": ([p, p, i64, i32, p, p, p], ctypes.c_int),
        "wf_eval_plans_phi": ([p, p, p, p, p, p], ctypes.c_int),
        "wf_topk_phi": ([p, p, p, p, i64, i32, p, p, p], ctypes.c_int),
        "wf_mutate_plans": ([p, p, p, ctypes.c_uint64, i64, i32, p], ctypes.c_int),
        "wf_merge_elite": ([p, p, p, p, p, p], ctypes.c_int),
        "wf_local_search": ([p, p, p, p, p, ctypes.c_uint64, i64, i32, i32, p], ctypes.c_int),
        "wf_construct_plans": ([p, p, ctypes.c_uint64, i64, p], ctypes.c_int),
        "wf_ctx_set_reclaim": ([p, i32], ctypes.c_int),
        "wf_ctx_status": ([p, p], ctypes.c_int),
        "wf_ctx_check_wait_expiry": ([p, p], ctypes.c_int),
        "wf_ctx_destroy": ([p], None),
        "wf_strerror": ([ctypes.c_int], ctypes.c_char_p),
        "wf_last_error": ([], ctypes.c_char_p),
        "wf_eval_plans_static": ([p, p, p, p], ctypes.c_int),
        "wf_static_status": ([p], ctypes.c_int),
        "wf_ctx_set_eval_path": ([p, i32], ctypes.c_int),
        "wf_ctx_set_batch": ([p, i32], ctypes.c_int),
        "wf_eval_topk_host": ([p, p, i32, p, p, p, p, p, p], ctypes.c_int),
        "wf_ctx_reserve_host": ([p], ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def _strerror(code: int) -> str:
    try:
        return load_library().wf_strerror(code).decode()
    except Exception:
        return "error"


def _check(code: int, where: str):
    if code != WF_OK:
        detail = load_library().wf_last_error().decode()
        raise WfError(code, where, detail)


def _stream_handle(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream or None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


class HostProblem:
    """A problem marshalled into a wf_problem (keeps the host arrays alive)."""

    def __init__(self, prob):
        def a(x, dt):
            return np.ascontiguousarray(np.asarray(x, dtype=dt))
        self.keep = dict(
            pred_off=a(prob.pred_off, np.int32), pred_idx=a(prob.pred_idx, np.int32),
            model=a(prob.model, np.uint8), session=a(prob.session, np.int32),
            arrival_us=a(prob.arrival_us, np.int64), lat_us=a(prob.lat_us, np.int32),
            peak_mib=a(prob.peak_mib, np.int32), weight_mib=a(prob.weight_mib, np.int32),
            load_us=a(prob.load_us, np.int32), cap_mib=a(prob.cap_mib, np.int32),
            bm_r=a(getattr(prob, "bm_r", np.zeros(0)), np.int32),
            bm_c=a(getattr(prob, "bm_c", np.zeros(0)), np.int32),
            bm_e=a(getattr(prob, "bm_e", np.zeros(0)), np.int32))
        k = self.keep
        ptr = {n: (v.ctypes.data if v.size else None) for n, v in k.items()}
        self.c = wf_problem(int(prob.N), int(prob.D), int(prob.M), int(prob.W),
                            ptr["pred_off"], ptr["pred_idx"], ptr["model"], ptr["session"],
                            ptr["arrival_us"], ptr["lat_us"], ptr["peak_mib"], ptr["weight_mib"],
                            ptr["load_us"], ptr["cap_mib"], int(prob.grant_us), int(prob.S),
                            int(prob.seed) & ((1 << 64) - 1), ptr["bm_r"], ptr["bm_c"], ptr["bm_e"],
                            int(k["bm_r"].size), int(k["bm_c"].size), int(k["bm_e"].size),
                            int(getattr(prob, "margin_mib", 0)))
        self.N, self.D, self.M, self.W, self.S = (int(prob.N), int(prob.D), int(prob.M),
                                                  int(prob.W), int(prob.S))


def wf_problem_check(prob) -> int:
    """Host-side validation; returns the WF_* code (no GPU needed)."""
    hp = prob if isinstance(prob, HostProblem) else HostProblem(prob)
    return int(load_library().wf_problem_check(ctypes.byref(hp.c)))


def wf_last_error() -> str:
    return load_library().wf_last_error().decode()


def wf_strerror(code: int) -> str:
    return _strerror(code)


class Ctx:
    """Owns a wf_ctx (device copy of one problem + scratch for max_P plans)."""

    def __init__(self, prob, max_P: int, device: int = 0):
        self.host = prob if isinstance(prob, HostProblem) else HostProblem(prob)
        self.max_P = int(max_P)
        self.device = int(device)
        self.ptr = ctypes.c_void_p()
        _check(load_library().wf_ctx_create(ctypes.byref(self.host.c), self.device, self.max_P,
                                            ctypes.byref(self.ptr)), "wf_ctx_create")
        reclaim = int(getattr(prob, "reclaim", 0))
        if reclaim:
            wf_ctx_set_reclaim(self, reclaim)
        batch = int(getattr(prob, "batch", 0))
        if batch:
            wf_ctx_set_batch(self, batch)

    @property
    def N(self):
        return self.host.N

    def close(self):
        if self.ptr:
            load_library().wf_ctx_destroy(self.ptr)
            self.ptr = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


RECLAIM_LRU, RECLAIM_NEXT_USE = 0, 1


def wf_ctx_set_reclaim(ctx: Ctx, policy: int):
    _check(load_library().wf_ctx_set_reclaim(ctx.ptr, int(policy)), "wf_ctx_set_reclaim")


def wf_ctx_create(prob, device: int = 0, max_P: int = 1) -> Ctx:
    return Ctx(prob, max_P, device)


def wf_ctx_destroy(ctx: Ctx):
    ctx.close()


def wf_ctx_status(ctx: Ctx, stream=None):
    _check(load_library().wf_ctx_status(ctx.ptr, _stream_handle(stream)), "wf_ctx_status")


PATH_AUTO, PATH_INT64, PATH_WIDE, PATH_RELATIVE = 0, 1, 2, 3


def wf_ctx_set_eval_path(ctx: Ctx, path: int):
    """PATH_AUTO (the sweeps), PATH_INT64 (every plan on the exact int64 path),
    PATH_WIDE (every plan starts in the 64-bit sweep) or PATH_RELATIVE (in the
    sweep with 32-bit times relative to a per-plan base)."""
    _check(load_library().wf_ctx_set_eval_path(ctx.ptr, int(path)), "wf_ctx_set_eval_path")


def wf_ctx_set_batch(ctx: Ctx, batch: int):
    """Replica batch limit B_q for later evaluations (0: one unit at a time per device)."""
    _check(load_library().wf_ctx_set_batch(ctx.ptr, int(batch)), "wf_ctx_set_batch")


def wf_ctx_check_wait_expiry(ctx: Ctx, stream=None):
    _check(load_library().wf_ctx_check_wait_expiry(ctx.ptr, _stream_handle(stream)), "wf_ctx_check_wait_expiry")


def wf_forecast_readiness(ctx: Ctx, rel, comp, stream=None):
    """rel, comp: device int64 tensors [N]."""
    _check(load_library().wf_forecast_readiness(ctx.ptr, rel.data_ptr(), comp.data_ptr(),
                                                _stream_handle(stream)), "wf_forecast_readiness")


class DevicePlans:
    """Plan arrays on the device (torch tensors) and their wf_plans view."""

    def __init__(self, place, order, fuse, prefetch, retain=None, plan_base: int = 0):
        self.place, self.order, self.fuse, self.prefetch, self.retain = place, order, fuse, prefetch, retain
        self.P = int(place.shape[0])
        self.plan_base = int(plan_base)

    @staticmethod
    def empty(P: int, N: int, with_retain: bool = False, device="cuda", plan_base: int = 0):
        """Uninitialised rows padded to 16 bytes."""
        import torch
        pad = lambda b: (b + 15) // 16 * 16
        words = pad(4 * ((N + 31) // 32)) // 4
        mk = lambda cols, dt: torch.empty((P, cols), dtype=dt, device=device)
        return DevicePlans(mk(pad(N), torch.uint8), mk(pad(2 * N) // 2, torch.int16), mk(words, torch.int32),
                           mk(words, torch.int32), mk(words, torch.int32) if with_retain else None,
                           plan_base=plan_base)

    def numpy(self, N: int):
        """Host copies of rows 0..P-1 without padding: place, order, fuse, prefetch, retain."""
        words = (N + 31) // 32
        out = [self.place[:, :N].cpu().numpy(), self.order[:, :N].cpu().numpy().view(np.uint16),
               self.fuse[:, :words].cpu().numpy().view(np.uint32),
               self.prefetch[:, :words].cpu().numpy().view(np.uint32)]
        out.append(None if self.retain is None else self.retain[:, :words].cpu().numpy().view(np.uint32))
        return out

    @staticmethod
    def host(plans, pin: bool = True):
        """The rows of a wfgen.Plans batch as host tensors (page-locked unless
        pin=False) for wf_eval_topk_host."""
        import torch

        def t(x):
            if x is None:
                return None
            h = torch.from_numpy(np.ascontiguousarray(x))
            return h.pin_memory() if pin else h
        return DevicePlans(t(plans.place), t(plans.order.view(np.int16)), t(plans.fuse.view(np.int32)),
                           t(plans.prefetch.view(np.int32)), t(None if plans.retain is None
                                                               else plans.retain.view(np.int32)),
                           plan_base=getattr(plans, "plan_base", 0))

    @staticmethod
    def from_host(plans, device="cuda", non_blocking=False):
        import torch

        def t(x):
            if x is None:
                return None
            h = torch.from_numpy(np.ascontiguousarray(x))
            return h.to(device, non_blocking=non_blocking)
        return DevicePlans(t(plans.place), t(plans.order.view(np.int16)), t(plans.fuse.view(np.int32)),
                           t(plans.prefetch.view(np.int32)), t(None if plans.retain is None
                                                               else plans.retain.view(np.int32)),
                           plan_base=getattr(plans, "plan_base", 0))

    def c(self, P: int | None = None, offset: int = 0) -> wf_plans:
        P = self.P - offset if P is None else P
        ps = self.place.stride(0)
        os_ = self.order.stride(0) * 2
        bs = self.fuse.stride(0) * 4
        return wf_plans(P, self.plan_base + offset,
                        self.place.data_ptr() + offset * ps, ps,
                        self.order.data_ptr() + offset * os_, os_,
                        self.fuse.data_ptr() + offset * bs, self.prefetch.data_ptr() + offset * bs,
                        None if self.retain is None else self.retain.data_ptr() + offset * bs, bs)


class Results:
    """Per-plan outputs on the device (or, with device="cpu", in host memory,
    page-locked unless pin=False, for wf_eval_topk_host)."""

    def __init__(self, P: int, device="cuda", pin: bool = True):
        import torch
        mk = lambda dt: torch.empty(P, dtype=dt, device=device)
        self.makespan, self.p95, self.gpu, self.status = (mk(torch.int64), mk(torch.int64), mk(torch.int64),
                                                          mk(torch.int32))
        if torch.device(device).type == "cpu" and pin:
            self.makespan, self.p95, self.gpu, self.status = (t.pin_memory() for t in
                                                              (self.makespan, self.p95, self.gpu, self.status))

    def c(self, offset: int = 0) -> wf_eval_out:
        return wf_eval_out(self.makespan.data_ptr() + 8 * offset, self.p95.data_ptr() + 8 * offset,
                           self.gpu.data_ptr() + 8 * offset, self.status.data_ptr() + 4 * offset)

    def numpy(self):
        return (self.makespan.cpu().numpy(), self.p95.cpu().numpy(), self.gpu.cpu().numpy(),
                self.status.cpu().numpy().view(np.uint32))


def wf_eval_topk_host(ctx: Ctx, plans: DevicePlans, k: int, ids, keys=None, out: Results | None = None,
                      rel=None, comp=None, stream=None):
    """One step from and to host memory: plans, ids [k] int32, keys [k, 3]
    int64, out (Results on "cpu") and the forecast rel / comp [N] int64 are
    HOST tensors (page-locked for overlap).  Asynchronous on `stream`: the
    results are there once the stream has passed the call."""
    pl = plans.c()
    oc = None if out is None else out.c()
    ptr = lambda t: None if t is None else t.data_ptr()
    _check(load_library().wf_eval_topk_host(ctx.ptr, ctypes.byref(pl), int(k), ptr(ids), ptr(keys),
                                            None if oc is None else ctypes.byref(oc), ptr(rel), ptr(comp),
                                            _stream_handle(stream)), "wf_eval_topk_host")


def wf_ctx_reserve_host(ctx: Ctx):
    _check(load_library().wf_ctx_reserve_host(ctx.ptr), "wf_ctx_reserve_host")


def wf_eval_plans(ctx: Ctx, plans: DevicePlans, out: Results, stream=None, P: int | None = None,
                  offset: int = 0):
    pl = plans.c(P, offset)
    oc = out.c(offset)
    _check(load_library().wf_eval_plans(ctx.ptr, ctypes.byref(pl), ctypes.byref(oc),
                                        _stream_handle(stream)), "wf_eval_plans")


def wf_topk(ctx: Ctx, res: Results, P: int, k: int, ids, keys=None, stream=None):
    """ids: device int32 [k]; keys: device int64 [k, 3] or None."""
    oc = res.c()
    _check(load_library().wf_topk(ctx.ptr, ctypes.byref(oc), int(P), int(k), ids.data_ptr(),
                                  None if keys is None else keys.data_ptr(), _stream_handle(stream)),
           "wf_topk")


def wf_eval_plans_phi(ctx: Ctx, plans: DevicePlans, out: Results, timely, life, stream=None):
    """wf_eval_plans plus Eq. 12's window terms; timely, life: device int64 [P]."""
    pl = plans.c(None, 0)
    oc = out.c(0)
    _check(load_library().wf_eval_plans_phi(ctx.ptr, ctypes.byref(pl), ctypes.byref(oc), timely.data_ptr(),
                                            life.data_ptr(), _stream_handle(stream)), "wf_eval_plans_phi")


def wf_topk_phi(ctx: Ctx, res: Results, timely, life, P: int, k: int, ids, keys=None, stream=None):
    """The k best by Eq. 12's window key; keys: device int64 [k, 3] (makespan, timely, life) or None."""
    oc = res.c()
    _check(load_library().wf_topk_phi(ctx.ptr, ctypes.byref(oc), timely.data_ptr(), life.data_ptr(), int(P),
                                      int(k), ids.data_ptr(), None if keys is None else keys.data_ptr(),
                                      _stream_handle(stream)), "wf_topk_phi")


def wf_mutate_plans(ctx: Ctx, parents: DevicePlans, children: DevicePlans, seed: int, round_: int,
                    n_ops: int, stream=None):
    pa, ch = parents.c(), children.c()
    _check(load_library().wf_mutate_plans(ctx.ptr, ctypes.byref(pa), ctypes.byref(ch), seed & ((1 << 64) - 1),
                                          int(round_), int(n_ops), _stream_handle(stream)), "wf_mutate_plans")


def wf_merge_elite(ctx: Ctx, elite: DevicePlans, elite_res: Results, children: DevicePlans,
                   child_res: Results, stream=None):
    el, er, ch, cr = elite.c(), elite_res.c(), children.c(), child_res.c()
    _check(load_library().wf_merge_elite(ctx.ptr, ctypes.byref(el), ctypes.byref(er), ctypes.byref(ch),
                                         ctypes.byref(cr), _stream_handle(stream)), "wf_merge_elite")


def wf_local_search(ctx: Ctx, elite: DevicePlans, elite_res: Results, children: DevicePlans,
                    child_res: Results, seed: int, round0: int, rounds: int, n_ops: int, stream=None):
    el, er, ch, cr = elite.c(), elite_res.c(), children.c(), child_res.c()
    _check(load_library().wf_local_search(ctx.ptr, ctypes.byref(el), ctypes.byref(er), ctypes.byref(ch),
                                          ctypes.byref(cr), seed & ((1 << 64) - 1), int(round0), int(rounds),
                                          int(n_ops), _stream_handle(stream)), "wf_local_search")


def wf_construct_plans(ctx: Ctx, out: DevicePlans, seed: int, jitter_us: int, stream=None):
    pl = out.c()
    _check(load_library().wf_construct_plans(ctx.ptr, ctypes.byref(pl), seed & ((1 << 64) - 1), int(jitter_us),
                                             _stream_handle(stream)), "wf_construct_plans")


def evaluate(ctx: Ctx, plans, k: int, stream=None):
    """End-to-end public call: host plans in (numpy / pinned), forecast, evaluation
    and top-k on the device, and the top-k ids and keys back on the host."""
    import torch
    dev = torch.device("cuda", ctx.device)
    dp = plans if isinstance(plans, DevicePlans) else DevicePlans.from_host(plans, dev, non_blocking=True)
    res = Results(dp.P, dev)
    rel = torch.empty(ctx.N, dtype=torch.int64, device=dev)
    comp = torch.empty_like(rel)
    ids = torch.empty(k, dtype=torch.int32, device=dev)
    keys = torch.empty((k, 3), dtype=torch.int64, device=dev)
    wf_forecast_readiness(ctx, rel, comp, stream)
    wf_eval_plans(ctx, dp, res, stream)
    wf_topk(ctx, res, dp.P, k, ids, keys, stream)
    return ids.cpu().numpy(), keys.cpu().numpy()


class DeviceProblem:
    """A problem whose tables already sit in device memory (torch tensors),
    viewed as a wf_problem of DEVICE pointers for wf_eval_plans_static."""

    def __init__(self, prob, device="cuda"):
        import torch
        hp = HostProblem(prob)
        self.tensors = {n: torch.from_numpy(v.view(np.int8) if v.dtype == np.uint8 else v).to(device)
                        for n, v in hp.keep.items() if v.size}
        ptr = {n: (self.tensors[n].data_ptr() if n in self.tensors else None) for n in hp.keep}
        self.c = wf_problem(hp.N, hp.D, hp.M, hp.W, ptr["pred_off"], ptr["pred_idx"], ptr["model"],
                            ptr["session"], ptr["arrival_us"], ptr["lat_us"], ptr["peak_mib"],
                            ptr["weight_mib"], ptr["load_us"], ptr["cap_mib"], int(prob.grant_us),
                            int(prob.S), int(prob.seed) & ((1 << 64) - 1), None, None, None, 0, 0, 0,
                            int(getattr(prob, "margin_mib", 0)))


def wf_eval_plans_static(prob: DeviceProblem, plans: DevicePlans, out: Results, stream=None):
    """wf_eval_plans without a context or any device allocation (deterministic
    problems; scratch in the library's static device array)."""
    pl = plans.c()
    oc = out.c()
    _check(load_library().wf_eval_plans_static(ctypes.byref(prob.c), ctypes.byref(pl), ctypes.byref(oc),
                                               _stream_handle(stream)), "wf_eval_plans_static")


def wf_static_status(stream=None):
    """Synchronize the stream and report (then clear) the device-side outcome
    of the last wf_eval_plans_static call on the current device."""
    _check(load_library().wf_static_status(_stream_handle(stream)), "wf_static_status")
