"""Top-k on synthetic result arrays, on both of its paths (one CTA up to
16,384 plans, per-tile thresholds beyond): ties within and across tiles,
invalid plans, a short last tile, and k up to its limit.  The keys are written straight into the result
arrays, so only the top-k kernels run."""
import numpy as np
import pytest

import oracle
import wfgen
from gpu_util import lib

pytestmark = pytest.mark.gpu


def run_topk(mk, p95, gpu, st, k):
    import torch
    wf = lib()
    P = len(mk)
    ctx = wf.Ctx(wfgen.config("tiny").problem, max_P=P)
    res = wf.Results(P)
    res.makespan.copy_(torch.from_numpy(mk))
    res.p95.copy_(torch.from_numpy(p95))
    res.gpu.copy_(torch.from_numpy(gpu))
    res.status.copy_(torch.from_numpy(st.view(np.int32)))
    ids = torch.empty(k, dtype=torch.int32, device="cuda")
    keys = torch.empty((k, 3), dtype=torch.int64, device="cuda")
    wf.wf_topk(ctx, res, P, k, ids, keys)
    torch.cuda.synchronize()
    return ids.cpu().numpy(), keys.cpu().numpy()


@pytest.mark.parametrize("P,spread,bad", [
    (16385, 10**9, 0.0),      # one plan past the single-CTA path
    (40000, 50, 0.1),         # heavy ties: more candidates than a sorting tile
    (65536 + 17, 10**6, 0.5),  # a 17-plan last tile, half the plans invalid
    (200000, 3000, 0.02),
])
@pytest.mark.parametrize("k", [1, 32, 1024])
def test_large_batches(P, spread, bad, k):
    rng = np.random.default_rng(P + k)
    mk = rng.integers(1000, 1000 + spread, P).astype(np.int64)
    p95 = rng.integers(0, 20, P).astype(np.int64)
    gpu = rng.integers(0, 5, P).astype(np.int64)
    st = np.where(rng.random(P) < bad, rng.integers(1, 16, P), 0).astype(np.uint32)
    ids, keys = run_topk(mk, p95, gpu, st, k)
    want_ids, want_keys = oracle.topk(mk, p95, gpu, st, k)
    assert np.array_equal(ids, want_ids) and np.array_equal(keys, want_keys)


def test_best_plans_in_one_tile():
    """All of the k best plans sit in one tile: the other tiles' k-th keys
    are all worse, so the threshold comes from that tile alone."""
    P, k = 50000, 64
    rng = np.random.default_rng(3)
    mk = rng.integers(10**6, 2 * 10**6, P).astype(np.int64)
    mk[4096:4096 + 200] = rng.integers(0, 1000, 200)
    zeros = np.zeros(P, np.int64)
    st = np.zeros(P, np.uint32)
    ids, keys = run_topk(mk, zeros, zeros, st, k)
    want_ids, want_keys = oracle.topk(mk, zeros, zeros, st, k)
    assert np.array_equal(ids, want_ids) and np.array_equal(keys, want_keys)


def test_all_plans_invalid_and_tied():
    P, k = 30000, 1024
    mk = np.full(P, 7, np.int64)
    zeros = np.zeros(P, np.int64)
    st = np.ones(P, np.uint32)
    ids, keys = run_topk(mk, zeros, zeros, st, k)
    want_ids, want_keys = oracle.topk(mk, zeros, zeros, st, k)
    assert np.array_equal(ids, want_ids) and np.array_equal(keys, want_keys)


@pytest.mark.parametrize("P,k", [
    (1, 1), (63, 5), (1024, 1024), (1025, 1024), (1025, 1), (2049, 683),
    (16383, 128), (16384, 128), (16384, 129), (16384, 32), (9000, 200),
    (31, 31), (32, 32), (33, 32), (1024, 32), (1025, 32), (2048, 17), (5000, 32), (16384, 1), (16383, 31),
])
def test_single_cta_batches(P, k):
    """Batches up to the single-CTA limit, k from 1 to P: ties and invalid
    plans."""
    rng = np.random.default_rng(P * 7 + k)
    mk = rng.integers(1000, 1000 + max(P // 8, 2), P).astype(np.int64)
    p95 = rng.integers(0, 3, P).astype(np.int64)
    gpu = rng.integers(0, 2, P).astype(np.int64)
    st = np.where(rng.random(P) < 0.2, rng.integers(1, 16, P), 0).astype(np.uint32)
    ids, keys = run_topk(mk, p95, gpu, st, k)
    want_ids, want_keys = oracle.topk(mk, p95, gpu, st, k)
    assert np.array_equal(ids, want_ids) and np.array_equal(keys, want_keys)


def test_paths_alternate_on_one_context():
    """The single-CTA and threshold paths alternate on one context's top-k
    scratch."""
    import torch
    wf = lib()
    P = 40000
    rng = np.random.default_rng(11)
    mk = rng.integers(0, 5000, P).astype(np.int64)
    zeros = np.zeros(P, np.int64)
    st = np.zeros(P, np.uint32)
    ctx = wf.Ctx(wfgen.config("tiny").problem, max_P=P)
    res = wf.Results(P)
    res.makespan.copy_(torch.from_numpy(mk))
    res.p95.zero_()
    res.gpu.zero_()
    res.status.zero_()
    for n, k in [(16384, 32), (P, 32), (4000, 16), (16384, 500), (P, 7), (1500, 1000), (2, 2)]:
        ids = torch.empty(k, dtype=torch.int32, device="cuda")
        keys = torch.empty((k, 3), dtype=torch.int64, device="cuda")
        wf.wf_topk(ctx, res, n, k, ids, keys)
        torch.cuda.synchronize()
        want_ids, want_keys = oracle.topk(mk[:n], zeros[:n], zeros[:n], st[:n], k)
        assert np.array_equal(ids.cpu().numpy(), want_ids) and np.array_equal(keys.cpu().numpy(), want_keys)
    ctx.close()
