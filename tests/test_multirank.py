"""Multi-rank host logic on the CPU (gloo, world size 2).

Plans are independent, so several GPUs split a batch by plan: rank r takes
plans [r*P, (r+1)*P) with plan_base = r*P, and no collective runs while they
are evaluated.  These tests check, with the oracle standing in for each
rank's GPU, that the shards reproduce the whole batch (latency samples are
seeded by the global plan index), that the ranks' top-k lists merge into the
batch's top-k, and that bench.py's rank helpers and its reference arm work
under torch.distributed.
"""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

import oracle
import wfgen
from randprob import random_problem

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
WORLD = 2


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def stochastic_problem():
    rng = np.random.default_rng(808)
    prob = random_problem(rng, n_sessions=3, D=3)
    r, c, e = wfgen.box_muller_tables()
    return prob.with_(S=8, seed=12345, bm_r=r, bm_c=c, bm_e=e)


def merge_topk(parts, k):
    """The k best of the ranks' candidates by (invalid, makespan, p95, gpu,
    global plan id); an invalid plan carries INT64_MAX keys."""
    ids = np.concatenate([p[0] for p in parts]).astype(np.int64)
    keys = np.concatenate([p[1] for p in parts])
    big = np.iinfo(np.int64).max
    order = sorted(range(len(ids)), key=lambda j: (int(keys[j, 0]) == big, int(keys[j, 0]),
                                                   int(keys[j, 1]), int(keys[j, 2]), int(ids[j])))
    sel = order[:k]
    return ids[sel], keys[sel]


def _worker(rank, port, P, k, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(WORLD),
                      RANK=str(rank), LOCAL_RANK=str(rank), WF_BENCH_BACKEND="gloo")
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    r, world, _ = bench.dist_setup()
    assert (r, world) == (rank, WORLD)
    prob = stochastic_problem()
    plans = wfgen.make_plans(prob, P, 21, plan_base=rank * P, p_retain=0.5)
    mk, p95, gpu, st = oracle.eval_plans(prob, plans)
    ids, keys = oracle.topk(mk, p95, gpu, st, k, plan_base=rank * P)
    bench.barrier(world)
    slowest = bench.max_over_ranks(float(rank + 1), world)
    gathered = [None] * world
    dist.all_gather_object(gathered, {"metrics": [mk, p95, gpu, st], "ids": ids, "keys": keys})
    if rank == 0:
        np.save(os.path.join(out_dir, "slowest.npy"), np.array([slowest]))
        np.save(os.path.join(out_dir, "metrics.npy"),
                np.stack([np.concatenate([g["metrics"][i].astype(np.int64) for g in gathered])
                          for i in range(4)]))
        ids_m, keys_m = merge_topk([(g["ids"], g["keys"]) for g in gathered], k)
        np.save(os.path.join(out_dir, "merged_ids.npy"), ids_m)
        np.save(os.path.join(out_dir, "merged_keys.npy"), keys_m)
    dist.destroy_process_group()


def test_shards_reproduce_the_batch_and_merge_to_its_topk(tmp_path):
    P, k = 60, 9
    mp.start_processes(_worker, args=(free_port(), P, k, str(tmp_path)), nprocs=WORLD,
                       join=True, start_method="spawn")
    prob = stochastic_problem()
    whole = wfgen.make_plans(prob, WORLD * P, 21, p_retain=0.5)
    want = oracle.eval_plans(prob, whole)
    got = np.load(tmp_path / "metrics.npy")
    for i in range(4):
        assert np.array_equal(got[i], want[i].astype(np.int64))
    ids, keys = oracle.topk(*want, k)
    assert np.array_equal(np.load(tmp_path / "merged_ids.npy"), ids)
    assert np.array_equal(np.load(tmp_path / "merged_keys.npy"), keys)
    assert float(np.load(tmp_path / "slowest.npy")[0]) == float(WORLD)


def test_shard_rows_equal_the_batch_rows():
    prob = stochastic_problem()
    whole = wfgen.make_plans(prob, 50, 3, p_retain=0.5)
    part = wfgen.make_plans(prob, 20, 3, plan_base=30, p_retain=0.5)
    for a in ("place", "order", "fuse", "prefetch", "retain"):
        assert np.array_equal(getattr(whole, a)[30:], getattr(part, a))


def test_bench_reference_arm_under_torchrun():
    """bench.py --impl reference launched the way a multi-GPU run is: rank 0
    alone prints one JSON line, the other rank exits 0 without work."""
    env = dict(os.environ, WF_BENCH_BACKEND="gloo")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={WORLD}",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()),
           "bench.py", "--impl", "reference", "--gpus", str(WORLD), "--steps", "1", "--warmup", "0"]
    out = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    rec = json.loads(lines[0])
    assert rec["impl"] == "reference" and rec["n_gpus"] == WORLD and rec["value"] > 0
    assert rec["e2e"]["h2d_bytes_per_step"] == 0


if __name__ == "__main__":
    pytest.main([__file__, "-q"])
