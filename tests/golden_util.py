"""Loader for the hand-worked fixtures under tests/golden/."""
import json
import os

import numpy as np

import wfgen

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def fixture_names():
    return sorted(f[:-5] for f in os.listdir(GOLDEN) if f.startswith("t") and f.endswith(".json"))


def load(name):
    with open(os.path.join(GOLDEN, name + ".json")) as f:
        return json.load(f)


def problem_of(fx, case=None):
    pb = fx["problem"]
    nodes = pb["nodes"]
    N, D = len(nodes), pb["D"]
    off = np.zeros(N + 1, np.int32)
    off[1:] = np.cumsum([len(n["preds"]) for n in nodes])
    lat = np.array([n["lat"] for n in nodes], np.int32)
    peak = np.array([n["peak"] for n in nodes], np.int32)
    grant = pb["grant"]
    cap = pb["cap"]
    batch = pb.get("batch", 0)
    if case is not None:
        if "patch_peak" in case:
            peak = np.array(case["patch_peak"], np.int32)
        if "patch_grant" in case:
            grant = case["patch_grant"]
        if "patch_cap" in case:
            cap = case["patch_cap"]
        if "patch_batch" in case:
            batch = case["patch_batch"]
    return wfgen.Problem(
        N=N, D=D, M=pb["M"], W=pb["W"], pred_off=off,
        pred_idx=np.array([u for n in nodes for u in n["preds"]], np.int32),
        model=np.array([n["model"] for n in nodes], np.uint8),
        session=np.array([n["session"] for n in nodes], np.int32),
        arrival_us=np.array(pb["arrival"], np.int64),
        lat_us=lat.reshape(-1), peak_mib=peak.reshape(-1),
        weight_mib=np.array(pb["weight"], np.int32),
        load_us=np.array(pb["load"], np.int32).reshape(-1),
        cap_mib=np.array(cap, np.int32), grant_us=grant, name=fx["name"], batch=batch)


def set_bits(row, nodes):
    for n in nodes:
        row[n >> 5] |= np.uint32(1 << (n & 31))


def plans_of(fx, cases):
    """One plan per case (rows in case order)."""
    N = len(fx["problem"]["nodes"])
    with_retain = any(c.get("retain_off") is not None for c in cases)
    pl = wfgen.Plans.empty(len(cases), N, with_retain=with_retain)
    for r, c in enumerate(cases):
        pl.place[r, :N] = c["place"]
        pl.order[r, :N] = c["order"]
        set_bits(pl.fuse[r], c["fuse"])
        set_bits(pl.prefetch[r], c["prefetch"])
        if with_retain:
            set_bits(pl.retain[r], [n for n in range(N) if n not in (c.get("retain_off") or [])])
    return pl
