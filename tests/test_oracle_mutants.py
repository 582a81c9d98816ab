"""The pins catch plausible mistakes.

Each mutant is a copy of the oracle's C source with one planted mistake (a
dropped term, a wrong comparison, a wrong index, a wrong rounding ...),
compiled on the CPU.  The golden, property and stochastic pin suites run
against every mutant and must fail.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "wf_oracle.c")

MUTANTS = {
    "drop_grant": ("start += pb->grant;", "start += 0;"),
    "prefetch_waits_for_release": ("bit_of(prefetch, h) ? imax64(t_free[d], pb->arrival[w])",
                                   "bit_of(prefetch, h) ? imax64(t_free[d], rel)"),
    "evict_most_recent": ("st[k] < st[victim]", "st[k] > st[victim]"),
    "no_check_on_hit": ("const int64_t need = hit ? kv_adm :", "const int64_t need = hit ? 0 :"),
    "kv_of_head_only": ("kv_adm = imax64(kv_adm, (int64_t)pb->peak[(int64_t)chain[j] * D + d] - pb->weight[m]);",
                        "kv_adm = (int64_t)pb->peak[(int64_t)chain[0] * D + d] - pb->weight[m];"),
    "fuse_ignores_device": (" || place[s] != place[h]", ""),
    "fuse_ignores_bit": ("!bit_of(fuse, s) || ", ""),
    "release_ignores_arrival": ("int64_t rel = pb->arrival[w];", "int64_t rel = 0;"),
    "p95_rank_floor": ("(q * n + 99) / 100", "(q * n) / 100"),
    "makespan_from_zero": ("*makespan = end - first;", "*makespan = end;"),
    "gpu_no_tail": ("gpu[d] += end - occ_since[d];", "gpu[d] += 0;"),
    "occupancy_from_load_end": ("if (occ_since[d] == ORC_NONE) occ_since[d] = ls;",
                                "if (occ_since[d] == ORC_NONE) occ_since[d] = ls + pb->load[(int64_t)m * D + d];"),
    "retain_ignored": ("if (retain && !bit_of(retain, last))", "if (0)"),
    "retain_bit_of_head": ("!bit_of(retain, last)", "!bit_of(retain, h)"),
    "always_load": ("const int hit = st[m] != 0;", "const int hit = 0;"),
    "hit_ignores_device_queue": ("start = imax64(t_free[d], rel);", "start = rel;"),
    "topo_check_reversed": ("if (pos[pb->pred_idx[e]] > pos[v]) st |= 8u;",
                            "if (pos[pb->pred_idx[e]] < pos[v]) st |= 8u;"),
    "forecast_first_feasible": ("if (pb->peak[(int64_t)n * D + d] <= pb->cap[d]) lmin = imin64(lmin, pb->lat[(int64_t)n * D + d]);",
                                "if (pb->peak[(int64_t)n * D + d] <= pb->cap[d] && lmin == ORC_INF) lmin = pb->lat[(int64_t)n * D + d];"),
    "fusion_ignores_model": (" && pb->model[u] == pb->model[v]", ""),
    "z_truncates": ("if (prod % 262144 != 0 && prod < 0) zq -= 1;", ""),
    "multiplier_no_rounding": ("(base * mult + 32768) >> 16", "(base * mult) >> 16"),
    "angle_from_low_bits": ("(h >> 32) & (uint64_t)(pb->bm_cn - 1)", "h & (uint64_t)(pb->bm_cn - 1)"),
    "hash_nests_sample_first": ("orc_splitmix64(orc_splitmix64(orc_splitmix64(pb->seed ^ plan) ^ sample) ^ node)",
                                "orc_splitmix64(orc_splitmix64(orc_splitmix64(pb->seed ^ sample) ^ plan) ^ node)"),
    "radius_from_bits_12": ("(int64_t)(h & (uint64_t)(pb->bm_rn - 1))", "(int64_t)((h >> 12) & (uint64_t)(pb->bm_rn - 1))"),
    "batch_admits_out_of_order": ("adm = imax64(imax64(rel, se[slot]), last_adm[d]);", "adm = imax64(rel, se[slot]);"),
    "batch_ignores_running_kv": ("if (se[j] > adm) running += sk[j];", "if (0) running += sk[j];"),
    "batch_latest_slot": ("if (se[j] < se[slot]) slot = j;", "if (se[j] > se[slot]) slot = j;"),
    "batch_switch_without_drain": ("for (int32_t j = 0; j < B; ++j) drain = imax64(drain, se[j]);",
                                   "for (int32_t j = 0; j < B; ++j) drain = imin64(drain, se[j]);"),
    "batch_other_slots_free_before_load": ("for (int32_t j = 0; j < B; ++j) { se[j] = ready; sk[j] = 0; }",
                                           "for (int32_t j = 0; j < B; ++j) { se[j] = drain; sk[j] = 0; }"),
    "mean_rounds_up": ("out3[0] = sum_mk / S;", "out3[0] = (sum_mk + S - 1) / S;"),
    "device_free_at_head_end": ("t_free[d] = c[last];", "t_free[d] = c[h];"),
    "hash_ignores_plan": ("orc_splitmix64(pb->seed ^ plan)", "orc_splitmix64(pb->seed)"),
    "evict_when_exactly_full": ("while (used[d] + need > pb->cap[d])", "while (used[d] + need >= pb->cap[d])"),
    "status_place_ge": ("if (place[n] >= D) st |= 1u;", "if (place[n] > D) st |= 1u;"),
    "release_ignores_preds": ("rel = imax64(rel, c[pb->pred_idx[e]]);", "rel = imax64(rel, 0);"),
    "chain_reuses_start": ("t += L[(int64_t)n * D + d];", "t = start + L[(int64_t)n * D + d];"),
    "swap_crosses_edges": ("if (v < N && !(u < N && is_pred(pb, u, v)))", "if (v < N)"),
    "move_ignores_capacity": ("if (pb->peak[(int64_t)n * D + d] <= pb->cap[d] && r-- == 0)", "if (r-- == 0)"),
    "child_of_wrong_parent": ("const int64_t p = c % n_parents;", "const int64_t p = (c / 2) % n_parents;"),
    "construct_rank_ignores_release": ("rank[y] = r + (jitter", "rank[y] = 0 + (jitter"),
    "construct_binding_ignores_residency": ("if (stamp[(int64_t)dd * M + m] != 0) {", "if (0) {"),
    "construct_prefetch_always": ("const int pf = !hit && t_free[d] < rel[u];", "const int pf = !hit;"),
    "next_use_ignores_redundancy": ("else if (red != best_red) better = red > best_red;", "else if (0) better = 0;"),
    "next_use_ignores_cost": ("else if (!inf && dist * best_cost != best_dist * cost) better = dist * best_cost > best_dist * cost;",
                              "else if (!inf && dist != best_dist) better = dist > best_dist;"),
    "next_use_nearest_first": ("better = dist * best_cost > best_dist * cost;", "better = dist * best_cost < best_dist * cost;"),
    "construct_no_fusion": ("s >= 0 && pb->peak[(int64_t)s * D + d] <= pb->cap[d]; s = fnext[s])",
                            "s >= 0 && 0; s = fnext[s])"),
}

PIN_FILES = ["tests/test_oracle_golden.py", "tests/test_oracle_properties.py",
             "tests/test_oracle_stochastic.py", "tests/test_oracle_search.py", "tests/test_oracle_construct.py",
             "tests/test_oracle_reclaim.py", "tests/test_oracle_batch.py"]


def _run_mutant(name, tmp):
    """A site that simulate_batched repeats (the same step of the play) is
    mutated at its first occurrence, which lies in simulate; the batched copy
    is pinned against simulate by the B_q = 1 test.  Every other site is
    unique."""
    old, new = MUTANTS[name]
    src = open(SRC).read()
    n = src.count(old)
    assert n >= 1, f"mutation site for {name} not found"
    if n > 1:
        assert src.index(old) < src.index("static int simulate_batched("), f"site for {name} not in simulate"
        assert n == 1 + src[src.index("static int simulate_batched("):].count(old), f"site for {name} not unique"
    path = os.path.join(tmp, f"{name}.c")
    with open(path, "w") as f:
        f.write(src.replace(old, new, 1))
    lib = os.path.join(tmp, f"lib{name}.so")
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", lib, path])
    env = dict(os.environ, WF_ORACLE_LIB=lib)
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", *PIN_FILES],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return name, r.returncode


def test_every_planted_mistake_is_caught(tmp_path):
    with ThreadPoolExecutor(min(8, os.cpu_count() or 1)) as ex:
        results = list(ex.map(lambda n: _run_mutant(n, str(tmp_path)), MUTANTS))
    survivors = [n for n, rc in results if rc == 0]
    assert not survivors, f"mutants not caught by any pin: {survivors}"


def test_unmutated_oracle_passes_the_pins(tmp_path):
    lib = os.path.join(str(tmp_path), "libclean.so")
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", lib, SRC])
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", *PIN_FILES],
                       cwd=ROOT, env=dict(os.environ, WF_ORACLE_LIB=lib), capture_output=True, text=True)
    assert r.returncode == 0, r.stdout[-2000:]
