"""Pins of the oracle's local search: the mutation operator and the elite merge.

The operator's draws come from SplitMix64 (pinned by its published vector in
test_oracle_stochastic.py); these tests pin what the draws are turned into:
children of valid plans stay valid (moves only to devices whose capacity holds
the activation, Eq. 8; swaps never cross a graph edge, Eq. 10), every child
is within n_ops changes of its parent, each change kind occurs at its rate,
and the merge keeps exactly the k smallest keys with stable slots.
"""
import numpy as np
import pytest

import oracle
import wfgen
from randprob import random_problem

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def parents_of(prob, P, seed, retain=False):
    return wfgen.make_plans(prob, P, seed, p_retain=0.5 if retain else None)


def rows_of(plans, idx, N):
    w = (N + 31) // 32
    return (plans.place[idx, :N], plans.order[idx, :N], plans.fuse[idx, :w], plans.prefetch[idx, :w])


def bits_differ(a, b, N):
    x = np.bitwise_xor(a.astype(np.uint64), b.astype(np.uint64))
    return sum(bin(int(v)).count("1") for v in x.ravel())


def test_zero_changes_copy_the_parents():
    rng = np.random.default_rng(1)
    prob = random_problem(rng, n_sessions=4, D=3)
    par = parents_of(prob, 5, 2, retain=True)
    ch = oracle.mutate(prob, par, 12, seed=9, round_=3, n_ops=0)
    N = prob.N
    for c in range(12):
        for a, b in zip(rows_of(par, c % 5, N), (ch.place[c], ch.order[c], ch.fuse[c], ch.prefetch[c])):
            assert np.array_equal(a, b)
        assert np.array_equal(par.retain[c % 5, :ch.retain.shape[1]], ch.retain[c])


@pytest.mark.parametrize("n_ops", [1, 4, 16])
def test_children_of_valid_plans_stay_valid_and_close(n_ops):
    for t in range(6):
        rng = np.random.default_rng(100 + t)
        prob = random_problem(rng, n_sessions=int(rng.integers(1, 6)), D=int(rng.integers(1, 5)))
        par = parents_of(prob, 7, t)
        ch = oracle.mutate(prob, par, 70, seed=1000 + t, round_=t, n_ops=n_ops)
        N = prob.N
        for c in range(70):
            assert oracle.status(prob, ch.place[c], ch.order[c]) == 0
            pp, po, pf, pr = rows_of(par, c % 7, N)
            assert sorted(ch.order[c].tolist()) == list(range(N))
            changes = (int((pp != ch.place[c]).sum()) + bits_differ(pf, ch.fuse[c], N) +
                       bits_differ(pr, ch.prefetch[c], N))
            moved = int((po != ch.order[c]).sum())
            assert changes + moved // 2 <= n_ops
            # the retain-less parents give retain-less children
            assert ch.retain is None


def test_change_kinds_occur_at_their_rates():
    """One change per child: a fuse or prefetch flip always changes one bit
    (1/4 each); a move or a swap may be a no-op (same device, or an edge)."""
    rng = np.random.default_rng(7)
    prob = random_problem(rng, n_sessions=5, D=4)
    par = parents_of(prob, 1, 3)
    C = 4000
    ch = oracle.mutate(prob, par, C, seed=77, round_=0, n_ops=1)
    N = prob.N
    pp, po, pf, pr = rows_of(par, 0, N)
    fuse = sum(bits_differ(pf, ch.fuse[c], N) for c in range(C))
    pref = sum(bits_differ(pr, ch.prefetch[c], N) for c in range(C))
    move = int(sum((pp != ch.place[c]).any() for c in range(C)))
    swap = int(sum((po != ch.order[c]).any() for c in range(C)))
    sd = np.sqrt(C * 0.25 * 0.75)
    assert abs(fuse - C / 4) < 5 * sd and abs(pref - C / 4) < 5 * sd
    assert 0 < move <= C / 4 + 5 * sd and 0 < swap <= C / 4 + 5 * sd
    assert fuse + pref + move + swap <= C


def test_swaps_never_cross_an_edge():
    """A single chain has exactly one topological order: no swap applies."""
    N = 9
    prob = wfgen.Problem(N=N, D=2, M=1, W=1, pred_off=np.r_[0, np.arange(N)].astype(np.int32),
                         pred_idx=np.arange(N - 1, dtype=np.int32), model=np.zeros(N, np.uint8),
                         session=np.zeros(N, np.int32), arrival_us=np.zeros(1, np.int64),
                         lat_us=np.full(2 * N, 5, np.int32), peak_mib=np.full(2 * N, 3, np.int32),
                         weight_mib=np.array([2], np.int32), load_us=np.array([4, 4], np.int32),
                         cap_mib=np.array([8, 8], np.int32))
    par = parents_of(prob, 2, 1)
    ch = oracle.mutate(prob, par, 400, seed=5, round_=1, n_ops=8)
    assert (ch.order == np.arange(N, dtype=np.uint16)).all()


def test_moves_land_uniformly_on_fitting_devices():
    """Activation 0 fits devices {1, 3, 4} only; moves of it spread evenly over them."""
    N, D = 1, 5
    peak = np.array([9, 3, 9, 3, 3], np.int32)
    prob = wfgen.Problem(N=N, D=D, M=1, W=1, pred_off=np.zeros(2, np.int32), pred_idx=np.zeros(0, np.int32),
                         model=np.zeros(1, np.uint8), session=np.zeros(1, np.int32),
                         arrival_us=np.zeros(1, np.int64), lat_us=np.full(D, 5, np.int32), peak_mib=peak,
                         weight_mib=np.array([2], np.int32), load_us=np.full(D, 4, np.int32),
                         cap_mib=np.full(D, 4, np.int32))
    par = parents_of(prob, 1, 1)
    ch = oracle.mutate(prob, par, 6000, seed=11, round_=0, n_ops=1)
    counts = np.bincount(ch.place[:, 0], minlength=D)
    assert counts[0] == counts[2] == 0
    moves = 6000 / 4
    for d in (1, 3, 4):
        # moves landing on d, plus the children whose change was not a move
        # and kept the parent's device
        extra = 6000 - moves if d == par.place[0, 0] else 0
        assert abs(counts[d] - extra - moves / 3) < 6 * np.sqrt(moves / 3)


def test_rounds_and_children_draw_independently():
    rng = np.random.default_rng(5)
    prob = random_problem(rng, n_sessions=4, D=3)
    par = parents_of(prob, 1, 2)
    a = oracle.mutate(prob, par, 50, seed=3, round_=0, n_ops=2)
    b = oracle.mutate(prob, par, 50, seed=3, round_=1, n_ops=2)
    c = oracle.mutate(prob, par, 50, seed=4, round_=0, n_ops=2)
    same_ab = sum(np.array_equal(a.place[i], b.place[i]) and np.array_equal(a.order[i], b.order[i]) and
                  np.array_equal(a.fuse[i], b.fuse[i]) and np.array_equal(a.prefetch[i], b.prefetch[i])
                  for i in range(50))
    same_ac = sum(np.array_equal(a.fuse[i], c.fuse[i]) and np.array_equal(a.prefetch[i], c.prefetch[i]) and
                  np.array_equal(a.place[i], c.place[i]) and np.array_equal(a.order[i], c.order[i])
                  for i in range(50))
    assert same_ab < 25 and same_ac < 25
    # distinct children of one parent differ from each other
    assert len({(a.place[i].tobytes(), a.order[i].tobytes(), a.fuse[i].tobytes(), a.prefetch[i].tobytes())
                for i in range(50)}) > 25


def test_merge_keeps_the_k_best_with_stable_slots():
    rng = np.random.default_rng(9)
    for t in range(30):
        k, C = int(rng.integers(1, 12)), int(rng.integers(0, 30))

        def metrics(n):
            st = (rng.random(n) < 0.2).astype(np.uint32) * 4
            mk = rng.integers(0, 6, n).astype(np.int64)
            p95 = rng.integers(0, 3, n).astype(np.int64)
            gpu = rng.integers(0, 3, n).astype(np.int64)
            big = np.iinfo(np.int64).max
            for a in (mk, p95, gpu):
                a[st != 0] = big
            return [mk, p95, gpu, st]

        el, chm = metrics(k), metrics(C)
        pairs, new = oracle.merge_elite(el, chm, k)
        union = [np.concatenate([a, b]) for a, b in zip(el, chm)]
        idx = np.arange(k + C)
        best = np.lexsort((idx, union[2], union[1], union[0], union[3] != 0))[:k]
        want = sorted(zip((union[3][best] != 0).tolist(), union[0][best].tolist(), union[1][best].tolist(),
                          union[2][best].tolist()))
        got = sorted(zip((new[3] != 0).tolist(), new[0].tolist(), new[1].tolist(), new[2].tolist()))
        assert got == want
        kept = set(int(i) for i in best if i < k)
        assert [s for s, _ in pairs] == [s for s in range(k) if s not in kept]
        assert [c for _, c in pairs] == [int(i) - k for i in best if i >= k]
        for s in kept:
            assert all(new[a][s] == el[a][s] for a in range(4))


def test_local_search_never_loses_its_best_plan():
    w = wfgen.config("tiny")
    prob = w.problem
    k = 6
    elite = parents_of(prob, k, 4)
    met = list(oracle.eval_plans(prob, elite))
    start = min(zip(met[0].tolist(), met[1].tolist(), met[2].tolist()))
    rows, new = oracle.local_search(prob, elite, met, n_children=48, seed=21, round0=0, rounds=4, n_ops=3)
    end = min(zip(new[0].tolist(), new[1].tolist(), new[2].tolist()))
    assert end <= start
    again = oracle.eval_plans(prob, rows)
    for a in range(4):
        assert np.array_equal(again[a], new[a])
    # with no changes every child copies a parent: the elite only ever holds
    # copies of the starting rows, and its best key stays
    rows0, new0 = oracle.local_search(prob, elite, met, n_children=12, seed=21, round0=0, rounds=2, n_ops=0)
    N = prob.N
    starts = {(elite.place[i, :N].tobytes(), elite.order[i, :N].tobytes()) for i in range(k)}
    assert all((rows0.place[i].tobytes(), rows0.order[i].tobytes()) in starts for i in range(k))
    assert min(zip(new0[0].tolist(), new0[1].tolist(), new0[2].tolist())) == start
