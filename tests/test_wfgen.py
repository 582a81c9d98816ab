"""The synthetic inputs have the shapes the workloads name."""
import numpy as np
import pytest

import oracle
import wfgen


@pytest.mark.parametrize("name,N,D,M,W", [("tiny", 12, 3, 4, 1), ("mix", None, 8, 6, 16),
                                          ("burst", 2000, 8, 8, 64), ("stochastic", 500, 8, 8, 16),
                                          ("large", 8192, 16, 12, 256)])
def test_config_shapes(name, N, D, M, W):
    w = wfgen.config(name)
    p = w.problem
    assert (p.D, p.M, p.W) == (D, M, W)
    if N is not None:
        assert p.N == N
    else:
        assert 150 <= p.N <= 220
    assert p.pred_off[0] == 0 and p.pred_off[-1] == p.E
    assert set(np.unique(p.session)) == set(range(W))
    assert p.fits().any(axis=1).all()
    assert (p.peak_mib.reshape(p.N, p.D) >= p.weight_mib[p.model][:, None]).all()
    assert p.arrival_us[0] == 0 and (np.diff(p.arrival_us) >= 0).all()
    rel, comp = oracle.forecast(p)  # acyclic and feasible
    assert (comp > rel).all()


def test_tiny_shape_is_fanout_fanin_with_reviewer_chain():
    p = wfgen.config("tiny").problem
    preds = [p.pred_idx[p.pred_off[v]:p.pred_off[v + 1]].tolist() for v in range(p.N)]
    assert preds[:6] == [[], [0], [0], [0], [0], [1, 2, 3, 4]]
    assert preds[6:] == [[5], [6], [7], [8], [9], [10]]
    assert len(set(p.model[6:].tolist())) == 1


def test_plans_valid_and_chunk_independent():
    w = wfgen.config("mix")
    a = wfgen.make_plans(w.problem, 64, 9, threads=1)
    b = wfgen.make_plans(w.problem, 64, 9, threads=4)
    c = wfgen.make_plans(w.problem, 16, 9, plan_base=48)
    for x in ("place", "order", "fuse", "prefetch"):
        assert (getattr(a, x) == getattr(b, x)).all()
        assert (getattr(a, x)[48:] == getattr(c, x)).all()
    mk, p95, gpu, st = oracle.eval_plans(w.problem, a)
    assert (st == 0).all()
    assert a.place_stride % 16 == 0 and a.order_stride % 16 == 0 and a.bits_stride % 16 == 0


def test_placement_uniform_over_fitting_devices():
    w = wfgen.config("burst")
    p = w.problem
    pl = wfgen.make_plans(p, 2000, 3)
    fits = p.fits()
    n = int(np.argmax(fits.sum(axis=1)))
    cnt = np.bincount(pl.place[:, n], minlength=p.D)
    assert (cnt[~fits[n]] == 0).all()
    share = cnt[fits[n]] / cnt.sum()
    assert np.abs(share - 1 / fits[n].sum()).max() < 0.05


def test_bit_probabilities():
    w = wfgen.config("burst")
    pl = wfgen.make_plans(w.problem, 256, 5, p_fuse=0.25, p_prefetch=1.0, p_retain=0.0)
    N = w.problem.N
    bits = np.unpackbits(pl.fuse.view(np.uint8), bitorder="little").reshape(256, -1)[:, :N]
    assert abs(bits.mean() - 0.25) < 0.01
    pf = np.unpackbits(pl.prefetch.view(np.uint8), bitorder="little").reshape(256, -1)
    assert pf[:, :N].all() and not pf[:, N:].any()
    assert not pl.retain.any()


def test_box_muller_tables_deterministic():
    a = wfgen.box_muller_tables()
    b = wfgen.box_muller_tables()
    for x, y in zip(a, b):
        assert (x == y).all()
