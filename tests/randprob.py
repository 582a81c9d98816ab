"""Small random problems for property tests (input data only)."""
import numpy as np

import wfgen


def random_problem(rng, n_sessions=4, sizes=(4, 9), D=3, M=4, tight=True, permute=True,
                   grant=None, arrivals=True, name="rand"):
    """Sessions from the three DAG families, random tables; tight capacities
    force reclamation; node ids optionally permuted so that index order is
    not a topological order."""
    sess = []
    for w in range(n_sessions):
        n = int(rng.integers(sizes[0], sizes[1] + 1))
        f = int(rng.integers(0, 3))
        sess.append(wfgen.fam_softdev(n) if f == 0 else wfgen.fam_research(n, width=3) if f == 1
                    else wfgen.fam_layered(n, rng, width=3))
    weights = [int(x) for x in rng.integers(5, 40, size=M)]
    wmax = max(weights) + 20
    caps = [int(x) for x in rng.integers(wmax, wmax * (2 if tight else 8), size=D)]
    dev = wfgen.DeviceSpec(cap_gib=[c / wfgen.GIB for c in caps],
                           speed=[float(x) for x in rng.uniform(0.5, 2.0, size=D)],
                           bw_gbps=[1] * D)
    arr = (np.sort(rng.integers(0, 500, size=n_sessions)) if arrivals
           else np.zeros(n_sessions, np.int64)).astype(np.int64)
    arr[0] = 0 if arrivals else arr[0]
    prob = wfgen.assemble(name, sess, arr, dev, [w / wfgen.GIB for w in weights], rng,
                          lat_median_us=100, lat_sigma=0.6, kv_lo=1, kv_hi=20)
    prob = prob.with_(load_us=rng.integers(0, 60, size=M * D).astype(np.int32),
                      grant_us=int(rng.integers(0, 5)) if grant is None else grant)
    # Some nodes infeasible on some devices: raise a random subset of peaks.
    peak = prob.peak_mib.reshape(prob.N, D).copy()
    for n in range(prob.N):
        if rng.random() < 0.3:
            d = int(rng.integers(0, D))
            if (peak[n] <= prob.cap_mib).sum() > 1:
                peak[n, d] = prob.cap_mib[d] + 1
    prob = prob.with_(peak_mib=peak.reshape(-1).astype(np.int32))
    if permute:
        prob = permute_nodes(prob, rng.permutation(prob.N))
    return prob


def permute_nodes(prob, perm):
    """Relabel node n as perm[n]."""
    N, D = prob.N, prob.D
    inv = np.argsort(perm)
    preds = [[int(perm[u]) for u in prob.pred_idx[prob.pred_off[inv[v]]:prob.pred_off[inv[v] + 1]]]
             for v in range(N)]
    off = np.zeros(N + 1, np.int32)
    off[1:] = np.cumsum([len(p) for p in preds])
    return prob.with_(pred_off=off, pred_idx=np.array([u for p in preds for u in p], np.int32),
                      model=prob.model[inv], session=prob.session[inv],
                      lat_us=prob.lat_us.reshape(N, D)[inv].reshape(-1),
                      peak_mib=prob.peak_mib.reshape(N, D)[inv].reshape(-1))


def preds_of(prob, v):
    return [int(u) for u in prob.pred_idx[prob.pred_off[v]:prob.pred_off[v + 1]]]
