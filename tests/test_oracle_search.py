"""Pins of the oracle's search against what the paper and plain mathematics fix.

* ranking == an fp64 numpy sort of query-centroid inner products (Sec. 2.3);
* nprobe = nlist with W = infinity == exhaustive filtered top-k (Sec. 6.1),
  computed here with numpy, independently of the oracle's C code;
* W >= nprobe == fixed-probe IVF over the union of the first nprobe lists;
* sequential == lookahead under 32 seeded completion orders (Sec. 4.3);
* probes == the stop-line fixed point of each query's hit pattern;
* probes and retained fixed-probe neighbours are non-decreasing in W (App. A);
* hand-built indexes with exactly representable scores fix the tau boundary
  (sim >= tau qualifies, Sec. 2.2), self exclusion, the id tie-break, padding,
  physically empty partitions, and the Fig. 4 walk end to end.
"""
import numpy as np
import pytest

import oracle
from conftest import index_of
from test_oracle_stopping import stop_line_fixed_point


def np_rank(Q, C, nprobe):
    S = Q.astype(np.float64) @ C.astype(np.float64).T
    out = np.empty((Q.shape[0], nprobe), np.int32)
    cid = np.arange(C.shape[0])
    for i in range(Q.shape[0]):
        out[i] = np.lexsort((cid, -S[i]))[:nprobe]
    return out


def np_filtered_topk(X, ids, Q, qids, tau, k, rows=None):
    """Exhaustive filtered top-k with numpy fp64 (score desc, id asc)."""
    res_ids = np.full((Q.shape[0], k), -1, np.int64)
    res_sc = np.full((Q.shape[0], k), -np.inf)
    cnt = np.zeros(Q.shape[0], np.int32)
    for i in range(Q.shape[0]):
        R = np.arange(X.shape[0]) if rows is None else rows[i]
        s = X[R].astype(np.float64) @ Q[i].astype(np.float64)
        keep = (s >= np.float64(np.float32(tau))) & (ids[R] != qids[i])
        s, rid = s[keep], ids[R][keep]
        o = np.lexsort((rid, -s))[:k]
        cnt[i] = len(o)
        res_ids[i, :len(o)] = rid[o]
        res_sc[i, :len(o)] = s[o]
    return res_ids, res_sc, cnt


def test_rank_matches_numpy_sort(tiny):
    order, sc = oracle.rank(tiny["Q"][:300], tiny["centroids"], 16, return_scores=True)
    ref = np_rank(tiny["Q"][:300], tiny["centroids"], 16)
    assert (order == ref).all()
    assert (np.diff(sc, axis=1) <= 0).all()


def test_full_probe_equals_bruteforce(deep):
    cfg = deep["cfg"]
    nq = 120
    Q, qids = deep["Q"][:nq], deep["qids"][:nq]
    r = oracle.search(index_of(deep), Q, cfg.tau, cfg.k, cfg.nlist, 2**40, qids=qids)
    assert (r["probes"] == cfg.nlist).all()
    ids, sc, cnt = np_filtered_topk(deep["X"], deep["ids"], Q, qids, cfg.tau, cfg.k)
    assert (r["count"] == cnt).all()
    assert (r["ids"] == ids).all()
    np.testing.assert_allclose(r["scores"], sc, rtol=0, atol=1e-12)
    bf = oracle.bruteforce(deep["X"], deep["ids"], Q, cfg.tau, cfg.k, qids=qids)
    assert (bf["ids"] == ids).all() and (bf["count"] == cnt).all()


@pytest.mark.parametrize("W", [16, 17, 2**31 - 1])
def test_window_at_least_nprobe_is_fixed_probe(tiny, W):
    cfg = tiny["cfg"]
    Q, qids = tiny["Q"][:200], tiny["qids"][:200]
    r = oracle.search(index_of(tiny), Q, cfg.tau, cfg.k, cfg.nprobe, W, qids=qids)
    assert (r["probes"] == cfg.nprobe).all()
    order = oracle.rank(Q, tiny["centroids"], cfg.nprobe)
    fp = oracle.fixed_probe(index_of(tiny), Q, cfg.tau, cfg.k, cfg.nprobe, order, qids=qids)
    assert (fp["ids"] == r["ids"]).all() and (fp["count"] == r["count"]).all()
    part_rows = [np.flatnonzero(np.isin(tiny["assign"], order[i])) for i in range(len(Q))]
    ids, sc, cnt = np_filtered_topk(tiny["X"], tiny["ids"], Q, qids, cfg.tau, cfg.k, part_rows)
    assert (r["ids"] == ids).all() and (r["count"] == cnt).all()


def test_lookahead_equals_sequential(deep, tiny):
    for w in (deep, tiny):
        cfg = w["cfg"]
        seq = oracle.search(index_of(w), w["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                            qids=w["qids"])
        for seed in range(32):
            la = oracle.search(index_of(w), w["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                               qids=w["qids"], mode="lookahead", seed=seed)
            for key in ("ids", "scores", "count", "probes"):
                assert (la[key] == seq[key]).all(), (key, seed)


def test_probes_follow_hit_pattern(deep):
    cfg = deep["cfg"]
    order = oracle.rank(deep["Q"], deep["centroids"], cfg.nprobe)
    hits = oracle.hit_matrix(index_of(deep), deep["Q"], cfg.tau, cfg.nprobe, order,
                             qids=deep["qids"])
    assert hits[:, 1:].any(), "workload must hit beyond rank 1 to exercise the stop line"
    for W in (1, 2, 3, 5):
        r = oracle.search(index_of(deep), deep["Q"], cfg.tau, cfg.k, cfg.nprobe, W,
                          qids=deep["qids"], order=order)
        expect = [stop_line_fixed_point(hits[i].tolist(), W) for i in range(len(hits))]
        assert (r["probes"] == np.array(expect)).all()
        # a query has a result iff some searched partition hit
        searched_hit = np.array([hits[i, :r["probes"][i]].any() for i in range(len(hits))])
        assert ((r["count"] > 0) == searched_hit).all()


def test_monotone_in_window(deep):
    cfg = deep["cfg"]
    fixed = oracle.search(index_of(deep), deep["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.nprobe,
                          qids=deep["qids"])
    prev_p, prev_keep = None, None
    for W in range(1, cfg.nprobe + 1):
        r = oracle.search(index_of(deep), deep["Q"], cfg.tau, cfg.k, cfg.nprobe, W,
                          qids=deep["qids"])
        keep = np.array([len(set(r["ids"][i][:r["count"][i]]) &
                             set(fixed["ids"][i][:fixed["count"][i]]))
                         for i in range(len(r["probes"]))])
        if prev_p is not None:
            assert (r["probes"] >= prev_p).all()
            assert (keep >= prev_keep).all()
        prev_p, prev_keep = r["probes"], keep
    assert (prev_p == cfg.nprobe).all()


def test_exact_assignment_puts_query_in_rank_one(tiny):
    cfg = tiny["cfg"]
    order, sc = oracle.rank(tiny["Q"], tiny["centroids"], cfg.nprobe, return_scores=True)
    own = tiny["assign"][tiny["qids"]]
    ok = order[:, 0] == own
    near_tie = (sc[:, 0] - sc[:, 1]) < 1e-5
    assert (ok | near_tie).all()


# ---------------------------------------------------------------------------
# hand-built indexes, every score exactly representable


def _unit_axis(d, i):
    v = np.zeros(d, np.float32)
    v[i] = 1.0
    return v


def test_tau_boundary_self_and_ties():
    d = 4
    q = _unit_axis(d, 0)
    X = np.array([
        [0.5, 0.5, 0.5, 0.5],     # sim 0.5 exactly
        [0.5, 0.5, 0.5, 0.5],     # duplicate, sim 0.5, larger id
        [1.0, 0.0, 0.0, 0.0],     # the query itself (id 7)
        [0.0, 1.0, 0.0, 0.0],     # sim 0
        [0.5, -0.5, 0.5, 0.5],    # sim 0.5 exactly, smallest id
    ], np.float32)
    ids = np.array([5, 9, 7, 3, 1], np.int64)
    idx = {"X": X, "ids": ids, "assign": np.zeros(5, np.int32), "centroids": q[None, :]}
    Q = q[None, :]
    r = oracle.search(idx, Q, 0.5, 4, 1, 1, qids=np.array([7]))
    assert r["count"][0] == 3
    assert r["ids"][0].tolist() == [1, 5, 9, -1]          # tie at 0.5 -> id asc, self excluded
    assert r["scores"][0][:3].tolist() == [0.5, 0.5, 0.5] and r["scores"][0][3] == -np.inf
    r = oracle.search(idx, Q, 0.5, 2, 1, 1, qids=None)    # no exclusion: self first
    assert r["ids"][0].tolist() == [7, 1]
    r = oracle.search(idx, Q, np.nextafter(np.float32(0.5), np.float32(1)), 4, 1, 1,
                      qids=np.array([7]))
    assert r["count"][0] == 0 and r["probes"][0] == 1     # just above 0.5: empty


def _walk_index(pattern, d=16):
    """One query along e0; partition j (centroid rank j+1) holds a row with sim
    0.75 (a hit at tau 0.7) iff pattern[j] == 'H', else a row with sim 0.5;
    centroid scores decrease strictly with j so the rank order is fixed."""
    nl = len(pattern)
    q = _unit_axis(d, 0)
    C, X, assign = [], [], []
    for j, c in enumerate(pattern):
        a = 1.0 - j / 64.0                       # exact in binary
        b = np.sqrt(1.0 - a * a)
        cen = np.zeros(d, np.float64)
        cen[0], cen[1 + j % (d - 1)] = a, b
        C.append(cen)
        s = 0.75 if c == "H" else 0.5
        x = np.zeros(d, np.float64)
        x[0], x[1 + j % (d - 1)] = s, np.sqrt(1 - s * s)
        X.append(x)
        assign.append(j)
    idx = {"X": np.array(X, np.float32), "ids": np.arange(100, 100 + nl, dtype=np.int64),
           "assign": np.array(assign, np.int32), "centroids": np.array(C, np.float32)}
    return idx, q[None, :]


def test_fig4_walk_end_to_end():
    pattern = "EEHEEEHE"                          # Fig. 4: W = 3, hit at rank 3 -> stop line 6
    idx, Q = _walk_index(pattern)
    assert oracle.rank(Q, idx["centroids"], len(pattern))[0].tolist() == list(range(8))
    for mode in ("sequential", "lookahead"):
        r = oracle.search(idx, Q, 0.7, 10, len(pattern), 3, mode=mode)
        assert r["probes"][0] == 6
        assert r["count"][0] == 1 and r["ids"][0][0] == 102   # rank-7 hit (id 106) unseen
        assert r["scores"][0][0] == pytest.approx(0.75, abs=1e-6)
    r = oracle.search(idx, Q, 0.7, 10, len(pattern), 8)       # fixed probe sees both
    assert r["ids"][0][:2].tolist() == [102, 106]


def test_physically_empty_partition_is_an_empty_probe():
    idx, Q = _walk_index("HEEEH")
    # move partition 1's only row into partition 0, leaving partition 1 empty
    idx["assign"] = idx["assign"].copy()
    idx["assign"][1] = 0
    r = oracle.search(idx, Q, 0.7, 10, 5, 3)
    assert r["probes"][0] == 4 and r["count"][0] == 1


def test_bad_arguments(tiny):
    idx = index_of(tiny)
    with pytest.raises(ValueError):
        oracle.search(idx, tiny["Q"][:2], 0.9, 10, 65, 4)     # nprobe > nlist
    with pytest.raises(ValueError):
        oracle.search(idx, tiny["Q"][:2], 0.9, 0, 16, 4)      # k < 1
    with pytest.raises(ValueError):
        oracle.search(idx, tiny["Q"][:2], float("nan"), 10, 16, 4)
