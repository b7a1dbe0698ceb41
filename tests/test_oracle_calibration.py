"""Pins of the oracle's in-call window calibration (Appendix A, Algorithm 3).

The histogram of required windows is checked against the literal definition
of loss(W): for every W, the sampled queries are searched again with that W
and their results intersected with the fixed-probe results.  The selected
window, the fallbacks and the per-query outputs are checked against plain
searches."""
import numpy as np
import pytest

import oracle
from conftest import index_of


def _sample(nq, ns, seed):
    return np.sort(np.random.default_rng(seed).choice(nq, ns, replace=False)).astype(np.int64)


def _retained(a_ids, a_cnt, f_ids, f_cnt):
    tot = 0
    for i in range(len(f_cnt)):
        tot += len(set(a_ids[i, :a_cnt[i]]) & set(f_ids[i, :f_cnt[i]]))
    return tot


@pytest.mark.parametrize("eps", [0.0, 0.005, 0.05, 0.3, 2.0])
def test_calibration_matches_brute_force_loss(deep, eps):
    w, c = deep, deep["cfg"]
    idx = index_of(w)
    sample = _sample(c.nq, 120, 5)
    res = oracle.calibrate(idx, w["Q"], sample, c.tau, c.k, c.nprobe, eps, min_queries=0,
                           qids=w["qids"])
    Qs, qs = w["Q"][sample], w["qids"][sample]
    fixed = oracle.search(idx, Qs, c.tau, c.k, c.nprobe, c.nprobe, qids=qs)
    Z = int(fixed["count"].sum())
    assert res["Z"] == Z and Z > 0
    assert res["hist"][0] == 0 and res["hist"].sum() == Z
    # the histogram's prefix sums are the retained neighbours of every window
    pref = np.cumsum(res["hist"])
    best = c.nprobe
    for W in range(1, c.nprobe + 1):
        a = oracle.search(idx, Qs, c.tau, c.k, c.nprobe, W, qids=qs)
        kept = _retained(a["ids"], a["count"], fixed["ids"], fixed["count"])
        assert kept == pref[W], W
        if W < c.nprobe and best == c.nprobe and 1.0 - kept / Z < eps:
            best = W
    assert res["W"] == best
    # sampled rows keep their fixed-probe results, the rest run with W*
    assert np.array_equal(res["ids"][sample], fixed["ids"])
    assert np.array_equal(res["count"][sample], fixed["count"])
    assert (res["probes"][sample] == c.nprobe).all()
    rest = np.setdiff1d(np.arange(c.nq), sample)
    r = oracle.search(idx, w["Q"][rest], c.tau, c.k, c.nprobe, best, qids=w["qids"][rest])
    for key in ("ids", "count", "probes"):
        assert np.array_equal(res[key][rest], r[key]), key


def test_calibration_window_extremes_and_fallbacks(deep):
    w, c = deep, deep["cfg"]
    idx = index_of(w)
    sample = _sample(c.nq, 80, 9)
    # a loss target above 1 accepts the smallest window; 0 accepts none
    assert oracle.calibrate(idx, w["Q"], sample, c.tau, c.k, c.nprobe, 1.5, min_queries=0,
                            qids=w["qids"])["W"] == 1
    assert oracle.calibrate(idx, w["Q"], sample, c.tau, c.k, c.nprobe, 0.0, min_queries=0,
                            qids=w["qids"])["W"] == c.nprobe
    # small calls and empty samples use the fallback window
    small = oracle.calibrate(idx, w["Q"], sample, c.tau, c.k, c.nprobe, 0.01,
                             min_queries=c.nq + 1, fallback=5, qids=w["qids"])
    assert small["W"] == 5 and small["Z"] == 0
    plain = oracle.search(idx, w["Q"], c.tau, c.k, c.nprobe, 5, qids=w["qids"])
    assert np.array_equal(small["ids"], plain["ids"])
    empty = oracle.calibrate(idx, w["Q"], np.zeros(0, np.int64), c.tau, c.k, c.nprobe, 0.01,
                             min_queries=0, fallback=3, qids=w["qids"])
    assert empty["W"] == 3
    # a sample with no neighbours at all (tau above every similarity)
    none = oracle.calibrate(idx, w["Q"], sample, 1.5, c.k, c.nprobe, 0.01, min_queries=0,
                            fallback=6, qids=w["qids"])
    assert none["Z"] == 0 and none["W"] == 6


def test_calibration_required_window_rule():
    """Window W reaches rank j iff no run of W empty ranks ends before j: checked
    against the stopping state machine over every hit pattern of 9 ranks."""
    nprobe = 9
    for bits in range(1 << nprobe):
        hits = np.array([(bits >> j) & 1 for j in range(nprobe)], np.uint8)
        # longest run of empties strictly before rank j (1-based j = idx + 1)
        before, run, best = [], 0, 0
        for j in range(nprobe):
            before.append(best)
            run = 0 if hits[j] else run + 1
            best = max(best, run)
        for W in range(1, nprobe + 1):
            probes = oracle.stop_pattern(hits, W)
            for j in range(nprobe):
                assert (j < probes) == (W >= 1 + before[j]), (bits, W, j)


def _gapped_index():
    """One query whose qualifying rows sit at ranks 1, 3 and 6 of its probe
    order (8 partitions, every other partition empty of neighbours)."""
    def vec(a):
        return np.array([a, np.sqrt(1.0 - a * a), 0.0, 0.0], np.float32)
    cents = np.stack([vec(0.9 - 0.1 * p) for p in range(8)])      # rank p+1 = partition p
    rows, assign = [], []
    for p in range(8):
        rows.append(vec(0.1)); assign.append(p)                   # never qualifies
    for p, s in ((0, 0.95), (2, 0.93), (5, 0.91)):
        rows.append(vec(s)); assign.append(p)
    X = np.stack(rows)
    idx = {"X": X, "ids": np.arange(len(X), dtype=np.int64),
           "assign": np.array(assign, np.int32), "centroids": cents}
    return idx, np.array([[1.0, 0.0, 0.0, 0.0]], np.float32)


def test_calibration_histogram_of_gapped_hits():
    """Neighbours at ranks 1, 3, 6 (empty ranks 2 and 4-5 before the third)
    need windows 1, 2 and 3: the longest empty run before a rank, plus one."""
    idx, Q = _gapped_index()
    res = oracle.calibrate(idx, Q, np.array([0], np.int64), 0.9, 10, 8, 0.5, min_queries=0)
    assert res["Z"] == 3
    assert list(res["hist"]) == [0, 1, 1, 1, 0, 0, 0, 0, 0]
    # loss(1) = 2/3, loss(2) = 1/3, loss(3) = 0: eps 0.5 selects W = 2
    assert res["W"] == 2
    for W, kept in ((1, 1), (2, 2), (3, 3), (8, 3)):
        a = oracle.search(idx, Q, 0.9, 10, 8, W)
        assert a["count"][0] == kept, W
