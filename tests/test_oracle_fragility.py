"""Pins of the oracle's fragility tags, the rule that decides which GPU/oracle
mismatches are allowed (a decision within 1e-5 of a rounding flip; the tau
test of R(q, tau), Sec. 2.2, the top-k boundary of MergeTopK, Algorithm 1,
and the centroid order of Sec. 4.1).

For a query and its first ``upto`` ranks (at most nprobe):

* tau_gap = min |sim - tau| over the rows of those partitions other than the
  query's own row;
* kth_gap = the k-th minus the (k+1)-th qualifying similarity of those rows,
  +inf when fewer than k + 1 qualify;
* cen_gap = the smallest gap between consecutive sorted centroid scores
  among ranks 1 .. min(nprobe + 1, nlist).

Pinned two ways, neither re-typing the oracle's C: (1) hand-built indexes
whose similarities are multiples of 1/64, exact in fp32 and fp64, so every
gap is a known dyadic number (exact ties, fewer than k + 1 qualifiers,
``upto`` below nprobe, nlist <= nprobe + 1, the query's own row at exactly
tau); (2) on the deep workload, a numpy restatement that forms the full
similarity matrix with a BLAS product and sorts it, against the oracle's
per-row fp64 loop (agreement to 1e-12: the two sum in different orders).
"""
import numpy as np
import pytest

import oracle
from conftest import index_of


def _e0_index(first, centroid_scores, part_of_row):
    """Rows and centroids in d = 4 whose similarity with q = e0 is their
    first coordinate (the rest is a fixed orthogonal filler, so every row has
    the same norm pattern and no score is accidental)."""
    X = np.zeros((len(first), 4), np.float32)
    X[:, 0] = first
    X[:, 1] = 0.25
    C = np.zeros((len(centroid_scores), 4), np.float32)
    C[:, 0] = centroid_scores
    C[:, 2] = 0.125
    return {"X": X, "ids": np.arange(len(first), dtype=np.int64) + 100,
            "assign": np.asarray(part_of_row, np.int32), "centroids": C}


# centroid scores of q = e0, by centroid id; sorted: 0.75, 0.625, 0.5, 31/64, 0.25,
# so with nprobe = 3 the ranks are 0, 2, 1 and rank 4 (centroid 3) sits 1/64 below rank 3
CENT = [0.75, 0.5, 0.625, 31 / 64, 0.25]
# (first coordinate, partition): rank 1 = partition 0, rank 2 = partition 2, rank 3 = partition 1
ROWS = [
    (1.0, 0),        # id 100: the self row of query A (see below)
    (0.875, 0),      # id 101
    (0.8125, 0),     # id 102
    (0.5, 0),        # id 103
    (0.75, 0),       # id 104: exactly tau
    (50 / 64, 2),    # id 105
    (45 / 64, 2),    # id 106
    (49 / 64, 1),    # id 107
    (0.125, 3),      # id 108: rank 4, never searched with nprobe = 3
    (0.8125, 4),     # id 109: rank 5
]
TAU = 0.75


def hand_index():
    first, part = zip(*ROWS)
    return _e0_index(np.array(first), np.array(CENT), np.array(part))


@pytest.fixture(scope="module")
def hand():
    return hand_index()


def _frag(idx, qids, k, nprobe, upto, nq=None):
    nq = len(qids) if nq is None else nq
    Q = np.tile(np.array([[1, 0, 0, 0]], np.float32), (nq, 1))
    order = oracle.rank(Q, idx["centroids"], nprobe)
    return oracle.fragility(idx, Q, TAU, k, nprobe, order, np.full(nq, upto, np.int32),
                            qids=np.asarray(qids, np.int64))


def test_hand_built_gaps(hand):
    # query A excludes row 100 (its own row, sim 1.0); query B has no row of
    # its own; query C excludes the row at exactly tau
    tg, kg, cg = _frag(hand, [100, -5, 104], k=2, nprobe=3, upto=3)
    # non-self rows of ranks 1-3: 0.875, 0.8125, 0.5, 0.75, 50/64, 45/64, 49/64
    assert tg[0] == 0.0 and tg[1] == 0.0            # the row at exactly tau counts
    assert tg[2] == 1 / 64                           # without it: |49/64 - 3/4|
    # qualifiers (>= tau) for A: 0.875, 0.8125, 50/64, 49/64, 0.75 -> 2nd minus 3rd
    assert kg[0] == 0.8125 - 50 / 64
    # for B and C the row 100 (1.0) is not their own: 1.0, 0.875, 0.8125, ...
    assert kg[1] == kg[2] == 0.875 - 0.8125
    # centroid scores of ranks 1..4: 0.75, 0.625, 0.5, 31/64 -> smallest gap 1/64
    assert (cg == 1 / 64).all()


def test_upto_below_nprobe_limits_the_rows(hand):
    # query C (own row: the one at tau); row 100 (1.0) is not its own
    # ranks 1-2 only (partitions 0 and 2): the 49/64 row of rank 3 is not seen
    tg, kg, cg = _frag(hand, [104], k=2, nprobe=3, upto=2)
    assert tg[0] == 50 / 64 - 0.75
    assert kg[0] == 0.875 - 0.8125
    _, kg, _ = _frag(hand, [104], k=4, nprobe=3, upto=2)
    assert np.isinf(kg[0])                          # four qualify: 1, 0.875, 0.8125, 50/64
    _, kg, _ = _frag(hand, [104], k=4, nprobe=3, upto=3)
    assert kg[0] == 50 / 64 - 49 / 64               # rank 3 adds the fifth
    tg, kg, _ = _frag(hand, [104], k=3, nprobe=3, upto=1)
    assert tg[0] == 0.0625                          # 0.8125 - 0.75
    assert np.isinf(kg[0])                          # three qualify: 1, 0.875, 0.8125
    # upto past nprobe is cut at nprobe: the rank-5 row (0.8125) stays unseen
    tg9, kg9, _ = _frag(hand, [104], k=3, nprobe=3, upto=9)
    tg3, kg3, _ = _frag(hand, [104], k=3, nprobe=3, upto=3)
    assert tg9[0] == tg3[0] == 1 / 64
    assert kg9[0] == kg3[0] == 0.8125 - 50 / 64


def test_fewer_than_k_plus_one_qualifiers_give_infinity(hand):
    # query A, ranks 1-3: five qualifiers (0.875, 0.8125, 50/64, 49/64, 0.75)
    _, kg, _ = _frag(hand, [100], k=4, nprobe=3, upto=3)
    assert kg[0] == 49 / 64 - 0.75
    _, kg, _ = _frag(hand, [100], k=5, nprobe=3, upto=3)
    assert np.isinf(kg[0])
    _, kg, _ = _frag(hand, [100], k=50, nprobe=3, upto=3)
    assert np.isinf(kg[0])


def test_exact_ties_give_zero_gaps():
    # two rows tie at the k-th place; two centroids tie inside ranks 1..nprobe+1
    idx = _e0_index(np.array([0.875, 0.8125, 0.8125, 0.5]), np.array([0.75, 0.75, 0.5]),
                    np.array([0, 1, 1, 2]))
    tg, kg, cg = _frag(idx, [-1], k=2, nprobe=2, upto=2)
    assert kg[0] == 0.0 and cg[0] == 0.0
    assert tg[0] == 0.0625
    # the tie moved past rank nprobe + 1: not a centroid-order decision
    idx = _e0_index(np.array([0.875]), np.array([0.75, 0.5, 0.25, 0.25]), np.array([0]))
    _, _, cg = _frag(idx, [-1], k=1, nprobe=2, upto=2)
    assert cg[0] == 0.25
    _, _, cg = _frag(idx, [-1], k=1, nprobe=3, upto=3)
    assert cg[0] == 0.0


def test_nlist_at_most_nprobe_plus_one(hand):
    # nprobe = nlist - 1 and nlist: every centroid is compared, the last gap
    # (31/64 - 0.25) included; a single centroid has no gap at all
    for nprobe in (4, 5):
        _, _, cg = _frag(hand, [100], k=2, nprobe=nprobe, upto=nprobe)
        assert cg[0] == 1 / 64
    idx = _e0_index(np.array([0.875, 0.8125]), np.array([0.75, 0.25]), np.array([0, 1]))
    _, _, cg = _frag(idx, [-1], k=1, nprobe=2, upto=2)
    assert cg[0] == 0.5
    idx = _e0_index(np.array([0.875]), np.array([0.75]), np.array([0]))
    _, _, cg = _frag(idx, [-1], k=1, nprobe=1, upto=1)
    assert np.isinf(cg[0])


def _np_fragility(w, Q, qids, tau, k, nprobe, order, upto):
    """The three tags from a full BLAS similarity matrix and sorts."""
    X, ids, assign, C = w["X"], w["ids"], w["assign"], w["centroids"]
    S = Q.astype(np.float64) @ X.astype(np.float64).T            # [nq][n]
    CS = Q.astype(np.float64) @ C.astype(np.float64).T           # [nq][nlist]
    nlist = C.shape[0]
    tg, kg, cg = (np.empty(len(Q)) for _ in range(3))
    for i in range(len(Q)):
        parts = order[i, :min(int(upto[i]), nprobe)]
        rows = np.flatnonzero(np.isin(assign, parts) & (ids != qids[i]))
        s = S[i, rows]
        tg[i] = np.abs(s - np.float64(np.float32(tau))).min() if len(s) else np.inf
        q = np.sort(s[s >= np.float64(np.float32(tau))])[::-1]
        kg[i] = q[k - 1] - q[k] if len(q) > k else np.inf
        top = np.sort(CS[i])[::-1][:min(nprobe + 1, nlist)]
        cg[i] = (top[:-1] - top[1:]).min() if len(top) > 1 else np.inf
    return tg, kg, cg


@pytest.mark.parametrize("k", [1, 3, 10])
def test_tags_equal_numpy_restatement(deep, k):
    cfg = deep["cfg"]
    nq = 150
    Q, qids = deep["Q"][:nq], deep["qids"][:nq]
    order = oracle.rank(Q, deep["centroids"], cfg.nprobe)
    rng = np.random.default_rng(5 + k)
    upto = rng.integers(1, cfg.nprobe + 4, nq).astype(np.int32)   # some past nprobe
    tg, kg, cg = oracle.fragility(index_of(deep), Q, cfg.tau, k, cfg.nprobe, order, upto,
                                  qids=qids)
    rtg, rkg, rcg = _np_fragility(deep, Q, qids, cfg.tau, k, cfg.nprobe, order, upto)
    for got, ref in ((tg, rtg), (kg, rkg), (cg, rcg)):
        assert (np.isinf(got) == np.isinf(ref)).all()
        fin = np.isfinite(ref)
        assert np.abs(got[fin] - ref[fin]).max(initial=0.0) <= 1e-12
    # the workload exercises both branches of the k-th gap
    assert np.isinf(kg).any() and np.isfinite(kg).any()
