"""Pins of the oracle's RaBitQ-style quantized local search (the paper's
IVF_RQ7 local search: RaBitQ codes with 7 bits, Sec. 3.1 and Sec. 6.1).

The estimator is exact for rows whose rotated unit residual lies on the code
grid, its error shrinks with more bits, and it is unbiased over many rows;
the quantized search reduces to the exact one as the bits grow."""
import numpy as np
import pytest

import oracle
import synth
from conftest import index_of


def _one_partition_index(X, c):
    n = len(X)
    return {"X": X.astype(np.float32), "ids": np.arange(n, dtype=np.int64),
            "assign": np.zeros(n, np.int32), "centroids": c[None, :].astype(np.float32)}


def test_grid_aligned_rows_are_estimated_exactly():
    d, bits = 32, 7
    rng = np.random.default_rng(3)
    P = synth.make_rotation(d, seed=5)
    mid = (2 ** bits - 1) / 2
    c = rng.standard_normal(d) * 0.1
    rows, codes_want = [], []
    for _ in range(40):
        u = rng.integers(0, 2 ** bits, d).astype(np.float64)
        u[rng.integers(d)] = rng.choice([0, 2 ** bits - 1])   # one coordinate at the edge
        ob = (u - mid) / np.linalg.norm(u - mid)              # a grid direction, unit
        x = c + 0.7 * (P @ ob)                                 # o = P o', o' = ob
        rows.append(x)
        codes_want.append(u)
    X = np.array(rows, np.float32)
    idx = _one_partition_index(X, c)
    codes, f = oracle.rq_encode(idx, P, bits)
    assert np.array_equal(codes.astype(np.float64), np.array(codes_want))
    # estimate = <q, c> + f (<u, P^T q> - mid sum(P^T q)) equals <q, x> on these rows
    Q = rng.standard_normal((5, d))
    for q in Q:
        qr = P.T @ q
        est = q @ c.astype(np.float32) + f.astype(np.float64) * (codes @ qr - mid * qr.sum())
        assert np.abs(est - X.astype(np.float64) @ q).max() < 2e-5


def test_estimator_error_shrinks_with_bits_and_is_unbiased(tiny):
    idx = index_of(tiny)
    d = idx["X"].shape[1]
    P = synth.make_rotation(d, seed=11)
    rng = np.random.default_rng(1)
    rows = rng.choice(len(idx["X"]), 3000, replace=False)
    Q = tiny["Q"][:20].astype(np.float64)
    errs = {}
    for bits in (3, 5, 7, 8):
        codes, f = oracle.rq_encode(idx, P, bits)
        mid = (2 ** bits - 1) / 2
        C = idx["centroids"].astype(np.float64)
        e = []
        for q in Q:
            qr = P.T @ q
            cp = C[idx["assign"][rows]]
            est = cp @ q + f[rows].astype(np.float64) * (codes[rows] @ qr - mid * qr.sum())
            e.append(est - idx["X"][rows].astype(np.float64) @ q)
        e = np.concatenate(e)
        errs[bits] = e
        # no systematic offset: the mean error is within 4 standard errors of 0
        assert abs(e.mean()) < 4 * e.std() / np.sqrt(len(e)) + 1e-9, bits
    rms = {b: np.sqrt((e ** 2).mean()) for b, e in errs.items()}
    assert rms[3] > rms[5] > rms[7] > rms[8]
    assert rms[7] < 2e-3


def test_quantized_search_approaches_exact(deep):
    w, c = deep, deep["cfg"]
    idx = index_of(w)
    P = synth.make_rotation(idx["X"].shape[1], seed=2)
    exact = oracle.search(idx, w["Q"], c.tau, c.k, c.nprobe, c.nprobe, qids=w["qids"])
    tot = exact["count"].sum()
    kept = {}
    for bits in (4, 8):
        codes, f = oracle.rq_encode(idx, P, bits)
        r = oracle.rq_search(idx, codes, f, P, w["Q"], c.tau, c.k, c.nprobe, c.nprobe, bits=bits,
                             qids=w["qids"])
        kept[bits] = sum(len(set(r["ids"][i, :r["count"][i]]) & set(exact["ids"][i, :exact["count"][i]]))
                         for i in range(len(r["count"])))
    assert kept[8] >= kept[4]
    assert kept[8] >= 0.97 * tot


def test_rows_at_their_centroid_and_bounds(tiny):
    idx = index_of(tiny)
    d = idx["X"].shape[1]
    X = idx["X"].copy()
    X[:3] = idx["centroids"][idx["assign"][:3]]      # three rows equal to their centroid
    idx2 = dict(idx, X=X)
    codes, f = oracle.rq_encode(idx2, synth.make_rotation(d, seed=4), 7)
    assert (codes[:3] == 64).all() and (f[:3] == 0).all()
    assert codes.max() <= 127 and np.isfinite(f).all() and (f[3:] > 0).all()


def test_quantized_fragility_measures_the_estimates(deep):
    """oracle_rq_fragility (the parity tests' allowance for the quantized
    search) reports the distance of the nearest estimate from tau over the
    searched partitions, and the centroid gaps of the exact ranking."""
    w, c = deep, deep["cfg"]
    idx = index_of(w)
    d = idx["X"].shape[1]
    P = synth.make_rotation(d, seed=6)
    codes, f = oracle.rq_encode(idx, P, 7)
    Q = w["Q"][:25]
    qids = w["qids"][:25]
    order = oracle.rank(Q, idx["centroids"], c.nprobe)
    upto = np.full(len(Q), 5, np.int32)
    tg, kg, cg = oracle.fragility(idx, Q, c.tau, c.k, c.nprobe, order, upto, qids=qids,
                                  rq=(codes, f, P, 7))
    tg0, _, cg0 = oracle.fragility(idx, Q, c.tau, c.k, c.nprobe, order, upto, qids=qids)
    assert np.array_equal(cg, cg0)
    mid = 63.5
    C = idx["centroids"].astype(np.float64)
    for i, q in enumerate(Q.astype(np.float64)):
        qr = P.T @ q
        rows = np.flatnonzero(np.isin(idx["assign"], order[i, :5]) & (idx["ids"] != qids[i]))
        est = C[idx["assign"][rows]] @ q + f[rows].astype(np.float64) * (codes[rows] @ qr - mid * qr.sum())
        assert abs(tg[i] - np.abs(est - np.float64(np.float32(c.tau))).min()) < 1e-9
    assert not np.array_equal(tg, tg0)   # the estimates, not the exact similarities
