"""fp64 CPU oracle for SieveIVF's threshold-aware IVF search (arXiv 2608.03199).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product library
(``paper_2608_03199_gb300``) never imports, links or calls it, and this package
never imports the product library: the two share no code, only input arrays.

The arithmetic lives in ``oracle.c`` (plain C, fp64, OpenMP over queries); this
module compiles it with gcc on first use and wraps each entry point for numpy
arrays.  What each function follows in the paper:

* :func:`rank`        -- centroid ranking of Sec. 2.3 / Sec. 4.1 (P_i).
* :func:`search`      -- the threshold-aware traversal of Sec. 4.1 with the
  sequential form of Algorithm 1 (``mode="sequential"``) or the lookahead
  scheduler of Algorithm 2 (``mode="lookahead"``), then MergeTopK.
* :func:`fixed_probe` -- fixed-probe IVF of Sec. 2.3 (union of nprobe lists).
* :func:`bruteforce`  -- exhaustive filtered top-k, the G_{tau,k} of Sec. 6.1.
* :func:`stop_pattern` -- the stopping rule alone over a given hit pattern.
* :func:`hit_matrix`  -- per (query, rank) hit bits, every rank.
* :func:`fragility`   -- distances of each query's decisions from a rounding
  flip (score vs tau, k-th vs (k+1)-th score, consecutive centroid scores).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` into ``oracle/_build/liboracle.so`` (gcc, -O2, OpenMP)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_variants = {}


def _declare(lib):
    P, I32, I64, U64, F32 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64, C.c_float
    lib.oracle_rank.argtypes = [P, I64, P, I64, I32, I32, P, P, I32]
    lib.oracle_stop_pattern.argtypes = [P, I32, I64, I32, U64, P]
    lib.oracle_search.argtypes = [P, P, P, I64, I32, P, I64, P, I64, P, P, F32, I32, I32,
                                  I64, I32, U64, P, P, P, P, I32]
    lib.oracle_hit_matrix.argtypes = [P, P, P, I64, I32, I64, P, I64, P, P, F32, I32, P, I32]
    lib.oracle_fixed_probe.argtypes = [P, P, P, I64, I32, I64, P, I64, P, P, F32, I32, I32,
                                       P, P, P, I32]
    lib.oracle_bruteforce.argtypes = [P, P, I64, I32, P, I64, P, F32, I32, P, P, P, I32]
    lib.oracle_fragility.argtypes = [P, P, P, I64, I32, P, I64, P, I64, P, P, P, F32, I32,
                                     I32, P, P, P, I32]
    lib.oracle_rq_encode.argtypes = [P, P, I64, I32, P, I64, P, I32, P, P, I32]
    lib.oracle_rq_fragility.argtypes = [P, P, P, I64, I32, P, I64, P, P, P, I32, P, I64, P, P, P,
                                        F32, I32, I32, P, P, P, I32]
    lib.oracle_rq_search.argtypes = [P, P, P, I64, I32, P, I64, P, P, P, I32, P, I64, P, P, F32,
                                     I32, I32, I64, I32, U64, P, P, P, P, I32]
    lib.oracle_calibrate.argtypes = [P, P, P, I64, I32, P, I64, P, I64, P, P, I64, F32, I32,
                                     I32, C.c_double, I64, I64, P, P, P, P, P, P, P, I32]
    for name in ("oracle_rank", "oracle_stop_pattern", "oracle_search", "oracle_hit_matrix",
                 "oracle_fixed_probe", "oracle_bruteforce", "oracle_fragility",
                 "oracle_calibrate", "oracle_rq_encode", "oracle_rq_search",
                 "oracle_rq_fragility"):
        getattr(lib, name).restype = C.c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _declare(C.CDLL(build()))
        return _lib


def use_library(path: str | None):
    """Route every wrapper below to another build of ``oracle.c`` (``None`` =
    the default build).  Used by the tests that plant mistakes in a copy of
    the oracle to show that the pins catch them."""
    global _lib
    with _lock:
        if path is None:
            _lib = None
            return
        if path not in _variants:
            _variants[path] = _declare(C.CDLL(path))
        _lib = _variants[path]


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _check(rc, what):
    if rc != 0:
        raise ValueError(f"{what} failed with status {rc}")


def rank(Q, Cent, nprobe, threads=None, return_scores=False):
    """P_i for every query: int32 [nq][nprobe] (0-based centroid ids)."""
    lib = _load()
    Q = _c(Q, np.float32)
    Cent = _c(Cent, np.float32)
    nq, d = Q.shape
    order = np.empty((nq, nprobe), np.int32)
    sc = np.empty((nq, nprobe), np.float64) if return_scores else None
    _check(lib.oracle_rank(_p(Q), nq, _p(Cent), Cent.shape[0], d, nprobe, _p(order), _p(sc),
                           threads or default_threads()), "oracle_rank")
    return (order, sc) if return_scores else order


def stop_pattern(hits, W, mode="sequential", seed=0):
    """Partitions searched for one query whose rank-j probe hit iff hits[j-1].

    Lookahead mode also returns the per-rank search counts."""
    lib = _load()
    h = _c(np.asarray(hits, dtype=np.uint8), np.uint8)
    nprobe = h.shape[0]
    if mode == "sequential":
        r = lib.oracle_stop_pattern(_p(h), nprobe, int(W), 0, seed, None)
        if r < 0:
            raise ValueError("bad pattern arguments")
        return r
    visits = np.zeros(nprobe, np.int32)
    r = lib.oracle_stop_pattern(_p(h), nprobe, int(W), 1, seed, _p(visits))
    if r < 0:
        raise ValueError("bad pattern arguments")
    return r, visits


_MODES = {"sequential": 0, "lookahead": 1}


def search(index, Q, tau, k, nprobe, W, qids=None, order=None, mode="sequential", seed=0,
           threads=None):
    """SieveIVF result per query.

    index: dict with X [n][d] f32, ids [n] i64, assign [n] i32, centroids [nlist][d] f32.
    Returns dict(ids [nq][k] i64, scores [nq][k] f64, count [nq] i32, probes [nq] i32).
    """
    lib = _load()
    X, ids, assign, Cent = (_c(index["X"], np.float32), _c(index["ids"], np.int64),
                            _c(index["assign"], np.int32), _c(index["centroids"], np.float32))
    Q = _c(Q, np.float32)
    nq, d = Q.shape
    qids = None if qids is None else _c(qids, np.int64)
    order = None if order is None else _c(order, np.int32)
    out_ids = np.empty((nq, k), np.int64)
    out_sc = np.empty((nq, k), np.float64)
    cnt = np.empty(nq, np.int32)
    probes = np.empty(nq, np.int32)
    rc = lib.oracle_search(_p(X), _p(ids), _p(assign), X.shape[0], d, _p(Cent), Cent.shape[0],
                           _p(Q), nq, _p(qids), _p(order), float(tau), k, nprobe, int(W),
                           _MODES[mode], seed, _p(out_ids), _p(out_sc), _p(cnt), _p(probes),
                           threads or default_threads())
    _check(rc, "oracle_search")
    return {"ids": out_ids, "scores": out_sc, "count": cnt, "probes": probes}


def hit_matrix(index, Q, tau, nprobe, order, qids=None, threads=None):
    lib = _load()
    X, ids, assign = (_c(index["X"], np.float32), _c(index["ids"], np.int64),
                      _c(index["assign"], np.int32))
    Q = _c(Q, np.float32)
    order = _c(order, np.int32)
    qids = None if qids is None else _c(qids, np.int64)
    nq, d = Q.shape
    hits = np.empty((nq, nprobe), np.uint8)
    _check(lib.oracle_hit_matrix(_p(X), _p(ids), _p(assign), X.shape[0], d,
                                 index["centroids"].shape[0], _p(Q), nq, _p(qids), _p(order),
                                 float(tau), nprobe, _p(hits), threads or default_threads()),
           "oracle_hit_matrix")
    return hits


def fixed_probe(index, Q, tau, k, nprobe, order, qids=None, threads=None):
    lib = _load()
    X, ids, assign = (_c(index["X"], np.float32), _c(index["ids"], np.int64),
                      _c(index["assign"], np.int32))
    Q = _c(Q, np.float32)
    order = _c(order, np.int32)
    qids = None if qids is None else _c(qids, np.int64)
    nq, d = Q.shape
    out_ids = np.empty((nq, k), np.int64)
    out_sc = np.empty((nq, k), np.float64)
    cnt = np.empty(nq, np.int32)
    _check(lib.oracle_fixed_probe(_p(X), _p(ids), _p(assign), X.shape[0], d,
                                  index["centroids"].shape[0], _p(Q), nq, _p(qids), _p(order),
                                  float(tau), k, nprobe, _p(out_ids), _p(out_sc), _p(cnt),
                                  threads or default_threads()), "oracle_fixed_probe")
    return {"ids": out_ids, "scores": out_sc, "count": cnt}


def bruteforce(X, ids, Q, tau, k, qids=None, threads=None):
    lib = _load()
    X, ids, Q = _c(X, np.float32), _c(ids, np.int64), _c(Q, np.float32)
    qids = None if qids is None else _c(qids, np.int64)
    nq, d = Q.shape
    out_ids = np.empty((nq, k), np.int64)
    out_sc = np.empty((nq, k), np.float64)
    cnt = np.empty(nq, np.int32)
    _check(lib.oracle_bruteforce(_p(X), _p(ids), X.shape[0], d, _p(Q), nq, _p(qids), float(tau),
                                 k, _p(out_ids), _p(out_sc), _p(cnt),
                                 threads or default_threads()), "oracle_bruteforce")
    return {"ids": out_ids, "scores": out_sc, "count": cnt}


def fragility(index, Q, tau, k, nprobe, order, upto, qids=None, threads=None, rq=None):
    """Per-query (tau_gap, kth_gap, cen_gap); see oracle_fragility in oracle.c.
    rq = (codes, factors, P, bits): the gaps of the quantized estimates
    (oracle_rq_fragility)."""
    lib = _load()
    X, ids, assign, Cent = (_c(index["X"], np.float32), _c(index["ids"], np.int64),
                            _c(index["assign"], np.int32), _c(index["centroids"], np.float32))
    Q = _c(Q, np.float32)
    order = _c(order, np.int32)
    upto = _c(upto, np.int32)
    qids = None if qids is None else _c(qids, np.int64)
    nq, d = Q.shape
    tg = np.empty(nq, np.float64)
    kg = np.empty(nq, np.float64)
    cg = np.empty(nq, np.float64)
    if rq is None:
        _check(lib.oracle_fragility(_p(X), _p(ids), _p(assign), X.shape[0], d, _p(Cent),
                                    Cent.shape[0], _p(Q), nq, _p(qids), _p(order), _p(upto),
                                    float(tau), k, nprobe, _p(tg), _p(kg), _p(cg),
                                    threads or default_threads()), "oracle_fragility")
    else:
        codes, factors, P, bits = rq
        codes, factors, P = _c(codes, np.uint8), _c(factors, np.float32), _c(P, np.float64)
        _check(lib.oracle_rq_fragility(_p(X), _p(ids), _p(assign), X.shape[0], d, _p(Cent),
                                       Cent.shape[0], _p(codes), _p(factors), _p(P), int(bits),
                                       _p(Q), nq, _p(qids), _p(order), _p(upto), float(tau), k,
                                       nprobe, _p(tg), _p(kg), _p(cg),
                                       threads or default_threads()), "oracle_rq_fragility")
    return tg, kg, cg


def calibrate(index, Q, sample, tau, k, nprobe, eps, min_queries=10_000, fallback=8, qids=None,
              threads=None):
    """In-call window calibration (Appendix A, Algorithm 3) on the sample rows
    `sample` (sorted, distinct indices into Q): dict(ids, scores, count, probes
    for every query, W = the selected window, hist [nprobe + 1] = H[W] for
    W = 1..nprobe, Z = sum of the sampled fixed-probe result sizes)."""
    lib = _load()
    X, ids, assign, Cent = (_c(index["X"], np.float32), _c(index["ids"], np.int64),
                            _c(index["assign"], np.int32), _c(index["centroids"], np.float32))
    Q = _c(Q, np.float32)
    sample = _c(sample, np.int64)
    qids = None if qids is None else _c(qids, np.int64)
    nq, d = Q.shape
    out_ids = np.empty((nq, k), np.int64)
    out_sc = np.empty((nq, k), np.float64)
    cnt = np.empty(nq, np.int32)
    probes = np.empty(nq, np.int32)
    W = np.zeros(1, np.int64)
    hist = np.zeros(nprobe + 1, np.int64)
    Z = np.zeros(1, np.int64)
    rc = lib.oracle_calibrate(_p(X), _p(ids), _p(assign), X.shape[0], d, _p(Cent), Cent.shape[0],
                              _p(Q), nq, _p(qids), _p(sample), len(sample), float(tau), k, nprobe,
                              float(eps), int(min_queries), int(fallback), _p(out_ids), _p(out_sc),
                              _p(cnt), _p(probes), _p(W), _p(hist), _p(Z),
                              threads or default_threads())
    _check(rc, "oracle_calibrate")
    return {"ids": out_ids, "scores": out_sc, "count": cnt, "probes": probes, "W": int(W[0]),
            "hist": hist, "Z": int(Z[0])}


def _merge_shards(parts, k):
    """Global top-k by (score desc, id asc) over per-shard results."""
    nq = len(parts[0]["count"])
    ids = np.concatenate([p["ids"] for p in parts], axis=1)
    sc = np.concatenate([p["scores"] for p in parts], axis=1)
    out_ids = np.full((nq, k), -1, np.int64)
    out_sc = np.full((nq, k), -np.inf)
    cnt = np.zeros(nq, np.int32)
    for i in range(nq):
        valid = ids[i] >= 0
        order = np.lexsort((ids[i][valid], -sc[i][valid]))[:k]
        n = len(order)
        out_ids[i, :n] = ids[i][valid][order]
        out_sc[i, :n] = sc[i][valid][order]
        cnt[i] = n
    shard_probes = np.stack([p["probes"] for p in parts], axis=1)
    return {"ids": out_ids, "scores": out_sc, "count": cnt,
            "probes": shard_probes.sum(axis=1).astype(np.int32), "shard_probes": shard_probes}


def sharded_calibrated_search(shards, Q, sample, tau, k, nprobe, eps, min_queries=10_000,
                              fallback=8, qids=None, threads=None):
    """Every shard calibrates its own window on the same sample (Appendix A's
    scale-out evaluation), then the global top-k.  Adds Ws (per shard)."""
    parts = [calibrate(sh, Q, sample, tau, k, nprobe, eps, min_queries=min_queries,
                       fallback=fallback, qids=qids, threads=threads) for sh in shards]
    out = _merge_shards(parts, k)
    out["Ws"] = [p["W"] for p in parts]
    return out


def sharded_search(shards, Q, tau, k, nprobe, W, qids=None, threads=None):
    """A query batch over several independent IVF indexes (the public-100M
    layout of Sec. 6.1: coarse shards, each with its own IVF index): every
    shard runs the search on its own (its own ranking and stopping; W is one
    window or one per shard), then the global top-k by (score desc, id asc)
    merges the shards' results.  Returns dict(ids, scores, count, probes =
    partitions searched over all shards, shard_probes [nq][nshards])."""
    Ws = list(W) if isinstance(W, (list, tuple, np.ndarray)) else [W] * len(shards)
    parts = [search(sh, Q, tau, k, nprobe, w, qids=qids, threads=threads) for sh, w in zip(shards, Ws)]
    return _merge_shards(parts, k)


def rq_encode(index, P, bits=7, threads=None):
    """RaBitQ-style codes of the rows (oracle_rq_encode): codes [n][d] uint8,
    factors [n] float32, for the rotation P [d][d] (float64, orthogonal)."""
    lib = _load()
    X, assign, Cent = (_c(index["X"], np.float32), _c(index["assign"], np.int32),
                       _c(index["centroids"], np.float32))
    P = _c(P, np.float64)
    n, d = X.shape
    codes = np.empty((n, d), np.uint8)
    factors = np.empty(n, np.float32)
    _check(lib.oracle_rq_encode(_p(X), _p(assign), n, d, _p(Cent), Cent.shape[0], _p(P), bits,
                                _p(codes), _p(factors), threads or default_threads()),
           "oracle_rq_encode")
    return codes, factors


def rq_search(index, codes, factors, P, Q, tau, k, nprobe, W, bits=7, qids=None, order=None,
              mode="sequential", seed=0, threads=None):
    """search() with the quantized local search on the given codes."""
    lib = _load()
    X, ids, assign, Cent = (_c(index["X"], np.float32), _c(index["ids"], np.int64),
                            _c(index["assign"], np.int32), _c(index["centroids"], np.float32))
    codes, factors, P = _c(codes, np.uint8), _c(factors, np.float32), _c(P, np.float64)
    Q = _c(Q, np.float32)
    nq, d = Q.shape
    qids = None if qids is None else _c(qids, np.int64)
    order = None if order is None else _c(order, np.int32)
    out_ids = np.empty((nq, k), np.int64)
    out_sc = np.empty((nq, k), np.float64)
    cnt = np.empty(nq, np.int32)
    probes = np.empty(nq, np.int32)
    rc = lib.oracle_rq_search(_p(X), _p(ids), _p(assign), X.shape[0], d, _p(Cent), Cent.shape[0],
                              _p(codes), _p(factors), _p(P), bits, _p(Q), nq, _p(qids), _p(order),
                              float(tau), k, nprobe, int(W), _MODES[mode], seed, _p(out_ids),
                              _p(out_sc), _p(cnt), _p(probes), threads or default_threads())
    _check(rc, "oracle_rq_search")
    return {"ids": out_ids, "scores": out_sc, "count": cnt, "probes": probes}
