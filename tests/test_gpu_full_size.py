"""Parity at the benchmark's full size (1M x 256 rows, 1,024 partitions, 100K
queries, tau 0.90, k 10, nprobe 64, W 8, lookahead on) in the launch
configuration ``bench.py`` times.

The whole batch runs on the GPU; the oracle recomputes a seeded sample of the
queries one by one (per-query results do not depend on the batch, Sec. 4.3),
and properties that hold at any size are checked on every query."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_03199_gb300 as sieve
import synth
from parity import assert_parity, compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def full():
    assert torch.cuda.is_available()
    dev = torch.device("cuda:0")
    cfg = synth.CONFIGS["1m"]
    wl = synth.make_workload(cfg, device=dev)
    index = sieve.build_layout(wl["X"], wl["assign"], cfg.nlist, wl["centroids"])
    host = {k: wl[k].cpu().numpy() for k in ("X", "ids", "assign", "centroids", "Q", "qids")}
    return cfg, wl, index, host


def _np(out):
    return {"ids": out[0].cpu().numpy(), "scores": out[1].cpu().numpy(),
            "count": out[2].cpu().numpy(), "probes": out[3].cpu().numpy()}


def test_full_size_sampled_parity(full):
    cfg, wl, index, h = full
    out = sieve.search(index, wl["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W, lookahead=True,
                       query_ids=wl["qids"], stats=True)
    got, st = _np(out), out[4]
    assert st["status"] == 0
    assert st["items"] == got["probes"].sum()
    assert ((got["probes"] >= cfg.W) & (got["probes"] <= cfg.nprobe)).all()
    rng = np.random.default_rng(1234)
    sample = np.sort(rng.choice(cfg.nq, 1500, replace=False))
    idx = {k: h[k] for k in ("X", "ids", "assign", "centroids")}
    Q, qids = h["Q"][sample], h["qids"][sample]
    ref = oracle.search(idx, Q, cfg.tau, cfg.k, cfg.nprobe, cfg.W, qids=qids)
    order = oracle.rank(Q, h["centroids"], cfg.nprobe)
    rep = compare({k: v[sample] for k, v in got.items()}, ref, idx, Q, qids, cfg.tau, cfg.k,
                  cfg.nprobe, order)
    assert_parity(rep)
    # sorted output rows, padding
    valid = np.arange(cfg.k)[None, :] < got["count"][:, None]
    sc = got["scores"]
    assert ((sc[:, 1:] <= sc[:, :-1]) | ~valid[:, 1:]).all()
    assert ((got["ids"] == -1) == ~valid).all()
    assert (got["scores"][valid] >= np.float32(cfg.tau)).all()


def test_full_size_schedule_invariance_and_fixed_probe(full):
    cfg, wl, index, h = full
    runs = [_np(sieve.search(index, wl["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W, query_ids=wl["qids"],
                             scan_path="tensor", **kw))
            for kw in (dict(lookahead=True), dict(lookahead=False),
                       dict(lookahead=True, max_items_per_round=65536))]
    for key in runs[0]:
        assert all(np.array_equal(runs[0][key], r[key]) for r in runs[1:]), key
    a = _np(sieve.search(index, wl["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.W, lookahead=True,
                         query_ids=wl["qids"]))
    fx = _np(sieve.search(index, wl["Q"], cfg.tau, cfg.k, cfg.nprobe, cfg.nprobe, lookahead=True,
                          query_ids=wl["qids"]))
    assert (fx["probes"] == cfg.nprobe).all()
    # fixed probe sees a superset of partitions: it never returns fewer results
    assert (fx["count"] >= a["count"]).all()
    sample = np.arange(0, cfg.nq, 400)
    idx = {k: h[k] for k in ("X", "ids", "assign", "centroids")}
    Q, qids = h["Q"][sample], h["qids"][sample]
    order = oracle.rank(Q, h["centroids"], cfg.nprobe)
    ref = oracle.fixed_probe(idx, Q, cfg.tau, cfg.k, cfg.nprobe, order, qids=qids)
    ref["probes"] = np.full(len(sample), cfg.nprobe, np.int32)
    rep = compare({k: v[sample] for k, v in fx.items()}, ref, idx, Q, qids, cfg.tau, cfg.k,
                  cfg.nprobe, order)
    assert_parity(rep)


@pytest.mark.parametrize("W,tau", [(2, None), (4, None), (16, None), (8, 0.3)])
def test_full_size_other_windows_and_loose_tau(full, W, tau):
    """The whole 100K-query batch at other windows (W = 16 takes the screening
    scan on the automatic path) and at tau = 0.3, where most probes hit and
    the epilogue keeps the most candidates (the loose end of Sec. 6.4); the
    oracle recomputes 600 sampled queries."""
    cfg, wl, index, h = full
    tau = cfg.tau if tau is None else tau
    got = _np(sieve.search(index, wl["Q"], tau, cfg.k, cfg.nprobe, W, lookahead=True,
                           query_ids=wl["qids"]))
    assert ((got["probes"] >= min(W, cfg.nprobe)) & (got["probes"] <= cfg.nprobe)).all()
    rng = np.random.default_rng(100 + W)
    sample = np.sort(rng.choice(cfg.nq, 600, replace=False))
    idx = {k: h[k] for k in ("X", "ids", "assign", "centroids")}
    Q, qids = h["Q"][sample], h["qids"][sample]
    ref = oracle.search(idx, Q, tau, cfg.k, cfg.nprobe, W, qids=qids)
    order = oracle.rank(Q, h["centroids"], cfg.nprobe)
    rep = compare({k: v[sample] for k, v in got.items()}, ref, idx, Q, qids, tau, cfg.k,
                  cfg.nprobe, order)
    assert_parity(rep)
    if tau < 0.5:   # loose threshold: nearly every query fills its k results
        assert (got["count"] == cfg.k).mean() > 0.9
