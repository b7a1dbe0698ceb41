"""Pins of the oracle's sharded search (the public-100M layout of Sec. 6.1:
independent IVF indexes over coarse shards, each searched with its own
ranking and stopping, then a global top-k)."""
import numpy as np
import pytest

import oracle
import synth


@pytest.fixture(scope="module")
def sharded():
    cfg = synth.scaled("tiny", n=8_000, d=32, ncomp=16, nlist=16, nq=300, dup_frac=0.08,
                       dup_counts=("uniform", 2, 8), dup_sigma=(0.02, 0.08), tau=0.88,
                       nprobe=8, W=2, seed=31)
    w = synth.make_sharded_workload(cfg, nshards=4, nlist_per_shard=12, device="cpu")
    shards = [{k: v.numpy() for k, v in sh.items()} for sh in w["shards"]]
    return cfg, shards, w["Q"].numpy(), w["qids"].numpy()


def test_shards_partition_the_corpus(sharded):
    cfg, shards, _, _ = sharded
    ids = np.concatenate([s["ids"] for s in shards])
    assert np.array_equal(np.sort(ids), np.arange(cfg.n))


def test_one_shard_is_the_plain_search(sharded):
    cfg, shards, Q, qids = sharded
    s = shards[1]
    a = oracle.sharded_search([s], Q, cfg.tau, cfg.k, cfg.nprobe, cfg.W, qids=qids)
    b = oracle.search(s, Q, cfg.tau, cfg.k, cfg.nprobe, cfg.W, qids=qids)
    for key in ("ids", "count", "probes"):
        assert np.array_equal(a[key], b[key]), key
    assert np.array_equal(a["scores"][a["ids"] >= 0], b["scores"][b["ids"] >= 0])


def test_full_probe_of_every_shard_is_bruteforce(sharded):
    """Every shard fully probed (nprobe = its nlist, W = infinity): the merged
    result is the filtered top-k over the whole corpus."""
    cfg, shards, Q, qids = sharded
    nl = min(s["centroids"].shape[0] for s in shards)
    full = oracle.sharded_search(shards, Q, cfg.tau, cfg.k, nl, 2**31 - 1, qids=qids)
    # the shards with more centroids than nl are searched fully too when nl == every nlist
    assert all(s["centroids"].shape[0] == nl for s in shards)
    X = np.zeros((cfg.n, Q.shape[1]), np.float32)
    for s in shards:
        X[s["ids"]] = s["X"]
    bf = oracle.bruteforce(X, np.arange(cfg.n, dtype=np.int64), Q, cfg.tau, cfg.k, qids=qids)
    assert np.array_equal(full["ids"], bf["ids"])
    assert np.array_equal(full["count"], bf["count"])


def test_per_shard_windows(sharded):
    cfg, shards, Q, qids = sharded
    Ws = [1, 2, 4, 8]
    a = oracle.sharded_search(shards, Q, cfg.tau, cfg.k, cfg.nprobe, Ws, qids=qids)
    for s, (sh, W) in enumerate(zip(shards, Ws)):
        b = oracle.search(sh, Q, cfg.tau, cfg.k, cfg.nprobe, W, qids=qids)
        assert np.array_equal(a["shard_probes"][:, s], b["probes"])
    assert np.array_equal(a["probes"], a["shard_probes"].sum(axis=1))
    # a larger window per shard never keeps fewer results
    b = oracle.sharded_search(shards, Q, cfg.tau, cfg.k, cfg.nprobe, 8, qids=qids)
    assert (b["count"] >= a["count"]).all()


def test_per_shard_calibration(sharded):
    """Each shard calibrates on the same sample: its window equals a separate
    calibration of that shard alone, and the merge equals the sharded search
    run with those windows except on the sampled rows (fixed-probe results)."""
    cfg, shards, Q, qids = sharded
    sample = np.sort(np.random.default_rng(8).choice(len(Q), 60, replace=False)).astype(np.int64)
    res = oracle.sharded_calibrated_search(shards, Q, sample, cfg.tau, cfg.k, cfg.nprobe, 0.02,
                                           min_queries=0, qids=qids)
    for sh, W in zip(shards, res["Ws"]):
        assert W == oracle.calibrate(sh, Q, sample, cfg.tau, cfg.k, cfg.nprobe, 0.02,
                                     min_queries=0, qids=qids)["W"]
    rest = np.setdiff1d(np.arange(len(Q)), sample)
    plain = oracle.sharded_search(shards, Q, cfg.tau, cfg.k, cfg.nprobe, res["Ws"], qids=qids)
    assert np.array_equal(res["ids"][rest], plain["ids"][rest])
    assert (res["shard_probes"][sample] == cfg.nprobe).all()
