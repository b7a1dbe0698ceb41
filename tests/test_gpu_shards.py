"""Sharded search on the GPU (sieve_sharded_search) against the oracle's:
every shard searched with its own ranking and stopping, then the global
top-k (the public-100M layout of Sec. 6.1)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_03199_gb300 as sieve
import synth
from parity import TOL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sharded():
    assert torch.cuda.is_available()
    dev = torch.device("cuda:0")
    cfg = synth.scaled("tiny", n=8_000, d=32, ncomp=16, nlist=16, nq=300, dup_frac=0.08,
                       dup_counts=("uniform", 2, 8), dup_sigma=(0.02, 0.08), tau=0.88,
                       nprobe=8, W=2, seed=31)
    w = synth.make_sharded_workload(cfg, nshards=4, nlist_per_shard=12, device="cpu")
    host = [{k: v.numpy() for k, v in sh.items()} for sh in w["shards"]]
    gshards = []
    for sh in w["shards"]:
        idx = sieve.build_layout(sh["X"].to(dev), sh["assign"].to(dev), sh["centroids"].shape[0],
                                 sh["centroids"].to(dev))
        # the layout numbers rows 0..n_s-1; the shard's own ids are the corpus rows
        gshards.append(sieve.Index(idx.vectors, sh["ids"].to(dev)[idx.ids], idx.list_offsets,
                                   idx.centroids, idx.tc_rows, idx.tc_row_blocks, idx.tc_centroids))
    return cfg, host, gshards, w["Q"].numpy(), w["qids"].numpy(), dev


@pytest.mark.parametrize("W", [2, [1, 2, 4, 8], 2**31 - 1])
def test_sharded_search_matches_oracle(sharded, W):
    cfg, host, gshards, Q, qids, dev = sharded
    out = sieve.sharded_search(gshards, torch.from_numpy(Q).to(dev), cfg.tau, cfg.k, cfg.nprobe, W,
                               query_ids=torch.from_numpy(qids).to(dev))
    torch.cuda.synchronize()
    ref = oracle.sharded_search(host, Q, cfg.tau, cfg.k, cfg.nprobe, W, qids=qids)
    got = [o.cpu().numpy() for o in out]
    assert np.array_equal(got[4], ref["shard_probes"])
    assert np.array_equal(got[3], ref["probes"])
    assert np.array_equal(got[2], ref["count"])
    assert np.array_equal(got[0], ref["ids"])
    valid = got[0] >= 0
    assert np.abs(got[1][valid] - ref["scores"][valid]).max(initial=0) <= TOL
    assert np.isneginf(got[1][~valid]).all()


def test_per_shard_calibration_matches_oracle(sharded):
    cfg, host, gshards, Q, qids, dev = sharded
    sample = np.sort(np.random.default_rng(8).choice(len(Q), 60, replace=False)).astype(np.int64)
    out = sieve.sharded_calibrated_search(gshards, torch.from_numpy(Q).to(dev), cfg.tau, cfg.k,
                                          cfg.nprobe, torch.from_numpy(sample).to(dev), 0.02,
                                          min_queries=0, query_ids=torch.from_numpy(qids).to(dev))
    torch.cuda.synchronize()
    ref = oracle.sharded_calibrated_search(host, Q, sample, cfg.tau, cfg.k, cfg.nprobe, 0.02,
                                           min_queries=0, qids=qids)
    assert out[5] == ref["Ws"]
    got = [o.cpu().numpy() for o in out[:5]]
    assert np.array_equal(got[4], ref["shard_probes"])
    assert np.array_equal(got[2], ref["count"])
    assert np.array_equal(got[0], ref["ids"])
    valid = got[0] >= 0
    assert np.abs(got[1][valid] - ref["scores"][valid]).max(initial=0) <= TOL
