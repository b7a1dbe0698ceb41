"""In-call window calibration on the GPU (sieve_calibrated_search, Appendix A,
Algorithm 3) against the oracle's calibration: the same selected window, the
same histogram of required windows, and per-query parity of every output."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_03199_gb300 as sieve
from conftest import index_of
from parity import assert_parity, compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _index(w, dev):
    X = torch.from_numpy(w["X"]).to(dev)
    return sieve.build_layout(X, torch.from_numpy(w["assign"]).to(dev), w["centroids"].shape[0],
                              torch.from_numpy(w["centroids"]).to(dev))


def _sample(nq, ns, seed):
    return np.sort(np.random.default_rng(seed).choice(nq, ns, replace=False)).astype(np.int64)


def _run(w, gidx, dev, sample, eps, **kw):
    c = w["cfg"]
    Q = torch.from_numpy(w["Q"]).to(dev)
    qids = torch.from_numpy(w["qids"]).to(dev)
    out = sieve.calibrated_search(gidx, Q, c.tau, c.k, c.nprobe, torch.from_numpy(sample).to(dev),
                                  eps, query_ids=qids, **kw)
    torch.cuda.synchronize()
    got = {"ids": out[0].cpu().numpy(), "scores": out[1].cpu().numpy(),
           "count": out[2].cpu().numpy(), "probes": out[3].cpu().numpy()}
    return got, out[4]


@pytest.mark.parametrize("which,ns,eps", [("deep", 120, 0.0), ("deep", 120, 0.005),
                                          ("deep", 120, 0.05), ("deep", 150, 0.3),
                                          ("deep", 120, 2.0), ("tiny", 200, 0.01)])
def test_calibration_matches_oracle(request, dev, which, ns, eps):
    w = request.getfixturevalue(which)
    c = w["cfg"]
    gidx = _index(w, dev)
    sample = _sample(c.nq, ns, 17 + ns)
    got, info = _run(w, gidx, dev, sample, eps, min_queries=0)
    ref = oracle.calibrate(index_of(w), w["Q"], sample, c.tau, c.k, c.nprobe, eps, min_queries=0,
                           qids=w["qids"])
    assert info["W"] == ref["W"]
    assert info["Z"] == ref["Z"]
    assert np.array_equal(info["hist"], ref["hist"])
    assert (got["probes"][sample] == c.nprobe).all()
    order = oracle.rank(w["Q"], w["centroids"], c.nprobe)
    rep = compare(got, ref, index_of(w), w["Q"], w["qids"], c.tau, c.k, c.nprobe, order)
    assert_parity(rep)


def test_calibration_fallbacks_and_bad_samples(deep, dev):
    c = deep["cfg"]
    gidx = _index(deep, dev)
    sample = _sample(c.nq, 60, 3)
    # a small call: the fallback window, no sample
    got, info = _run(deep, gidx, dev, sample, 0.01, min_queries=c.nq + 1, fallback_W=5)
    assert info["W"] == 5 and info["Z"] == 0 and (info["hist"] == 0).all()
    Q = torch.from_numpy(deep["Q"]).to(dev)
    qids = torch.from_numpy(deep["qids"]).to(dev)
    plain = sieve.search(gidx, Q, c.tau, c.k, c.nprobe, 5, query_ids=qids)
    assert np.array_equal(got["ids"], plain[0].cpu().numpy())
    assert np.array_equal(got["probes"], plain[3].cpu().numpy())
    # a sample without any neighbour: the fallback window
    out = sieve.calibrated_search(gidx, Q, 1.5, c.k, c.nprobe, torch.from_numpy(sample).to(dev),
                                  0.01, min_queries=0, fallback_W=6, query_ids=qids)
    assert out[4]["W"] == 6 and out[4]["Z"] == 0
    # samples that are not strictly increasing rows of Q are rejected
    for bad in (sample[::-1].copy(), np.array([0, 0, 5], np.int64),
                np.array([3, c.nq], np.int64)):
        with pytest.raises(sieve.SieveError):
            sieve.calibrated_search(gidx, Q, c.tau, c.k, c.nprobe, torch.from_numpy(bad).to(dev),
                                    0.01, min_queries=0, query_ids=qids)
