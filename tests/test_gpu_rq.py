"""The quantized local search on the GPU (RaBitQ-style codes, the paper's
IVF_RQ7 index: Sec. 3.1 and Sec. 6.1) against the oracle:

- the codes and factors the device encoder writes equal oracle.rq_encode's
  bit for bit (both keep the fp64 operation order the encoder's definition
  fixes);
- sieve_rq_search equals oracle.rq_search query by query, up to decisions
  within rounding distance of a flip of the estimates (oracle_rq_fragility).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_03199_gb300 as sieve
import synth
from conftest import index_of
from parity import assert_parity, compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _workload(name):
    if name == "w256":   # full-width rows, partitions of several ragged 128-row blocks
        cfg = synth.scaled("1m", n=40_000, nlist=64, ncomp=64, nq=600, dup_frac=0.05,
                           train_cap=None, nprobe=16, W=4, seed=21)
    elif name == "w96":  # a K-block that is only half used
        cfg = synth.scaled("100m", n=30_000, nlist=80, ncomp=80, nq=600, nprobe=20, W=4, dup_frac=0.15,
                           train_cap=None, seed=22)
    else:
        raise KeyError(name)
    wl = synth.make_workload(cfg, device="cpu")
    w = synth.to_numpy(wl)
    w["cfg"] = cfg
    return w


@pytest.fixture(scope="module")
def w256():
    return _workload("w256")


@pytest.fixture(scope="module")
def w96():
    return _workload("w96")


def _gpu_index(w, dev):
    return sieve.build_layout(torch.from_numpy(w["X"]).to(dev), torch.from_numpy(w["assign"]).to(dev),
                              w["centroids"].shape[0], torch.from_numpy(w["centroids"]).to(dev))


def _run(w, gidx, rqi, dev, tau, k, nprobe, W, **kw):
    Q = torch.from_numpy(w["Q"]).to(dev)
    qids = torch.from_numpy(w["qids"]).to(dev)
    out = sieve.rq_search(gidx, rqi, Q, tau, k, nprobe, W, query_ids=qids, **kw)
    torch.cuda.synchronize()
    got = {"ids": out[0].cpu().numpy(), "scores": out[1].cpu().numpy(),
           "count": out[2].cpu().numpy(), "probes": out[3].cpu().numpy()}
    return got, (out[4] if len(out) > 4 else None)


@pytest.mark.parametrize("which", ["tiny", "deep", "w256", "w96"])
def test_device_codes_equal_oracle_codes(request, dev, which):
    w = request.getfixturevalue(which)
    idx = index_of(w)
    d = idx["X"].shape[1]
    P = synth.make_rotation(d, seed=31)
    ref_codes, ref_f = oracle.rq_encode(idx, P, 7)
    gidx = _gpu_index(w, dev)
    codes, f = sieve.rq_encode(gidx, torch.from_numpy(P).to(dev), 7)
    torch.cuda.synchronize()
    rows = gidx.ids.cpu().numpy()          # sorted row i is row ids[i] of X
    assert np.array_equal(codes.cpu().numpy(), ref_codes[rows])
    assert np.array_equal(f.cpu().numpy().view(np.uint32), ref_f[rows].view(np.uint32))


def test_rows_at_their_centroid_and_other_bit_widths(tiny, dev):
    idx = index_of(tiny)
    X = idx["X"].copy()
    X[:5] = idx["centroids"][idx["assign"][:5]]
    idx2 = dict(idx, X=X)
    P = synth.make_rotation(X.shape[1], seed=4)
    w2 = dict(tiny, X=X)
    gidx = _gpu_index(w2, dev)
    rows = gidx.ids.cpu().numpy()
    for bits in (1, 3, 7, 8):
        ref_codes, ref_f = oracle.rq_encode(idx2, P, bits)
        codes, f = sieve.rq_encode(gidx, torch.from_numpy(P).to(dev), bits)
        assert np.array_equal(codes.cpu().numpy(), ref_codes[rows]), bits
        assert np.array_equal(f.cpu().numpy(), ref_f[rows]), bits
    at = np.isin(rows, np.arange(5))
    assert (codes.cpu().numpy()[at] == 128).all() and (f.cpu().numpy()[at] == 0).all()


CASES = [  # workload, k, W, lookahead
    ("tiny", 10, 4, True), ("tiny", 10, 4, False), ("deep", 10, 3, True), ("deep", 1, 2, True),
    ("deep", 50, 3, True), ("deep", 10, 10 ** 6, True), ("w256", 10, 4, True),
    ("w256", 20, 8, False), ("w96", 10, 4, True),
]


@pytest.mark.parametrize("which,k,W,lookahead", CASES)
def test_rq_search_matches_oracle(request, dev, which, k, W, lookahead):
    w = request.getfixturevalue(which)
    c = w["cfg"]
    idx = index_of(w)
    d = idx["X"].shape[1]
    P = synth.make_rotation(d, seed=41)
    codes, f = oracle.rq_encode(idx, P, 7)
    gidx = _gpu_index(w, dev)
    rqi = sieve.build_rq_layout(gidx, torch.from_numpy(P).to(dev), 7)
    got, st = _run(w, gidx, rqi, dev, c.tau, k, c.nprobe, W, lookahead=lookahead, stats=True)
    assert st["status"] == 0 and st["items"] == got["probes"].sum()
    assert st["pairs_tc"] == st["pairs"] and st["kernel_launches"]["rq_rotate"] == 1
    ref = oracle.rq_search(idx, codes, f, P, w["Q"], c.tau, k, c.nprobe, W, qids=w["qids"])
    order = oracle.rank(w["Q"], idx["centroids"], c.nprobe)
    rep = compare(got, ref, idx, w["Q"], w["qids"], c.tau, k, c.nprobe, order, rq=(codes, f, P, 7))
    assert_parity(rep)
    # the quantized search is not the exact one: some decisions differ
    exact = oracle.search(idx, w["Q"], c.tau, k, c.nprobe, W, qids=w["qids"])
    assert not np.array_equal(exact["scores"], ref["scores"])


def test_rq_search_modes_agree(deep, dev):
    """Host-driven rounds, profiling, a precomputed order with its scores and
    small round caps change nothing."""
    c = deep["cfg"]
    P = torch.from_numpy(synth.make_rotation(deep["X"].shape[1], seed=5)).to(dev)
    gidx = _gpu_index(deep, dev)
    rqi = sieve.build_rq_layout(gidx, P, 7)
    base, _ = _run(deep, gidx, rqi, dev, c.tau, c.k, c.nprobe, c.W)
    Q = torch.from_numpy(deep["Q"]).to(dev)
    order, cs = sieve.rank_partitions(gidx, Q, c.nprobe, return_scores=True)
    for kw in ({"loop": 1}, {"profile": True}, {"order": order, "cscores": cs},
               {"max_items_per_round": 97}):
        got, st = _run(deep, gidx, rqi, dev, c.tau, c.k, c.nprobe, c.W, **kw)
        for key in base:
            assert np.array_equal(got[key], base[key]), (kw, key)
        if kw.get("profile"):
            assert st["kernel_ms"]["rq_rotate"] > 0
    with pytest.raises(sieve.SieveError):   # an order without its scores
        _run(deep, gidx, rqi, dev, c.tau, c.k, c.nprobe, c.W, order=order)


def test_rq_rejects_wide_rows_and_bad_bits(dev):
    cfg = synth.scaled("tiny", n=3000, d=264, nlist=16, ncomp=16, nq=10, seed=3)
    w = synth.to_numpy(synth.make_workload(cfg, device="cpu"))
    gidx = _gpu_index(w, dev)
    P = torch.eye(264, dtype=torch.float64, device=dev)
    with pytest.raises(sieve.SieveError):
        sieve.rq_encode(gidx, P, 7)
    cfg = synth.scaled("tiny", n=3000, nlist=16, ncomp=16, nq=10, seed=3)
    w = synth.to_numpy(synth.make_workload(cfg, device="cpu"))
    gidx = _gpu_index(w, dev)
    P = torch.eye(cfg.d, dtype=torch.float64, device=dev)
    for bits in (0, 9):
        with pytest.raises(sieve.SieveError):
            sieve.rq_encode(gidx, P, bits)
