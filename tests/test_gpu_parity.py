"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Element by element on seeded inputs that span many tiles with ragged tails:
probe counts, result ids and counts identical (up to the counted, tagged
rounding divergences of ``parity.py``), scores within 1e-5.  Also the
invariances the paper fixes (lookahead / per-round caps / loop mode change
nothing, Sec. 4.2-4.3; W >= nprobe is fixed probing; nprobe = nlist with
W = infinity is brute force) and the edge cases of the boundary.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_03199_gb300 as sieve
import synth
from conftest import index_of
from parity import TOL, assert_parity, compare

pytestmark = pytest.mark.gpu

BIG_W = 2**31 - 1


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def gpu_index(w, dev, tc_layout=None):
    X = torch.from_numpy(w["X"]).to(dev)
    assign = torch.from_numpy(w["assign"]).to(dev)
    cent = torch.from_numpy(w["centroids"]).to(dev)
    return sieve.build_layout(X, assign, cent.shape[0], cent, tc_layout=tc_layout)


@pytest.fixture(scope="module")
def g_tiny(tiny, dev):
    return gpu_index(tiny, dev)


@pytest.fixture(scope="module")
def g_deep(deep, dev):
    return gpu_index(deep, dev)


def run(index, Q, qids, tau, k, nprobe, W, **kw):
    dev = index.vectors.device
    Qd = torch.from_numpy(np.ascontiguousarray(Q)).to(dev)
    qd = None if qids is None else torch.from_numpy(np.ascontiguousarray(qids)).to(dev)
    out = sieve.search(index, Qd, tau, k, nprobe, W, query_ids=qd, **kw)
    torch.cuda.synchronize()
    res = {"ids": out[0].cpu().numpy(), "scores": out[1].cpu().numpy(),
           "count": out[2].cpu().numpy(), "probes": out[3].cpu().numpy()}
    if kw.get("stats"):
        res["stats"] = out[4]
    return res


def check(w, gidx, Q, qids, tau, k, nprobe, W, lookahead, **kw):
    ref = oracle.search(index_of(w), Q, tau, k, nprobe, W, qids=qids)
    got = run(gidx, Q, qids, tau, k, nprobe, W, lookahead=lookahead, **kw)
    order = oracle.rank(Q, w["centroids"], nprobe)
    rep = compare(got, ref, index_of(w), Q, qids, tau, k, nprobe, order)
    assert_parity(rep)
    return got, ref, rep


# ---------------------------------------------------------------------------
def test_layout_is_a_stable_counting_sort(tiny, g_tiny):
    perm = np.argsort(tiny["assign"], kind="stable")
    assert (g_tiny.ids.cpu().numpy() == perm).all()
    assert np.array_equal(g_tiny.vectors.cpu().numpy(), tiny["X"][perm])
    off = np.concatenate([[0], np.cumsum(np.bincount(tiny["assign"], minlength=64))])
    assert (g_tiny.list_offsets.cpu().numpy() == off).all()


def test_rank_parity(tiny, g_tiny, dev):
    Q = torch.from_numpy(tiny["Q"]).to(dev)
    for nprobe in (1, 16, 63, 64):
        order, sc = sieve.rank_partitions(g_tiny, Q, nprobe, return_scores=True)
        order, sc = order.cpu().numpy(), sc.cpu().numpy()
        ref, rsc = oracle.rank(tiny["Q"], tiny["centroids"], min(nprobe + 1, 64), return_scores=True)
        assert np.abs(sc - rsc[:, :nprobe]).max() <= TOL
        gaps = np.diff(rsc, axis=1).__neg__().min(axis=1) if rsc.shape[1] > 1 else np.full(len(rsc), np.inf)
        bad = (order != ref[:, :nprobe]).any(axis=1)
        assert (gaps[bad] < TOL).all()
        assert bad.sum() <= 2


@pytest.mark.parametrize("nlist", [1, 33, 64, 100, 1000, 2048, 2049, 4100, 9000])
def test_rank_selection_exact_ties(nlist, dev):
    """Scores that are exact in fp32 and fp64 (multiples of 1/64 from
    coordinates in {-2..2}/8), so equal scores tie exactly: the order must be
    the (score desc, id asc) sort, for every nprobe shape, including all-equal
    rows and far more ties than nprobe."""
    rng = np.random.default_rng(nlist)
    d = 8
    C = (rng.integers(-2, 3, size=(nlist, d)) / 8).astype(np.float32)
    if nlist >= 64:
        C[nlist // 2:nlist // 2 + 20] = C[3]          # a block of identical centroids
    Q = (rng.integers(-2, 3, size=(300, d)) / 8).astype(np.float32)
    Q[0] = 0.0                                        # every score 0: ids in order
    Cd = torch.from_numpy(C).to(dev)
    index = sieve.build_layout(Cd.clone(), torch.arange(nlist, dtype=torch.int32, device=dev),
                               nlist, Cd)
    Qd = torch.from_numpy(Q).to(dev)
    ref_sc = Q.astype(np.float64) @ C.astype(np.float64).T
    for nprobe in sorted({1, 2, 5, max(1, nlist // 2), min(nlist, 64), min(nlist, 512), nlist}):
        if nprobe > min(nlist, 512):
            continue
        order, sc = sieve.rank_partitions(index, Qd, nprobe, return_scores=True)
        order, sc = order.cpu().numpy(), sc.cpu().numpy()
        ref = np.stack([np.lexsort((np.arange(nlist), -row))[:nprobe] for row in ref_sc])
        assert np.array_equal(order, ref), nprobe
        assert np.array_equal(sc.astype(np.float64), np.take_along_axis(ref_sc, ref, 1))


def test_rank_single_range_ties(dev):
    """A batch large enough for one centroid range per query tile (80,100
    queries): exact ties must come out in (score desc, id asc) order for every
    query, from the screen's starting threshold through the exact pass with
    two sub-tiles to the final sort."""
    rng = np.random.default_rng(17)
    nlist, d = 9000, 8   # 141 groups of 64 (nprobe 64), 282 of 32 (nprobe 128): the screen's first pass
    C = (rng.integers(-2, 3, size=(nlist, d)) / 8).astype(np.float32)
    C[nlist // 2:nlist // 2 + 20] = C[3]
    U = (rng.integers(-2, 3, size=(300, d)) / 8).astype(np.float32)
    U[0] = 0.0
    Q = np.tile(U, (267, 1))
    Cd = torch.from_numpy(C).to(dev)
    index = sieve.build_layout(Cd.clone(), torch.arange(nlist, dtype=torch.int32, device=dev), nlist, Cd)
    ref_sc = U.astype(np.float64) @ C.astype(np.float64).T
    for nprobe in (64, 128):
        order, sc = sieve.rank_partitions(index, torch.from_numpy(Q).to(dev), nprobe, return_scores=True)
        order, sc = order.cpu().numpy(), sc.cpu().numpy()
        ref = np.stack([np.lexsort((np.arange(nlist), -row))[:nprobe] for row in ref_sc])
        assert np.array_equal(order, np.tile(ref, (267, 1))), nprobe
        assert np.array_equal(sc.astype(np.float64), np.tile(np.take_along_axis(ref_sc, ref, 1), (267, 1)))


def test_rank_single_range_parity(dev):
    """80,003 queries against 32,868 centroids (d = 96, nprobe 256, 514
    groups of 64, the 100M workload's shape of first pass): one range
    per query tile, so the first pass, the starting threshold, the exact pass
    with two sub-tiles and the final selection all run at their large-batch
    shapes; sampled queries and the ragged tail against the fp64 oracle."""
    rng = np.random.default_rng(23)
    nlist, d, nprobe, nq = 32_868, 96, 256, 80_003
    C = rng.standard_normal((nlist, d)).astype(np.float32)
    C /= np.linalg.norm(C, axis=1, keepdims=True)
    Q = (C[rng.integers(0, nlist, nq)] + 0.3 * rng.standard_normal((nq, d))).astype(np.float32)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    Cd = torch.from_numpy(C).to(dev)
    index = sieve.build_layout(Cd.clone(), torch.arange(nlist, dtype=torch.int32, device=dev), nlist, Cd)
    order, sc = sieve.rank_partitions(index, torch.from_numpy(Q).to(dev), nprobe, return_scores=True)
    order, sc = order.cpu().numpy(), sc.cpu().numpy()
    pick = np.concatenate([rng.choice(nq - 7, 1500, replace=False), np.arange(nq - 7, nq)])
    ref, rsc = oracle.rank(Q[pick], C, nprobe + 1, return_scores=True)
    assert np.abs(sc[pick] - rsc[:, :nprobe]).max() <= TOL
    gaps = (rsc[:, :-1] - rsc[:, 1:]).min(axis=1)
    bad = (order[pick] != ref[:, :nprobe]).any(axis=1)
    # every rank swap sits on a centroid-score gap below the tolerance; with
    # 32,868 centroids such near-ties are common (a few percent of queries)
    assert (gaps[bad] < TOL).all()
    print(f"\none-range ranking: {len(pick) - bad.sum()} of {len(pick)} sampled queries exact, "
          f"{bad.sum()} swapped across gaps < {TOL} ({(gaps < TOL).sum()} have such a gap)")
    assert ((order >= 0) & (order < nlist)).all()


@pytest.mark.parametrize("nlist,d,nprobe", [(5000, 96, 256), (2500, 36, 100), (16384, 64, 128),
                                             (9000, 96, 200), (65536, 32, 256), (8192, 160, 128)])
def test_rank_parity_many_centroids(nlist, d, nprobe, dev):
    """Rankings over more centroids than one selecting warp holds, with d not
    a multiple of the 64-element K-block, against the fp64 oracle ranking;
    rank swaps only across score gaps below the tolerance.  Fewer 32-centroid
    groups than nprobe take the level-by-level selection, the others the
    group-maximum threshold: with a score table and one compacting pass for
    d > 128, else with a second contraction that keeps only the scores that
    reach it."""
    rng = np.random.default_rng(nlist + d)
    C = rng.standard_normal((nlist, d)).astype(np.float32)
    C /= np.linalg.norm(C, axis=1, keepdims=True)
    Q = (C[rng.integers(0, nlist, 700)] + 0.3 * rng.standard_normal((700, d))).astype(np.float32)
    Q /= np.linalg.norm(Q, axis=1, keepdims=True)
    Cd = torch.from_numpy(C).to(dev)
    index = sieve.build_layout(Cd.clone(), torch.arange(nlist, dtype=torch.int32, device=dev),
                               nlist, Cd)
    order, sc = sieve.rank_partitions(index, torch.from_numpy(Q).to(dev), nprobe, return_scores=True)
    order, sc = order.cpu().numpy(), sc.cpu().numpy()
    ref, rsc = oracle.rank(Q, C, nprobe + 1, return_scores=True)
    assert np.abs(sc - rsc[:, :nprobe]).max() <= TOL
    gaps = (rsc[:, :-1] - rsc[:, 1:]).min(axis=1)
    bad = (order != ref[:, :nprobe]).any(axis=1)
    assert (gaps[bad] < TOL).all()
    assert bad.sum() <= 0.02 * len(Q)
    # every row is a permutation prefix: distinct ids in range
    assert ((order >= 0) & (order < nlist)).all()
    assert all(len(set(r)) == nprobe for r in order[:50])


@pytest.mark.parametrize("lookahead", [0, 1])
def test_search_parity_tiny(tiny, g_tiny, lookahead):
    c = tiny["cfg"]
    got, ref, rep = check(tiny, g_tiny, tiny["Q"], tiny["qids"], c.tau, c.k, c.nprobe, c.W,
                          lookahead)
    assert rep["exact"] >= 0.99 * len(tiny["Q"])
    assert (got["count"] > 0).any()


@pytest.mark.parametrize("W", [1, 2, 3, 5, 24])
@pytest.mark.parametrize("lookahead", [0, 1])
def test_search_parity_deep(deep, g_deep, W, lookahead):
    c = deep["cfg"]
    check(deep, g_deep, deep["Q"], deep["qids"], c.tau, c.k, c.nprobe, W, lookahead)


@pytest.mark.parametrize("path", ["simt", "tensor"])
def test_schedule_changes_nothing(deep, g_deep, path):
    """Lookahead on/off, per-round caps and the loop mode give bit-identical
    output (Sec. 4.2: the microbatch cap only splits groups; Sec. 4.3).  The
    scan path is fixed: each path computes a pair's similarity the same way
    whatever group it lands in, the two paths round differently."""
    c = deep["cfg"]
    Q, qids = deep["Q"], deep["qids"]
    base = run(g_deep, Q, qids, c.tau, c.k, c.nprobe, c.W, lookahead=1, scan_path=path)
    variants = [dict(lookahead=0), dict(lookahead=1, max_items_per_round=4096),
                dict(lookahead=1, max_items_per_round=7), dict(lookahead=0, loop=1),
                dict(lookahead=1, loop=1, max_items_per_round=100),
                # the serial traversal (Sec. 6.3): every item its own partition call
                dict(lookahead=0, serial=True), dict(lookahead=1, serial=True),
                dict(lookahead=1, serial=True, loop=1, max_items_per_round=100)]
    for kw in variants:
        got = run(g_deep, Q, qids, c.tau, c.k, c.nprobe, c.W, scan_path=path, **kw)
        for key in ("ids", "scores", "count", "probes"):
            assert np.array_equal(got[key], base[key]), (kw, key)
    sub = slice(0, 25)   # a cap of one item per round: one search per round
    one = run(g_deep, Q[sub], qids[sub], c.tau, c.k, c.nprobe, c.W, lookahead=1,
              max_items_per_round=1, stats=True, scan_path=path)
    for key in ("ids", "scores", "count", "probes"):
        assert np.array_equal(one[key], base[key][sub]), key
    assert one["stats"]["rounds"] >= one["probes"].sum()
    # serial traversal: as many tiles as items, one query per partition call
    ser = run(g_deep, Q, qids, c.tau, c.k, c.nprobe, c.W, lookahead=0, serial=True, stats=True,
              scan_path=path)
    assert ser["stats"]["tiles"] == ser["stats"]["items"] == base["probes"].sum()


@pytest.mark.parametrize("path", ["simt", "tensor", "auto"])
def test_scan_paths_parity(tiny, g_tiny, deep, g_deep, path):
    """Both contraction paths (FP32 FMA, the tensor-core fp16 split) and the
    automatic choice meet the parity bar, on groups of every size (the
    automatic path screens at W = infinity)."""
    c = tiny["cfg"]
    for la in (0, 1):
        check(tiny, g_tiny, tiny["Q"], tiny["qids"], c.tau, c.k, c.nprobe, c.W, la, scan_path=path)
    c = deep["cfg"]
    check(deep, g_deep, deep["Q"], deep["qids"], c.tau, c.k, c.nprobe, c.W, 1, scan_path=path)
    check(deep, g_deep, deep["Q"], deep["qids"], c.tau, c.k, c.nprobe, BIG_W, 1, scan_path=path)


def test_tensor_path_scores_match_fp64(tiny, g_tiny, dev):
    """Every returned similarity of the three-product fp16 split is within 1e-6
    of the fp64 inner product of the same pair (the split's error bound, well
    inside the 1e-5 tolerance)."""
    c = tiny["cfg"]
    got = run(g_tiny, tiny["Q"], tiny["qids"], 0.5, 16, c.nprobe, BIG_W, lookahead=1,
              scan_path="tensor")
    ids, sc, cnt = got["ids"], got["scores"], got["count"]
    valid = np.arange(16)[None, :] < cnt[:, None]
    qi, kj = np.nonzero(valid)
    exact = np.einsum("ij,ij->i", tiny["Q"][qi].astype(np.float64),
                      tiny["X"][ids[qi, kj]].astype(np.float64))
    assert len(qi) > 1000
    assert np.abs(sc[qi, kj] - exact).max() <= 1e-6


@pytest.mark.parametrize("W", [16, BIG_W])
def test_window_at_least_nprobe_is_fixed_probe(tiny, g_tiny, W):
    c = tiny["cfg"]
    got = run(g_tiny, tiny["Q"], tiny["qids"], c.tau, c.k, c.nprobe, W, lookahead=1)
    assert (got["probes"] == c.nprobe).all()
    order = oracle.rank(tiny["Q"], tiny["centroids"], c.nprobe)
    fp = oracle.fixed_probe(index_of(tiny), tiny["Q"], c.tau, c.k, c.nprobe, order,
                            qids=tiny["qids"])
    fp["probes"] = np.full(len(order), c.nprobe, np.int32)
    assert_parity(compare(got, fp, index_of(tiny), tiny["Q"], tiny["qids"], c.tau, c.k,
                          c.nprobe, order))


def test_full_probe_is_bruteforce(tiny, g_tiny):
    c = tiny["cfg"]
    Q, qids = tiny["Q"][:300], tiny["qids"][:300]
    got = run(g_tiny, Q, qids, c.tau, c.k, 64, BIG_W, lookahead=1)
    bf = oracle.bruteforce(tiny["X"], tiny["ids"], Q, c.tau, c.k, qids=qids)
    bf["probes"] = np.full(len(Q), 64, np.int32)
    order = oracle.rank(Q, tiny["centroids"], 64)
    assert_parity(compare(got, bf, index_of(tiny), Q, qids, c.tau, c.k, 64, order))


def test_given_order_and_host_variant(tiny, g_tiny, dev):
    c = tiny["cfg"]
    Q = torch.from_numpy(tiny["Q"]).to(dev)
    qids = torch.from_numpy(tiny["qids"]).to(dev)
    base = sieve.search(g_tiny, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids)
    order = sieve.rank_partitions(g_tiny, Q, c.nprobe)
    given = sieve.search(g_tiny, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=order)
    host = sieve.search_host(g_tiny, torch.from_numpy(tiny["Q"]).pin_memory(), c.tau, c.k,
                             c.nprobe, c.W, query_ids_host=torch.from_numpy(tiny["qids"]))
    for a, b, h in zip(base, given, host):
        assert torch.equal(a.cpu(), b.cpu())
        assert torch.equal(a.cpu(), h)


def test_host_variant_uploads_in_chunks(dev):
    """50K queries: sieve_search_host uploads them in three chunks, ranking each
    as it lands (the copy overlaps the ranking); the results are the device
    call's, bit for bit, on the tensor and the FP32 ranking."""
    cfg = synth.scaled("tiny", n=60_000, nq=50_000, nlist=96, ncomp=96, seed=23)
    w = synth.to_numpy(synth.make_workload(cfg, device="cpu"))
    index = sieve.build_layout(torch.from_numpy(w["X"]).to(dev), torch.from_numpy(w["assign"]).to(dev),
                               cfg.nlist, torch.from_numpy(w["centroids"]).to(dev))
    Q = torch.from_numpy(w["Q"])
    qids = torch.from_numpy(w["qids"])
    for path in ("auto", "simt"):
        base = sieve.search(index, Q.to(dev), cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                            query_ids=qids.to(dev), scan_path=path)
        host = sieve.search_host(index, Q.pin_memory(), cfg.tau, cfg.k, cfg.nprobe, cfg.W,
                                 query_ids_host=qids, scan_path=path)
        for a, h in zip(base, host):
            assert torch.equal(a.cpu(), h), path


def test_stats_account_for_the_work(deep, g_deep):
    c = deep["cfg"]
    got = run(g_deep, deep["Q"], deep["qids"], c.tau, c.k, c.nprobe, c.W, lookahead=0, stats=True)
    st = got["stats"]
    assert st["status"] == 0
    assert st["items"] == got["probes"].sum()           # each committed rank searched once
    assert st["rounds"] == got["probes"].max() + 0      # one rank per query per round
    sizes = np.bincount(deep["assign"], minlength=c.nlist)
    order = oracle.rank(deep["Q"], deep["centroids"], c.nprobe)
    want_pairs = sum(sizes[order[i, :got["probes"][i]]].sum() for i in range(len(order)))
    assert st["pairs"] == want_pairs


# ---------------------------------------------------------------------------
# edge cases


def test_empty_and_single_query(tiny, g_tiny, dev):
    c = tiny["cfg"]
    empty = torch.empty((0, 64), dtype=torch.float32, device=dev)
    ids, sc, cnt, pr = sieve.search(g_tiny, empty, c.tau, c.k, c.nprobe, c.W)
    assert ids.shape == (0, c.k) and pr.shape == (0,)
    check(tiny, g_tiny, tiny["Q"][:1], tiny["qids"][:1], c.tau, c.k, c.nprobe, c.W, 1)


@pytest.mark.parametrize("k", [1, 3, 33, 64])
@pytest.mark.parametrize("path", ["auto", "simt"])
def test_k_range(deep, g_deep, k, path):
    """Large k on the tensor cores (bulk pipeline) and on FP32 FMA."""
    c = deep["cfg"]
    check(deep, g_deep, deep["Q"], deep["qids"], c.tau, k, c.nprobe, c.W, 1, scan_path=path)


def test_k_on_the_converter_pipeline(deep, g_deep):
    """Without the tensor layout the converter pipeline keeps k-lists up to
    k = 22 on the tensor cores; larger k falls back to FP32 FMA."""
    c = deep["cfg"]
    plain = g_deep.without_tc_layout()
    for k in (20, 22, 40):
        check(deep, plain, deep["Q"], deep["qids"], c.tau, k, c.nprobe, c.W, 1)


def test_no_query_ids_and_low_tau(deep, g_deep):
    c = deep["cfg"]
    check(deep, g_deep, deep["Q"][:100], None, 0.5, c.k, 8, 2, 1)


def _hand_index(dev, X, assign, C):
    Xd = torch.from_numpy(np.asarray(X, np.float32)).to(dev)
    a = torch.from_numpy(np.asarray(assign, np.int32)).to(dev)
    Cd = torch.from_numpy(np.asarray(C, np.float32)).to(dev)
    return sieve.build_layout(Xd, a, Cd.shape[0], Cd)


def test_tau_boundary_self_ties_padding(dev):
    q = np.array([[1, 0, 0, 0]], np.float32)
    X = np.array([[0.5, 0.5, 0.5, 0.5], [0.5, 0.5, 0.5, 0.5], [1, 0, 0, 0], [0, 1, 0, 0],
                  [0.5, -0.5, 0.5, 0.5]], np.float32)
    # external ids are row numbers; the query is row 2
    idx = _hand_index(dev, X, [0] * 5, q)
    Qd = torch.from_numpy(q).to(dev)
    ids, sc, cnt, pr = sieve.search(idx, Qd, 0.5, 4, 1, 1, query_ids=torch.tensor([2], device=dev))
    assert cnt.item() == 3 and pr.item() == 1
    assert ids[0].tolist() == [0, 1, 4, -1]
    assert sc[0, :3].tolist() == [0.5, 0.5, 0.5] and sc[0, 3].item() == float("-inf")
    above = float(np.nextafter(np.float32(0.5), np.float32(1)))
    ids, sc, cnt, pr = sieve.search(idx, Qd, above, 4, 1, 1, query_ids=torch.tensor([2], device=dev))
    assert cnt.item() == 0 and ids[0].tolist() == [-1] * 4


def test_empty_partitions_and_odd_dimension(dev):
    rng = np.random.default_rng(5)
    d, nlist = 36, 10
    C = rng.normal(size=(nlist, d)).astype(np.float32)
    C /= np.linalg.norm(C, axis=1, keepdims=True)
    X = np.repeat(C[:6], 150, axis=0) + 0.05 * rng.normal(size=(900, d)).astype(np.float32)
    X = (X / np.linalg.norm(X, axis=1, keepdims=True)).astype(np.float32)
    assign = np.argmax(X @ C.T, axis=1).astype(np.int32)       # partitions 6..9 stay empty
    w = {"X": X, "ids": np.arange(900, dtype=np.int64), "assign": assign, "centroids": C}
    gidx = _hand_index(dev, X, assign, C)
    Q = X[::9].copy()
    qids = np.arange(0, 900, 9, dtype=np.int64)
    for W in (1, 3, BIG_W):
        check(w, gidx, Q, qids, 0.9, 7, nlist, W, 1)


def test_invalid_arguments_raise(tiny, g_tiny, dev):
    Q = torch.from_numpy(tiny["Q"][:4]).to(dev)
    with pytest.raises(sieve.SieveError):   # converter pipeline: k-lists up to k = 22 fit
        sieve.search(g_tiny.without_tc_layout(), Q, 0.9, 23, 16, 4, scan_path="tensor")
    for kw in (dict(k=0), dict(k=65), dict(nprobe=65), dict(W=0)):
        args = dict(tau=0.9, k=10, nprobe=16, W=4)
        args.update(kw)
        with pytest.raises(sieve.SieveError):
            sieve.search(g_tiny, Q, **args)
    with pytest.raises(sieve.SieveError):
        sieve.search(g_tiny, Q, float("nan"), 10, 16, 4)
    tiny_ws = sieve.Workspace()
    tiny_ws.buf = torch.empty(256, dtype=torch.uint8, device=dev)
    tiny_ws.get = lambda n, d: tiny_ws.buf     # hand the call a too-small buffer
    with pytest.raises(sieve.SieveError) as e:
        sieve.search(g_tiny, Q, 0.9, 10, 16, 4, workspace=tiny_ws)
    assert e.value.status == -3


# ---------------------------------------------------------------------------
# tensor-core layout


def np_tc_layout(X, off, d):
    """The tensor-core layout written independently with numpy: blocks of 128
    rows, per K-block of 64 elements 16 KB hi fp16 + 16 KB lo fp16 with
    hi = fp16(256 x), lo = fp16(256 x - hi); 16-byte chunk c of row r at
    chunk c ^ (r & 7); rows past a partition's end are zero."""
    nkb = (d + 63) // 64
    parts = []
    for p in range(len(off) - 1):
        rows = X[off[p]:off[p + 1]].astype(np.float32)
        nb = -(-len(rows) // 128)
        pad = np.zeros((nb * 128, nkb * 64), np.float32)
        pad[:len(rows), :d] = rows
        for b in range(nb):
            for kb in range(nkb):
                blk = pad[b * 128:(b + 1) * 128, kb * 64:(kb + 1) * 64] * np.float32(256)
                hi = blk.astype(np.float16)
                lo = (blk - hi.astype(np.float32)).astype(np.float16)
                out = []
                for t in (hi, lo):
                    tile = np.zeros((128, 8, 8), np.float16)
                    for c in range(8):
                        for r in range(128):
                            tile[r, c ^ (r & 7)] = t[r, c * 8:(c + 1) * 8]
                    out.append(tile.reshape(-1).view(np.uint8))
                parts.append(np.concatenate(out))
    return np.concatenate(parts) if parts else np.zeros(0, np.uint8)


def test_tc_layout_bytes(deep, g_deep):
    assert g_deep.tc_rows is not None
    off = g_deep.list_offsets.cpu().numpy()
    X = g_deep.vectors.cpu().numpy()
    ref = np_tc_layout(X, off, X.shape[1])
    got = g_deep.tc_rows.cpu().numpy()[:ref.size]
    assert got.size == ref.size and np.array_equal(got, ref)
    nb = [-(-(off[p + 1] - off[p]) // 128) for p in range(len(off) - 1)]
    assert (g_deep.tc_row_blocks.cpu().numpy() == np.concatenate([[0], np.cumsum(nb)])).all()
    C = g_deep.centroids.cpu().numpy()
    refc = np_tc_layout(C, np.array([0, C.shape[0]]), C.shape[1])
    assert np.array_equal(g_deep.tc_centroids.cpu().numpy()[:refc.size], refc)


@pytest.mark.parametrize("which", ["tiny", "deep"])
def test_bulk_path_equals_converter_path(which, tiny, g_tiny, deep, g_deep):
    """The tensor-core scan fed by bulk copies of the pre-split layout computes
    the same products in the same order as the one that splits fp32 rows on
    the fly: identical ids, counts and probes, scores within 1e-6."""
    w, g = (tiny, g_tiny) if which == "tiny" else (deep, g_deep)
    c = w["cfg"]
    a = run(g, w["Q"], w["qids"], c.tau, c.k, c.nprobe, c.W, scan_path="tensor")
    b = run(g.without_tc_layout(), w["Q"], w["qids"], c.tau, c.k, c.nprobe, c.W, scan_path="tensor")
    for key in ("ids", "count", "probes"):
        assert np.array_equal(a[key], b[key]), key
    valid = np.arange(c.k)[None, :] < a["count"][:, None]
    assert np.abs(a["scores"][valid] - b["scores"][valid]).max(initial=0) <= 1e-6


def test_wide_rows_fall_back_and_match(dev):
    """d = 320 is beyond the resident-A limit of the bulk pipeline: the search
    uses the converter pipeline even with a layout present, and matches the
    oracle."""
    import synth
    cfg = synth.scaled("tiny", n=4_000, d=320, ncomp=8, nlist=16, nq=150, dup_frac=0.1,
                       dup_counts=("uniform", 1, 4), dup_sigma=(0.005, 0.02), tau=0.9,
                       nprobe=8, W=2, seed=21)
    w = synth.to_numpy(synth.make_workload(cfg))
    assert gpu_index(w, dev).tc_rows is None   # not built by default past d = 256
    gidx = gpu_index(w, dev, tc_layout=True)
    assert gidx.tc_rows is not None
    for path in ("tensor", "auto"):
        check(w, gidx, w["Q"], w["qids"], cfg.tau, cfg.k, cfg.nprobe, cfg.W, 1, scan_path=path)


def test_device_error_reported_without_stats(tiny, g_tiny, dev):
    """An order entry outside [0, nlist) is caught on the device.  In graph
    mode without stats the call returns at once; sieve_search_status then
    reads SIEVE_EINVAL from the workspace, and search(check=True) raises.
    Host-driven rounds return it directly.  A correct call on the same
    workspace afterwards reports 0."""
    c = tiny["cfg"]
    Q = torch.from_numpy(tiny["Q"][:200]).to(dev)
    qids = torch.from_numpy(tiny["qids"][:200]).to(dev)
    order = sieve.rank_partitions(g_tiny, Q, c.nprobe)
    bad = order.clone()
    bad[7, 3] = -1
    ws = sieve.Workspace()
    sieve.search(g_tiny, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=bad, workspace=ws)
    assert sieve.search_status(ws) == -1
    with pytest.raises(sieve.SieveError) as ei:
        sieve.search(g_tiny, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=bad,
                     workspace=ws, check=True)
    assert ei.value.status == -1
    with pytest.raises(sieve.SieveError):
        sieve.search(g_tiny, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=bad,
                     workspace=ws, loop=1)
    sieve.search(g_tiny, Q, c.tau, c.k, c.nprobe, c.W, query_ids=qids, order=order, workspace=ws,
                 check=True)
    assert sieve.search_status(ws) == 0
