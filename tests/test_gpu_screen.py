"""The screening scan (scan_path "screen", and the automatic path from a
window of 16 up or at d >= 192, from tau 0.85 up, with the tensor-core layout): one fp16 product of the hi
halves per (query, row) pair bounds every score, and only the rows whose
bound reaches the threshold are scored again in fp32.

The rows here are built so that their exact scores sit at chosen distances
from tau and from the k-th kept score, inside and outside the screen's error
band (about 1.3e-3 for unit vectors at d = 128), with rows and queries of
unit norm and of other norms.  Every distance is at least 2e-5, so no query
is fragile: ids, counts and probes must equal the oracle's exactly."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_03199_gb300 as sieve
from parity import TOL, assert_parity, compare

pytestmark = pytest.mark.gpu

BIG_W = 2**31 - 1
TAU = 0.9
# distances from tau of the planted rows: inside and outside the band
OFFSETS = (-3e-3, -1.2e-3, -6e-4, -3e-4, -1e-4, -2e-5, 2e-5, 1e-4, 3e-4, 6e-4, 1.2e-3)


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _unit(v):
    return v / np.linalg.norm(v, axis=-1, keepdims=True)


def planted(seed, d=128, nq=96, nlist=12, scaled=False):
    """Queries with planted rows at exact target scores t: row = (t / |q|) q^
    + c u, u a unit vector orthogonal to q, so <q, row> = t whatever c is.
    Per query: one row per offset from tau, and 14 rows above tau spaced
    2.5e-4 apart with rows 3e-5 below and above the 10th best (the kept
    list's own threshold), plus random rows.  scaled: query norms in
    [0.6, 1.6], planted rows with c in [0, 1.5] and random rows of norm
    0.4 to 1.8 (unrelated pairs stay far below tau at d = 128)."""
    rng = np.random.default_rng(seed)
    Q = _unit(rng.standard_normal((nq, d)))
    qn = rng.uniform(0.6, 1.6, nq) if scaled else np.ones(nq)
    rows = []
    for i in range(nq):
        qh = Q[i]
        targets = [TAU + o for o in OFFSETS]
        top = [TAU + 0.004 + 2.5e-4 * j for j in range(14)]
        kth = sorted(top, reverse=True)[9]
        targets += top + [kth - 3e-5, kth + 3e-5]
        for t in targets:
            u = rng.standard_normal(d)
            u = _unit(u - (u @ qh) * qh)
            a = t / qn[i]
            if scaled:
                c = rng.uniform(0.0, 1.5)
            else:
                c = np.sqrt(max(0.0, 1.0 - a * a))
            rows.append(a * qh + c * u)
    X = np.concatenate([np.asarray(rows), _unit(rng.standard_normal((4000, d)))])
    if scaled:
        X[-4000:] *= rng.uniform(0.4, 1.8, (4000, 1))
    Qs = (Q * qn[:, None]).astype(np.float32)
    X = X.astype(np.float32)
    C = _unit(rng.standard_normal((nlist, d))).astype(np.float32)
    assign = np.argmax(X.astype(np.float64) @ C.astype(np.float64).T, axis=1).astype(np.int32)
    return {"X": X, "ids": np.arange(len(X), dtype=np.int64), "assign": assign, "centroids": C,
            "Q": Qs}


def gpu_index(w, dev):
    X = torch.from_numpy(w["X"]).to(dev)
    cent = torch.from_numpy(w["centroids"]).to(dev)
    return sieve.build_layout(X, torch.from_numpy(w["assign"]).to(dev), cent.shape[0], cent,
                              tc_layout=True)


def run(index, Q, tau, k, nprobe, W, **kw):
    dev = index.vectors.device
    out = sieve.search(index, torch.from_numpy(Q).to(dev), tau, k, nprobe, W, **kw)
    torch.cuda.synchronize()
    return {"ids": out[0].cpu().numpy(), "scores": out[1].cpu().numpy(),
            "count": out[2].cpu().numpy(), "probes": out[3].cpu().numpy()}


def idx_of(w):
    return {key: w[key] for key in ("X", "ids", "assign", "centroids")}


def assert_exact(got, ref, k):
    """ids, counts and probes equal; scores within the parity tolerance."""
    assert np.array_equal(got["probes"], ref["probes"])
    assert np.array_equal(got["count"], ref["count"])
    assert np.array_equal(got["ids"], ref["ids"])
    valid = np.arange(k)[None, :] < ref["count"][:, None]
    assert np.abs(got["scores"][valid] - ref["scores"][valid]).max(initial=0) <= TOL


@pytest.mark.parametrize("scaled", [False, True])
@pytest.mark.parametrize("k", [10, 20])
def test_screen_band_matches_oracle(dev, scaled, k):
    w = planted(7 + scaled, scaled=scaled)
    g = gpu_index(w, dev)
    nlist = w["centroids"].shape[0]
    ref = oracle.search(idx_of(w), w["Q"], TAU, k, nlist, BIG_W)
    for path in ("auto", "screen", "tensor"):
        got = run(g, w["Q"], TAU, k, nlist, BIG_W, scan_path=path)
        assert_exact(got, ref, k)
    # each query keeps its planted rows at or above tau, and the top-k cut
    assert (ref["count"] == k).all()


def test_screen_band_with_stopping(dev):
    """The same rows under the stopping rule (W = 2, lookahead on and off):
    the hits that move the stop line are decided on the rescored values."""
    w = planted(11)
    g = gpu_index(w, dev)
    nlist = w["centroids"].shape[0]
    ref = oracle.search(idx_of(w), w["Q"], TAU, 10, nlist, 2)
    for la in (True, False):
        got = run(g, w["Q"], TAU, 10, nlist, 2, lookahead=la, scan_path="screen")
        assert_exact(got, ref, 10)


def test_screen_equals_three_products_on_tiny(tiny, dev):
    """The screen and the three-product scan on the tiny workload, each
    against the oracle (W = 4, the workload's own setting)."""
    c = tiny["cfg"]
    X = torch.from_numpy(tiny["X"]).to(dev)
    cent = torch.from_numpy(tiny["centroids"]).to(dev)
    g = sieve.build_layout(X, torch.from_numpy(tiny["assign"]).to(dev), cent.shape[0], cent,
                           tc_layout=True)
    idx = {key: tiny[key] for key in ("X", "ids", "assign", "centroids")}
    ref = oracle.search(idx, tiny["Q"], c.tau, c.k, c.nprobe, c.W, qids=tiny["qids"])
    order = oracle.rank(tiny["Q"], tiny["centroids"], c.nprobe)
    outs = {}
    for path in ("screen", "tensor"):
        qd = torch.from_numpy(tiny["qids"]).to(dev)
        out = sieve.search(g, torch.from_numpy(tiny["Q"]).to(dev), c.tau, c.k, c.nprobe, c.W,
                           query_ids=qd, scan_path=path)
        got = {"ids": out[0].cpu().numpy(), "scores": out[1].cpu().numpy(),
               "count": out[2].cpu().numpy(), "probes": out[3].cpu().numpy()}
        assert_parity(compare(got, ref, idx, tiny["Q"], tiny["qids"], c.tau, c.k, c.nprobe, order))
        outs[path] = got
    for key in ("ids", "count", "probes"):
        assert np.array_equal(outs["screen"][key], outs["tensor"][key]), key


def test_layout_block_norms(dev):
    """The fp32 after the layout's blocks: the largest row norm of each block
    of 128 rows of a partition (the screen's bound uses it)."""
    w = planted(3, scaled=True)
    g = gpu_index(w, dev)
    off = g.list_offsets.cpu().numpy()
    X = g.vectors.cpu().numpy().astype(np.float64)
    norms = []
    for p in range(len(off) - 1):
        for b0 in range(off[p], off[p + 1], 128):
            norms.append(np.linalg.norm(X[b0:min(b0 + 128, off[p + 1])], axis=1).max())
    nblocks = len(norms)
    blocks = g.tc_row_blocks.cpu().numpy()
    assert blocks[-1] == nblocks
    per_block = 32768 * ((X.shape[1] + 63) // 64)
    raw = g.tc_rows.cpu().numpy()[nblocks * per_block: nblocks * per_block + 4 * nblocks]
    got = raw.view(np.float32).astype(np.float64)
    assert np.allclose(got, norms, rtol=2e-6, atol=0)
