"""Seeded synthetic workloads for the threshold-aware IVF search.

This module only makes inputs: clustered unit-norm embeddings with planted
near-duplicates, database-drawn queries, and the IVF index those queries search
(spherical k-means centroids plus the exact nearest-centroid assignment of every
row, the build-time precondition of the method, Sec. 4.4).  It holds none of the
search's arithmetic: no ranking of centroids for queries, no partition scan, no
tau test, no top-k, no stopping rule.  Both the CUDA path and the fp64 oracle
read the arrays it returns; neither is imported here.

The paper's workloads (four proprietary 10M x 768 Hunyuan sets, LAION-100M and
DEEP-100M, Sec. 3.1 / Sec. 6.1) are not available, so these seeded sets stand
in for them with the shapes of the evaluated configurations:

* a Gaussian mixture on the sphere: component means mu_c = normalize(N(0, I_d)),
  component weights uniform or Zipf(s), base point
  x = normalize(mu_c + sigma_c * g / sqrt(d)) with sigma_c ~ U[0.7, 1.3], so
  two members of one component have cosine near 1 / (1 + sigma_c^2), well
  below the thresholds used (0.90 - 0.95);
* planted near-duplicates: a seeded set of parent records each gets a number
  of copies normalize(parent + sigma * g), g ~ N(0, I_d), whose cosine to the
  parent is about (1 + d sigma^2)^(-1/2) and straddles tau over sigma's range
  (heavy-tailed threshold-neighbour density, as in Fig. 1a);
* rows shuffled by a seeded permutation; the id of a row is its position;
* queries drawn uniformly without replacement from the rows (self-join
  deduplication: each query's own row is excluded by its id);
* the index: spherical k-means (seeded init from data points, Lloyd steps
  with re-normalised centroids, empty clusters re-seeded) on a seeded sample of
  at most ``train_cap`` rows, then every row assigned to its nearest centroid
  (largest inner product, lower centroid id on ties).
"""
from __future__ import annotations

import math
import os
from dataclasses import dataclass, field, replace

# deterministic cuBLAS reductions for the k-means matmuls (read when cuBLAS
# starts, so this must precede the first GPU matmul)
os.environ.setdefault("CUBLAS_WORKSPACE_CONFIG", ":4096:8")

import torch  # noqa: E402


@dataclass(frozen=True)
class Workload:
    name: str
    n: int                 # rows, copies included
    d: int
    ncomp: int             # mixture components
    zipf: float | None     # None = uniform component weights
    dup_frac: float        # parents as a fraction of n
    dup_counts: tuple      # ("uniform", lo, hi) or ("powerlaw", alpha, max)
    dup_sigma: tuple       # (lo, hi) of the copy noise sigma
    nlist: int
    nq: int
    tau: float
    k: int
    nprobe: int
    W: int
    kmeans_iters: int = 10
    train_cap: int | None = None
    seed: int = 1
    sweep_W: tuple = field(default_factory=tuple)


CONFIGS = {
    # N=20,000 d=64, 64 uniform components, 5% of records get 1-5 copies with
    # sigma 0.02, nlist 64, 1,000 queries, tau 0.90, k 10, nprobe 16, W 4
    "tiny": Workload("tiny", 20_000, 64, 64, None, 0.05, ("uniform", 1, 5), (0.02, 0.02),
                     64, 1_000, 0.90, 10, 16, 4, seed=1),
    # 1M d=256, 1,024 Zipf(1.1) components, power-law (alpha 2) copy counts,
    # sigma 0.01-0.05, nlist 1,024, 100K queries, tau 0.90, k 10, nprobe 64, W 8
    "1m": Workload("1m", 1_000_000, 256, 1024, 1.1, 0.03, ("powerlaw", 2.0, 1000), (0.01, 0.05),
                   1024, 100_000, 0.90, 10, 64, 8, train_cap=256 * 1024, seed=2,
                   sweep_W=(2, 4, 8, 16, 64)),
    # 10M d=512, 16,384 Zipf components, heavy-tailed duplicates (power-law
    # alpha 1.5 copy counts up to 1,000: about 23 copies per parent, so 0.2% of
    # the rows as parents make about 5% of the rows copies), nlist 16,384,
    # 1M queries, tau 0.92, nprobe 128, W 8
    "10m512": Workload("10m512", 10_000_000, 512, 16384, 1.1, 0.002, ("powerlaw", 1.5, 1000),
                       (0.005, 0.03), 16384, 1_000_000, 0.92, 10, 128, 8,
                       train_cap=256 * 16384, seed=3),
    # 10M d=256, near-uniform density, 0.5% planted duplicates, nlist 8,192,
    # 1M queries, tau 0.95, nprobe 128, W in {4, 8, 16}
    "10m256": Workload("10m256", 10_000_000, 256, 8192, None, 0.005, ("uniform", 1, 5),
                       (0.005, 0.03), 8192, 1_000_000, 0.95, 10, 128, 8,
                       train_cap=256 * 8192, seed=4, sweep_W=(4, 8, 16)),
    # 100M d=96, 65,536 components, 2% planted duplicates, nlist 65,536,
    # 1M queries, tau 0.90, nprobe 256, W 8
    "100m": Workload("100m", 100_000_000, 96, 65536, 1.1, 0.02, ("uniform", 1, 5),
                     (0.01, 0.08), 65536, 1_000_000, 0.90, 10, 256, 8,
                     train_cap=256 * 65536, seed=5),
}


def scaled(name: str, **overrides) -> Workload:
    """A copy of a named workload with some fields replaced (smaller test cases)."""
    return replace(CONFIGS[name], **overrides)


def _normalize(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=1, keepdim=True).clamp_min(1e-30)


def _copy_counts(cfg: Workload, m: int, g: torch.Generator, device) -> torch.Tensor:
    kind = cfg.dup_counts[0]
    if kind == "uniform":
        lo, hi = cfg.dup_counts[1], cfg.dup_counts[2]
        return torch.randint(lo, hi + 1, (m,), generator=g, device=device)
    if kind == "powerlaw":
        alpha, cmax = cfg.dup_counts[1], cfg.dup_counts[2]
        c = torch.arange(1, cmax + 1, device=device, dtype=torch.float64)
        w = c.pow(-alpha)
        return torch.multinomial(w / w.sum(), m, replacement=True, generator=g) + 1
    raise ValueError(kind)


@torch.no_grad()
def make_corpus(cfg: Workload, device="cpu", chunk: int = 1 << 20):
    """Rows X [n][d] fp32 unit-norm, in a seeded shuffled order (id = row)."""
    g = torch.Generator(device=device).manual_seed(cfg.seed)
    n, d = cfg.n, cfg.d
    mu = _normalize(torch.randn(cfg.ncomp, d, generator=g, device=device))
    sig_c = 0.7 + 0.6 * torch.rand(cfg.ncomp, generator=g, device=device)
    if cfg.zipf is None:
        w = torch.ones(cfg.ncomp, device=device, dtype=torch.float64)
    else:
        w = torch.arange(1, cfg.ncomp + 1, device=device, dtype=torch.float64).pow(-cfg.zipf)
    w = w / w.sum()

    m = int(round(cfg.dup_frac * n))
    counts = _copy_counts(cfg, m, g, device) if m > 0 else torch.zeros(0, dtype=torch.long,
                                                                         device=device)
    total_copies = int(counts.sum().item())
    n_base = n - total_copies
    if n_base < m:
        raise ValueError("duplicate settings leave fewer base rows than parents")

    X = torch.empty(n, d, device=device, dtype=torch.float32)
    # base rows
    for s in range(0, n_base, chunk):
        e = min(n_base, s + chunk)
        comp = torch.multinomial(w, e - s, replacement=True, generator=g)
        noise = torch.randn(e - s, d, generator=g, device=device)
        X[s:e] = _normalize(mu[comp] + sig_c[comp, None] * noise / math.sqrt(d))
    # copies: parents are base rows 0..m-1 (base rows are i.i.d.)
    parent = torch.repeat_interleave(torch.arange(m, device=device), counts)
    lo, hi = cfg.dup_sigma
    for s in range(0, total_copies, chunk):
        e = min(total_copies, s + chunk)
        sig = lo + (hi - lo) * torch.rand(e - s, generator=g, device=device)
        noise = torch.randn(e - s, d, generator=g, device=device)
        X[n_base + s:n_base + e] = _normalize(X[parent[s:e]] + sig[:, None] * noise)
    perm = torch.randperm(n, generator=g, device=device)
    X = X[perm]
    return X, g


@torch.no_grad()
def _nearest(X: torch.Tensor, Cn: torch.Tensor, chunk: int) -> torch.Tensor:
    out = torch.empty(X.shape[0], dtype=torch.int32, device=X.device)
    for s in range(0, X.shape[0], chunk):
        e = min(X.shape[0], s + chunk)
        out[s:e] = torch.argmax(X[s:e] @ Cn.T, dim=1).to(torch.int32)
    return out


@torch.no_grad()
def build_index(X: torch.Tensor, cfg: Workload, g: torch.Generator, chunk: int = 1 << 16):
    """Spherical k-means centroids [nlist][d] (unit) and exact assignment [n] int32."""
    prev = torch.backends.cuda.matmul.allow_tf32
    prev_det = torch.are_deterministic_algorithms_enabled()
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.use_deterministic_algorithms(True, warn_only=True)   # same index on every run
    try:
        n = X.shape[0]
        cap = cfg.train_cap or n
        if n > cap:
            T = X[torch.randperm(n, generator=g, device=X.device)[:cap]]
        else:
            T = X
        Cn = T[torch.randperm(T.shape[0], generator=g, device=X.device)[:cfg.nlist]].clone()
        for _ in range(cfg.kmeans_iters):
            a = _nearest(T, Cn, chunk).long()
            sums = torch.zeros_like(Cn).index_add_(0, a, T)
            cnt = torch.bincount(a, minlength=cfg.nlist)
            empty = (cnt == 0).nonzero().flatten()
            if empty.numel():
                pick = torch.randint(0, T.shape[0], (empty.numel(),), generator=g,
                                     device=X.device)
                sums[empty] = T[pick]
            Cn = _normalize(sums)
        assign = _nearest(X, Cn, chunk)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
        torch.use_deterministic_algorithms(prev_det)
    return Cn.contiguous(), assign


@torch.no_grad()
def make_workload(cfg: Workload | str, device="cpu", query_stream: int = 0):
    """Everything one search call needs, on ``device``.

    Returns a dict: X [n][d] f32, ids [n] i64 (= row), centroids [nlist][d] f32,
    assign [n] i32, Q [nq][d] f32, qids [nq] i64, and the search parameters.
    ``query_stream`` > 0 draws an independent query batch from the same index
    (one batch per process when queries are sharded over GPUs).
    """
    if isinstance(cfg, str):
        cfg = CONFIGS[cfg]
    X, g = make_corpus(cfg, device)
    cent, assign = build_index(X, cfg, g)
    if query_stream:
        g = torch.Generator(device=device).manual_seed(cfg.seed * 1_000_003 + query_stream)
    qrows = torch.randperm(cfg.n, generator=g, device=device)[:cfg.nq]
    return {
        "cfg": cfg,
        "X": X,
        "ids": torch.arange(cfg.n, device=device, dtype=torch.int64),
        "centroids": cent,
        "assign": assign,
        "Q": X[qrows].contiguous(),
        "qids": qrows.to(torch.int64),
        "tau": cfg.tau, "k": cfg.k, "nprobe": cfg.nprobe, "W": cfg.W,
    }


def to_numpy(wl: dict) -> dict:
    """Host numpy copies of a workload's arrays (for the oracle)."""
    out = {}
    for key in ("X", "ids", "centroids", "assign", "Q", "qids"):
        out[key] = wl[key].detach().cpu().numpy()
    return out


@torch.no_grad()
def make_sharded_workload(cfg: Workload | str, nshards: int, nlist_per_shard: int, device="cpu"):
    """The corpus of ``cfg`` split into coarse shards, each with its own IVF
    index (the public-100M layout of Sec. 6.1: coarse k-means shards, a
    separately built IVF index per shard): spherical k-means with ``nshards``
    centroids assigns every row a shard; each shard's rows get their own
    spherical k-means with ``nlist_per_shard`` centroids and exact assignment.
    Returns dict(Q, qids, shards = [dict(X, ids, centroids, assign)], cfg);
    ids are the rows' indices in the unsharded corpus, queries are drawn as in
    make_workload."""
    if isinstance(cfg, str):
        cfg = CONFIGS[cfg]
    X, g = make_corpus(cfg, device)
    coarse = replace(cfg, nlist=nshards, train_cap=min(cfg.n, 256 * nshards))
    _, shard_of = build_index(X, coarse, g)
    shards = []
    for s in range(nshards):
        rows = (shard_of == s).nonzero().flatten()
        Xs = X[rows].contiguous()
        scfg = replace(cfg, nlist=min(nlist_per_shard, rows.numel()),
                       train_cap=min(rows.numel(), 256 * nlist_per_shard))
        cent, assign = build_index(Xs, scfg, g)
        shards.append({"X": Xs, "ids": rows.to(torch.int64), "centroids": cent, "assign": assign})
    qrows = torch.randperm(cfg.n, generator=g, device=device)[:cfg.nq]
    return {"cfg": cfg, "Q": X[qrows].contiguous(), "qids": qrows.to(torch.int64), "shards": shards}


def make_rotation(d: int, seed: int = 7):
    """A seeded random orthogonal d x d matrix (float64, numpy): the rotation
    the quantized local search draws (QR of a Gaussian matrix, signs fixed so
    that R has a positive diagonal)."""
    import numpy as np
    g = torch.Generator(device="cpu").manual_seed(seed)
    A = torch.randn(d, d, generator=g, dtype=torch.float64)
    Qm, R = torch.linalg.qr(A)
    Qm = Qm * torch.sign(torch.diagonal(R)).unsqueeze(0)
    return np.ascontiguousarray(Qm.numpy())
