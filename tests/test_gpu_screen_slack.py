"""How much of the screen's proven error bound the tensor cores use.

The screen (the ranking's first pass, and the screening scan) scores a pair
with one fp16 product of the hi halves of the scaled split, summed in fp32 on
the tensor cores, and treats it as the exact score to within

    delta = (2^-10 + 2^-12 + d 2^-22) |q| |x| + 2^-26 sqrt(d) (|q| + |x|).

The bound is proven for round-to-nearest fp32 sums in any order
(tests/test_screen_bound.py checks it against emulated arithmetic); how the
tensor cores accumulate inside one MMA is not documented.  These tests read
the device's screened scores (sieve_screen_scores) for seeded pairs of the 1M
workload's distribution (d = 256, database-drawn queries against their own
rows, near duplicates and the rest), for the same pairs at other norms, and
for adversarial vectors whose every coordinate rounds the same way, and
report the slack: the largest |screen - fp64| / delta seen (must stay < 1)."""
import numpy as np
import pytest
import torch

import paper_2608_03199_gb300 as sieve
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def delta(q, x):
    d = q.shape[1]
    nq = np.linalg.norm(q.astype(np.float64), axis=1)[:, None]
    nx = np.linalg.norm(x.astype(np.float64), axis=1)[None, :]
    return (2.0**-10 + 2.0**-12 + d * 2.0**-22) * nq * nx + 2.0**-26 * np.sqrt(d) * (nq + nx)


def device_screen(x, q, dev):
    """Screened scores of every (q, x) pair: the rows of x as the index's
    centroids (their tensor-core layout), q as queries."""
    X = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(dev)
    index = sieve.build_layout(X.clone(), torch.arange(len(x), dtype=torch.int32, device=dev),
                               len(x), X)
    out = sieve.screen_scores(index, torch.from_numpy(np.ascontiguousarray(q, dtype=np.float32)).to(dev))
    torch.cuda.synchronize()
    return out.cpu().numpy().astype(np.float64)


def slack(x, q, dev):
    s = device_screen(x, q, dev)
    e = q.astype(np.float64) @ x.astype(np.float64).T
    return np.abs(s - e) / delta(q, x)


@pytest.fixture(scope="module")
def pairs():
    """1,000 database-drawn queries of a 1M-shaped workload (d = 256, Zipf
    clusters, power-law near-duplicate counts) against 8,192 of its rows: the
    queries' own rows, their near duplicates where the sample has them, and
    random rows."""
    cfg = synth.scaled("1m", n=60_000, nq=1_000, nlist=64, train_cap=None, seed=21)
    w = synth.to_numpy(synth.make_workload(cfg, device="cpu"))
    rng = np.random.default_rng(21)
    own = np.unique(w["qids"].astype(np.int64))
    rest = np.setdiff1d(np.arange(len(w["X"])), own)
    pick = np.concatenate([own, rng.choice(rest, 8192 - len(own), replace=False)])
    return w["X"][pick], w["Q"]


def test_screen_slack_on_the_workload(dev, pairs):
    x, q = pairs
    r = slack(x, q, dev)
    e = q.astype(np.float64) @ x.astype(np.float64).T
    hi = e > 0.8
    print(f"\nscreen slack, {r.size:,} pairs of the 1M workload's distribution (d = 256): "
          f"max {r.max():.3f}, 99.99th pct {np.quantile(r, 0.9999):.3f}, "
          f"mean {r.mean():.4f}; pairs scoring > 0.8: {int(hi.sum()):,}, max {r[hi].max():.3f}")
    assert hi.sum() >= len(q)          # every query's own row, and its near duplicates
    assert r.max() < 1.0


def test_screen_slack_at_other_norms(dev, pairs):
    x, q = pairs
    rng = np.random.default_rng(22)
    xs = (x * rng.uniform(0.05, 20, (len(x), 1))).astype(np.float32)
    qs = (q * rng.uniform(0.05, 20, (len(q), 1))).astype(np.float32)
    r = slack(xs, qs, dev)
    print(f"\nscreen slack at norms 0.05-20: max {r.max():.3f}, mean {r.mean():.4f}")
    assert r.max() < 1.0


def test_screen_slack_on_adversarial_rounding(dev):
    """Every coordinate just above 1 + 2^-11 in its fp16 binade (rounded down
    by nearly 2^-11 relative), q = x: every product's error has one sign, so
    the split's term alone is near the bound.  The device must stay below it,
    and come within a factor of two (the bound is not vacuous on the tensor
    cores either)."""
    rng = np.random.default_rng(23)
    d = 256
    base = 2.0 ** rng.integers(-4, 0, (384, d))
    v = base * (1.0 + 2.0**-11 * 0.999) / 256.0
    v *= rng.choice([-1.0, 1.0], (384, d))
    v = v.astype(np.float32)
    r = slack(v, v, dev)
    diag = np.diag(r)
    print(f"\nscreen slack, adversarial q = x: max {diag.max():.3f}, min {diag.min():.3f}; "
          f"all pairs max {r.max():.3f}")
    assert r.max() < 1.0
    assert diag.max() > 0.5
