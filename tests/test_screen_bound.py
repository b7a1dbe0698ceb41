"""The screening scan's error bound, checked on the CPU against the arithmetic
it bounds.

The screen scores a pair with one fp16 product per element: h(v) = fp16(256 v)
rounded to nearest, products exact in fp32, summed in fp32, times 2^-16.  The
scan skips a row only when that score is below threshold - delta with

    delta = (2^-10 + 2^-12 + d 2^-22) |q| |x| + 2^-26 sqrt(d) (|q| + |x|)

(sieve.h, scan_path).  Here numpy does the same arithmetic (float16 rounding
to nearest, float32 sums in two orders) on random vectors, on vectors of other
norms, on vectors deep in fp16's subnormal range and on adversarial vectors
whose every coordinate rounds with the largest relative error in the same
direction as its product; the error against the fp64 inner product must stay
below delta, and the adversarial case must come within a factor of two of it
(the bound is not vacuous)."""
import numpy as np
import pytest


def delta(q, x):
    d = q.shape[-1]
    nq = np.linalg.norm(q, axis=-1)
    nx = np.linalg.norm(x, axis=-1)
    return (2.0**-10 + 2.0**-12 + d * 2.0**-22) * nq * nx + 2.0**-26 * np.sqrt(d) * (nq + nx)


def screened(q, x, order="sequential"):
    """One product of the fp16 halves, fp32 accumulation, unscaled."""
    hq = (np.float32(256.0) * q.astype(np.float32)).astype(np.float16).astype(np.float32)
    hx = (np.float32(256.0) * x.astype(np.float32)).astype(np.float16).astype(np.float32)
    prod = hq * hx                                   # exact: 11-bit x 11-bit significands
    if order == "sequential":
        acc = np.zeros(prod.shape[:-1], np.float32)
        for i in range(prod.shape[-1]):
            acc = (acc + prod[..., i]).astype(np.float32)
    else:                                            # pairwise tree
        acc = prod
        while acc.shape[-1] > 1:
            if acc.shape[-1] % 2:
                acc = np.concatenate([acc, np.zeros(acc.shape[:-1] + (1,), np.float32)], -1)
            acc = (acc[..., 0::2] + acc[..., 1::2]).astype(np.float32)
        acc = acc[..., 0]
    return acc.astype(np.float64) * 2.0**-16


def exact(q, x):
    return np.einsum("...i,...i->...", q.astype(np.float32).astype(np.float64),
                     x.astype(np.float32).astype(np.float64))


def worst_ratio(q, x):
    e = exact(q, x)
    r = 0.0
    for order in ("sequential", "pairwise"):
        r = max(r, float(np.max(np.abs(screened(q, x, order) - e) / delta(q, x))))
    return r


def unit(v):
    return v / np.linalg.norm(v, axis=-1, keepdims=True)


@pytest.mark.parametrize("d", [4, 32, 96, 256])
def test_bound_holds_on_random_unit_vectors(d):
    rng = np.random.default_rng(d)
    q = unit(rng.standard_normal((3000, d))).astype(np.float32)
    x = unit(rng.standard_normal((3000, d))).astype(np.float32)
    x[:1000] = unit(q[:1000] + 0.05 * rng.standard_normal((1000, d))).astype(np.float32)  # near duplicates
    assert worst_ratio(q, x) < 1.0


@pytest.mark.parametrize("d", [64, 256])
def test_bound_holds_on_other_norms(d):
    rng = np.random.default_rng(100 + d)
    q = (unit(rng.standard_normal((3000, d))) * rng.uniform(0.05, 20, (3000, 1))).astype(np.float32)
    x = (unit(rng.standard_normal((3000, d))) * rng.uniform(0.05, 20, (3000, 1))).astype(np.float32)
    assert worst_ratio(q, x) < 1.0


def test_bound_holds_in_the_subnormal_range():
    """Coordinates of 1e-8 to 1e-5: 256 v is an fp16 subnormal (below 2^-14),
    so the rounding error is absolute (half of 2^-24), not relative."""
    rng = np.random.default_rng(7)
    d = 128
    mag = 10.0 ** rng.uniform(-8, -5, (2000, d))
    q = (mag * rng.choice([-1, 1], (2000, d))).astype(np.float32)
    x = (rng.uniform(-1e-5, 1e-5, (2000, d))).astype(np.float32)
    x[:, :4] = rng.standard_normal((2000, 4)).astype(np.float32)   # a few normal-range terms
    assert worst_ratio(q, x) < 1.0


def test_adversarial_rounding_stays_within_and_near_the_bound():
    """Every coordinate just above 1 + 2^-11 (in units of an fp16 binade), so
    fp16 rounds it down by nearly 2^-11 relative, with q = x: every product's
    error has the same sign, the worst case of the split's term."""
    rng = np.random.default_rng(11)
    d = 256
    base = 2.0 ** rng.integers(-4, 0, (500, d))                    # one binade per coordinate
    v = base * (1.0 + 2.0**-11 * 0.999) / 256.0
    v *= rng.choice([-1.0, 1.0], (500, d))
    q = v.astype(np.float32)
    x = q.copy()
    r = worst_ratio(q, x)
    assert r < 1.0
    assert r > 0.5
