"""Pins of the oracle's stopping rule (Sec. 4.1, Algorithms 1 and 2).

The state machines inside ``oracle.c`` are checked against
* the worked examples the paper prints (Fig. 2, Fig. 4, Sec. 4.3), stored in
  ``tests/golden/stopping_examples.json`` with their citations;
* two closed forms written independently of the state machines: "stop at the
  first rank that ends a run of W empties" and the fixed point
  s = min(nprobe, last_hit(<= s) + W) of the stop line;
* the equivalence of sequential and lookahead execution (Sec. 4.3) under many
  seeded completion orders, with every rank up to the stop line searched
  exactly once;
* W >= nprobe is fixed probing; probes are non-decreasing in W.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "stopping_examples.json")


def _pattern(s):
    return np.array([1 if c == "H" else 0 for c in s], np.uint8)


def first_run_end(hits, W):
    """Probes as the first rank r ending W consecutive empties, else nprobe."""
    nprobe = len(hits)
    run = 0
    for r, h in enumerate(hits, start=1):
        run = 0 if h else run + 1
        if run >= W:
            return r
    return nprobe


def stop_line_fixed_point(hits, W):
    """Probes as the fixed point of s = min(nprobe, h*(s) + W), h*(s) = last hit <= s."""
    nprobe = len(hits)
    s = min(W, nprobe)
    while True:
        last = max([j for j in range(1, s + 1) if hits[j - 1]], default=0)
        s2 = max(s, min(nprobe, last + W))
        if s2 == s:
            return s
        s = s2


def stop_line_trace(hits, W):
    nprobe = len(hits)
    s, trace = min(W, nprobe), []
    j = 1
    while j <= s:
        if hits[j - 1]:
            s = max(s, min(j + W, nprobe))
            trace.append(s)
        j += 1
    return trace


def test_golden_examples():
    cases = json.load(open(GOLDEN))["cases"]
    assert len(cases) >= 5
    for c in cases:
        h = _pattern(c["pattern"])
        assert oracle.stop_pattern(h, c["W"], "sequential") == c["probes"], c
        for seed in range(64):
            probes, visits = oracle.stop_pattern(h, c["W"], "lookahead", seed=seed)
            assert probes == c["probes"], (c, seed)
            assert (visits[:probes] == 1).all() and (visits[probes:] == 0).all()
        if "stop_line_trace" in c:
            assert stop_line_trace(h, c["W"]) == c["stop_line_trace"]


@pytest.mark.parametrize("nprobe", [1, 2, 3, 5, 8, 10])
def test_exhaustive_patterns(nprobe):
    for bits in itertools.product((0, 1), repeat=nprobe):
        h = np.array(bits, np.uint8)
        prev = 0
        for W in range(1, nprobe + 3):
            seq = oracle.stop_pattern(h, W, "sequential")
            assert seq == first_run_end(bits, W) == stop_line_fixed_point(bits, W), (bits, W)
            probes, visits = oracle.stop_pattern(h, W, "lookahead", seed=W * 7919 + sum(bits))
            assert probes == seq, (bits, W)
            assert (visits[:seq] == 1).all() and (visits[seq:] == 0).all()
            assert seq >= prev          # non-decreasing in W (prefix property, App. A)
            prev = seq
            if W >= nprobe:
                assert seq == nprobe    # fixed probing


def test_many_orders_long_pattern():
    rng = np.random.default_rng(3)
    for _ in range(200):
        nprobe = int(rng.integers(1, 65))
        h = (rng.random(nprobe) < rng.random()).astype(np.uint8)
        W = int(rng.integers(1, 20))
        seq = oracle.stop_pattern(h, W, "sequential")
        assert seq == first_run_end(h.tolist(), W)
        for seed in range(32):
            assert oracle.stop_pattern(h, W, "lookahead", seed=seed)[0] == seq


def test_infinite_window_is_fixed_probe():
    h = np.zeros(40, np.uint8)
    assert oracle.stop_pattern(h, 2**31 - 1, "sequential") == 40
    assert oracle.stop_pattern(h, 2**62, "lookahead")[0] == 40


def test_bad_arguments():
    with pytest.raises(ValueError):
        oracle.stop_pattern(np.zeros(4, np.uint8), 0, "sequential")
